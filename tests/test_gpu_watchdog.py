"""The kernels' bounded waits.  A pipeline stage whose data never arrives
(dropped on purpose through bp_debug_drop_stage, the way a lost message is
simulated on the host) makes the tensor-core warp's wait run out: the kernel
records BP_ERR_TIMEOUT in the device status word and returns -- no hang, no
fault -- and the context stays usable for a correct call afterwards."""
import pytest
import torch

import oracle
from paper_2111_11581_gb300 import bp, inputs
from tests._util import assert_close, dev16, host_bits

pytestmark = pytest.mark.gpu


def _gemm_layer():
    M, K, N, dtype = 512, 1024, 2048, bp.BF16
    W = inputs.normal((M, K), 0.05, dtype, 77)
    X = inputs.uniform((K, N), -1, 1, dtype, 78)
    lay = bp.layout(bp.BLOCK_BASED, dtype, M, K, 128, 32)
    Wd = dev16(W, dtype)
    mask = bp.prune(lay, Wd, 2.0)
    return W, X, mask, bp.pack(lay, Wd, mask), dev16(X, dtype), dtype


@pytest.mark.parametrize("kind", ["gemm", "conv"])
def test_lost_stage_times_out_and_context_survives(kind):
    if kind == "gemm":
        W, X, mask, pw, Xd, dtype = _gemm_layer()
        run = lambda: bp.gemm(pw, Xd)                      # noqa: E731
    else:
        dtype = bp.F16
        Wc = inputs.normal((16, 8, 3, 3), 0.2, dtype, 79)
        x = inputs.normal((2, 8, 12, 12), 1.0, dtype, 80)
        lay = bp.layout(bp.BLOCK_PUNCHED, dtype, 16, 72, 8, 4, 3, 3)
        Wd = dev16(Wc.reshape(16, -1), dtype)
        mask = bp.prune(lay, Wd, 3.0)
        pw = bp.pack(lay, Wd, mask)
        xd = dev16(x, dtype)
        run = lambda: bp.conv2d(pw, xd, pad=(1, 1))       # noqa: E731
    assert bp.device_status() == bp.OK
    try:
        bp.bp_set_watchdog_ns(50_000_000)       # 50 ms budget per wait
        bp.bp_debug_drop_stage(0)          # CTA 0 loses its first stage
        run()
        st = bp.device_status()
    finally:
        bp.bp_debug_drop_stage(-1)
        bp.bp_set_watchdog_ns(0)
    assert st == bp.ERR_TIMEOUT
    assert bp.device_status() == bp.OK         # reading the status cleared it
    out = run()
    torch.cuda.synchronize()
    assert bp.device_status() == bp.OK
    if kind == "gemm":
        ref = oracle.masked_gemm(W, mask.cpu().numpy(), X, dtype)
    else:
        ref = oracle.masked_conv2d(Wc, mask.cpu().numpy(), x, dtype, pad=(1, 1))
    assert_close(host_bits(out), ref, dtype, f"{kind} after timeout")
