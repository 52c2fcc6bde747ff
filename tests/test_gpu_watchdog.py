"""The kernels' bounded waits: with a watchdog budget far too small for the
work, the GEMM kernel gives up, records BP_ERR_TIMEOUT in the device status
word and returns (no hang, no fault); the context stays usable and the next
call with the normal budget is correct."""
import pytest
import torch

import oracle
from paper_2111_11581_gb300 import bp, inputs
from tests._util import assert_close, dev16, host_bits

pytestmark = pytest.mark.gpu


def test_expired_wait_reports_timeout_and_context_survives():
    M, K, N, dtype = 512, 1024, 2048, bp.BF16
    W = inputs.normal((M, K), 0.05, dtype, 77)
    X = inputs.uniform((K, N), -1, 1, dtype, 78)
    lay = bp.layout(bp.BLOCK_BASED, dtype, M, K, 128, 32)
    Wd = dev16(W, dtype)
    mask = bp.prune(lay, Wd, 2.0)
    pw = bp.pack(lay, Wd, mask)
    Xd = dev16(X, dtype)
    assert bp.device_status() == bp.OK
    try:
        bp.bp_set_watchdog_ns(1)            # every wait that does not succeed at once expires
        for _ in range(3):
            bp.gemm(pw, Xd)
        st = bp.device_status()
    finally:
        bp.bp_set_watchdog_ns(0)            # default budget again
    assert st == bp.ERR_TIMEOUT
    assert bp.device_status() == bp.OK      # reading the status cleared it
    Y = bp.gemm(pw, Xd)
    torch.cuda.synchronize()
    assert bp.device_status() == bp.OK
    ref = oracle.masked_gemm(W, mask.cpu().numpy(), X, dtype)
    assert_close(host_bits(Y), ref, dtype, "after timeout")
