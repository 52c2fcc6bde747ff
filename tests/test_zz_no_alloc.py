"""bp_prune_noalloc: pruning for callers that cannot allocate device memory
(it uses a fixed scratch array inside the library instead of a caller-provided
workspace).  Its masks must equal those of bp_prune with a workspace, on two
calls in a row (the second call reuses the scratch array the first one left
behind), on a layout whose workspace fills nearly all of the array, and a
layout whose workspace exceeds the array is rejected up front.  Once the
array's module is loaded, a call changes neither the device's free memory nor
torch's allocations.  This file is collected last on purpose."""
import ctypes

import numpy as np
import pytest
import torch

from paper_2111_11581_gb300 import bp, inputs

pytestmark = pytest.mark.gpu

CASES = [
    # scheme, dtype, M, K, kh, kw, bm, bk, rate   (two different layers, called in a row)
    (bp.BLOCK_BASED, bp.BF16, 1024, 2048, 1, 1, 32, 16, 5.0),       # base 3 + 819 extras
    (bp.BLOCK_PUNCHED, bp.F16, 128, 128 * 9, 3, 3, 8, 4, 8.0),
]


def _dev(bits, dtype):
    return inputs.as_torch(bits, dtype).cuda()


def test_noalloc_matches_workspace_prune_twice():
    stream = int(torch.cuda.current_stream().cuda_stream)
    for i, (scheme, dtype, M, K, kh, kw, bm, bk, rate) in enumerate(CASES):
        W = _dev(inputs.normal((M, K), 0.05, dtype, seed=900 + i), dtype)
        lay = bp.layout(scheme, dtype, M, K, bm, bk, kh, kw)
        ref = bp.prune(lay, W, rate)                       # existing entry point, own workspace
        got = torch.full((M, K), 7, dtype=torch.uint8, device="cuda")
        st = bp.bp_prune_noalloc(lay, W.data_ptr(), rate, got.data_ptr(), stream)
        assert st == bp.OK, bp.status_string(st)
        torch.cuda.synchronize()
        assert torch.equal(got, ref), f"call {i}: masks differ in {int((got != ref).sum())} bytes"


def test_noalloc_rejects_layout_beyond_its_scratch():
    lay = bp.layout(bp.BLOCK_BASED, bp.BF16, 8192, 8192, 1, 1)      # unstructured: 64M units
    assert bp.bp_workspace_size(lay) > 8 << 20
    W = torch.zeros(16, dtype=torch.bfloat16, device="cuda")
    mask = torch.zeros(16, dtype=torch.uint8, device="cuda")
    st = bp.bp_prune_noalloc(lay, W.data_ptr(), 2.0, mask.data_ptr(), 0)
    assert st == bp.ERR_WORKSPACE


# 768 filters x 1088 channels, 3x3, blocks of 4 x 4: bp_workspace_size is
# 8,358,912 bytes, 99.6 % of the 8 MiB array, so the array's tail is used.
BIG = (bp.BLOCK_PUNCHED, bp.BF16, 768, 1088 * 9, 3, 3, 4, 4, 3.0)


def test_noalloc_near_its_limit_allocates_nothing():
    scheme, dtype, M, K, kh, kw, bm, bk, rate = BIG
    lay = bp.layout(scheme, dtype, M, K, bm, bk, kh, kw)
    need = bp.bp_workspace_size(lay)
    assert (8 << 20) * 0.99 < need <= 8 << 20
    stream = int(torch.cuda.current_stream().cuda_stream)
    W = _dev(inputs.normal((M, K), 0.05, dtype, seed=977), dtype)
    ref = bp.prune(lay, W, rate)
    got = torch.full((M, K), 7, dtype=torch.uint8, device="cuda")
    # warm-up call: loads the array's module (its device memory is claimed then)
    assert bp.bp_prune_noalloc(lay, W.data_ptr(), rate, got.data_ptr(), stream) == bp.OK
    torch.cuda.synchronize()
    assert torch.equal(got, ref)
    got.fill_(7)
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    alloc0 = torch.cuda.memory_allocated()
    st = bp.bp_prune_noalloc(lay, W.data_ptr(), rate, got.data_ptr(), stream)
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert st == bp.OK, bp.status_string(st)
    assert torch.cuda.memory_allocated() == alloc0
    assert free1 == free0, f"free device memory changed by {free0 - free1} bytes"
    assert torch.equal(got, ref), f"masks differ in {int((got != ref).sum())} bytes"
