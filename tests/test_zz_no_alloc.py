"""bp_prune_noalloc: pruning for callers that cannot allocate device memory
(it uses a fixed scratch array inside the library instead of a caller-provided
workspace).  Its masks must equal those of bp_prune with a workspace, on two
calls in a row (the second call reuses the scratch array the first one left
behind), and a layout whose workspace exceeds the array is rejected up front.
This file is collected last on purpose."""
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
