"""GPU parity on every point of the block-sparse GEMM sweep at full size.

The sweep: M = K = N = 4096 and the BERT-base FC shapes 3072 x 768 and
768 x 3072 with N = 8192 tokens, fp16 and bf16, W ~ N(0, 0.02),
X ~ U(-1, 1), blocks bm in {8, 16, 32, 64, 128} x bk in {8, 16, 32, 128},
keep fraction in {1/2, 1/4, 1/8, 1/16}: 3 x 2 x 80 = 480 points, each run in
the launch configuration the benchmark uses.  Per point:

* the mask, rb_ptr, col_idx and compact values of bp_prune / bp_pack equal
  the oracle's bit for bit (Sec. 4.1 pruning rule, Sec. 4.3 storage);
* a sample of whole output rows (the first and last row, the rows on both
  sides of the first row-block boundary, and four seeded random rows)
  matches the oracle's masked GEMM within max |err| <= 1e-2 * max(1, |ref|);
* the whole output matches a second witness, cuBLAS in fp32 on the masked
  weight, within the same bound.

The weights and activations of one (shape, dtype) are the same for all of its
80 points (one seed per shape), so they are drawn once per module.
"""
import functools

import numpy as np
import pytest
import torch

import oracle
from paper_2111_11581_gb300 import bp, inputs
from tests._util import assert_close, dev16, host_bits

pytestmark = pytest.mark.gpu

POINTS = [(M, K, N, bm, bk, keep, dtype)
          for (M, K, N) in inputs.GEMM_SHAPES
          for dtype in (bp.BF16, bp.F16)
          for bm in inputs.SWEEP_BM
          for bk in inputs.SWEEP_BK
          for keep in inputs.SWEEP_KEEP]


def test_sweep_has_480_points():
    assert len(POINTS) == 480 and len(set(POINTS)) == 480


@functools.lru_cache(maxsize=1)
def _operands(M, K, N, dtype):
    L = inputs.gemm_point(M, K, N, 128, 128, 2.0, dtype)
    W = inputs.layer_weight(L, dtype)
    X = inputs.layer_input(L, dtype)
    return W, X, dev16(W, dtype), dev16(X, dtype)


@pytest.mark.parametrize("point", POINTS,
                         ids=[f"{M}x{K}x{N}_{inputs.dtype_name(d)}_bm{bm}_bk{bk}_keep1of{k}"
                              for (M, K, N, bm, bk, k, d) in POINTS])
def test_sweep_point_matches_oracle(point):
    M, K, N, bm, bk, keep, dtype = point
    rate = float(keep)
    W, X, Wd, Xd = _operands(M, K, N, dtype)
    lay = bp.layout(bp.BLOCK_BASED, dtype, M, K, bm, bk)
    mask = bp.prune(lay, Wd, rate)
    pw = bp.pack(lay, Wd, mask)
    Y = bp.gemm(pw, Xd)
    torch.cuda.synchronize()
    assert bp.device_status() == bp.OK

    ref_mask = oracle.prune(W, dtype, bp.BLOCK_BASED, bm, bk, rate)
    got_mask = mask.cpu().numpy()
    assert (got_mask == ref_mask).all(), f"{int((got_mask != ref_mask).sum())} mask bytes differ"
    rb_ptr, col_idx, values = oracle.pack(W, ref_mask, bm)
    assert (pw.rb_ptr.cpu().numpy() == rb_ptr).all(), "rb_ptr differs"
    assert (pw.col_idx.cpu().numpy() == col_idx).all(), "col_idx differs"
    assert (host_bits(pw.values) == values).all(), "packed values differ"

    rng = np.random.default_rng(M * 131 + K * 17 + bm * 7 + bk * 3 + keep)
    rows = np.unique(np.concatenate([[0, M - 1, min(bm, M) - 1, min(bm, M - 1)],
                                     rng.integers(0, M, 4)]))
    ref = oracle.masked_gemm(W[rows], ref_mask[rows], X, dtype)
    assert_close(host_bits(Y)[rows], ref, dtype, "sampled rows")

    ref2 = (Wd.float() * mask.float()) @ Xd.float()
    err = (Y.float() - ref2).abs()
    assert bool((err <= 1e-2 * ref2.abs().clamp_min(1.0)).all()), \
        f"cuBLAS witness: max err {float(err.max()):.4g}"
