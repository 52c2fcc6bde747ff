"""GPU parity of bp_reweighted_penalty against the oracle (fp64).

Tolerances follow from the kernel's fp32 arithmetic (u = 2^-24): a unit's
squared norm is a sum of n exact fp32 squares added in fp32, relative error at
most (n - 1) u (first order, nonnegative terms).  s + fp32(eps) adds at most
2 u more and the fp32 reciprocal u: alpha is within (n + 2) u.  The term
alpha^2 s (logarithmic derivative in s within [-1, 1]) is within (n + 4) u
after its two fp32 products; R, a sum of such nonnegative terms, as well.  The
gradient factor fp32(2 lambda) alpha alpha doubles alpha's error and adds three
roundings, the product with the weight one more: 2 (n + 2) u + 4 u."""
import numpy as np
import pytest
import torch

import oracle
from paper_2111_11581_gb300 import bp, inputs
from tests._util import dev16

pytestmark = pytest.mark.gpu

U32 = 2.0 ** -24

CASES = [
    # scheme, dtype, M, K, kh, kw, bm, bk
    (bp.BLOCK_BASED, bp.BF16, 512, 512, 1, 1, 16, 16),
    (bp.BLOCK_BASED, bp.F16, 100, 200, 1, 1, 8, 8),          # partial blocks, one ragged tile
    (bp.BLOCK_BASED, bp.F16, 33, 70, 1, 1, 1, 1),            # unstructured units, K % 8 != 0
    (bp.BLOCK_BASED, bp.BF16, 250, 1000, 1, 1, 100, 10),     # bm not a power of two, ragged tiles
    (bp.BLOCK_BASED, bp.BF16, 3000, 256, 1, 1, 3000, 256),   # bm = M: whole columns
    (bp.BLOCK_BASED, bp.F16, 20, 40, 1, 1, 4, 4),            # bm < row slices of a full tile
    (bp.BLOCK_PUNCHED, bp.F16, 128, 128 * 9, 3, 3, 8, 4),
    (bp.BLOCK_PUNCHED, bp.BF16, 24, 5 * 49, 7, 7, 8, 2),     # partial channel block
    (bp.BLOCK_BASED, bp.BF16, 4096, 4096, 1, 1, 128, 32),    # the benchmark's weight
]


def unit_size(scheme, M, K, bm, bk, groups):
    if groups == bp.GROUPS_ROWS:
        return min(bk, K)
    return min(bm, M) * (1 if scheme == bp.BLOCK_BASED else bk)


def check(case, W, eps, lam, groups=bp.GROUPS_LAYOUT):
    scheme, dtype, M, K, kh, kw, bm, bk = case
    lay = bp.layout(scheme, dtype, M, K, bm, bk, kh, kw)
    ws = bp.penalty_workspace(lay, groups=groups)
    a, R, g = bp.penalty(lay, dev16(W, dtype), eps, lam, ws=ws, groups=groups)
    torch.cuda.synchronize()
    a0, R0, g0 = oracle.reweighted_penalty(W, dtype, scheme, bm, bk, eps, lam, kh, kw,
                                           groups="rows" if groups == bp.GROUPS_ROWS else "layout")
    n = unit_size(scheme, M, K, bm, bk, groups)
    np.testing.assert_allclose(a.cpu().numpy(), a0, rtol=(n + 2) * U32, atol=0)
    assert float(R.cpu()[0]) == pytest.approx(R0, rel=(n + 4) * U32, abs=0)
    np.testing.assert_allclose(g.cpu().numpy(), g0, rtol=(2 * n + 8) * U32, atol=1e-37)
    # the workspace comes back zeroed and the same call gives the same bits
    assert int(ws[:4].count_nonzero()) == 0
    a2, R2, g2 = bp.penalty(lay, dev16(W, dtype), eps, lam, ws=ws, groups=groups)
    assert torch.equal(a, a2) and torch.equal(R, R2) and torch.equal(g, g2)
    return a, R, g


@pytest.mark.parametrize("case", CASES, ids=lambda c: f"s{c[0]}_{c[2]}x{c[3]}_b{c[6]}x{c[7]}")
def test_penalty_matches_oracle(case):
    scheme, dtype, M, K, kh, kw, bm, bk = case
    W = inputs.normal((M, K), 0.05, dtype, seed=3 * M + K)
    check(case, W, 1e-4, 0.5)


def test_penalty_zero_units_and_small_eps():
    # pruned (all-zero) columns: s = 0, alpha = 1/eps exactly, zero gradient
    case = (bp.BLOCK_BASED, bp.BF16, 256, 384, 1, 1, 64, 16)
    W = inputs.normal((256, 384), 0.05, bp.BF16, seed=11)
    W[:, ::3] = 0
    a, R, g = check(case, W, 1e-6, 2.0)
    a = a.cpu().numpy().reshape(4, 384)
    assert (a[:, ::3] == np.float64(np.float32(1.0) / np.float32(1e-6))).all()
    assert (g.cpu().numpy()[:, ::3] == 0).all()


def test_penalty_lambda_zero_and_negative():
    case = (bp.BLOCK_PUNCHED, bp.F16, 16, 8 * 9, 3, 3, 8, 4)
    W = inputs.normal((16, 72), 0.05, bp.F16, seed=5)
    _, R, g = check(case, W, 1e-4, 0.0)
    assert float(R.cpu()[0]) == 0.0 and int(g.count_nonzero()) == 0
    check(case, W, 1e-4, -0.25)


ROW_CASES = [
    # dtype, M, K, bk
    (bp.BF16, 256, 512, 16),
    (bp.F16, 100, 200, 8),          # partial last column block (200 = 25 x 8, fine) and odd M
    (bp.F16, 33, 70, 7),            # bk and K not multiples of 8: scalar path, partial block
    (bp.BF16, 64, 4096, 4096),      # whole rows
    (bp.F16, 40, 96, 40),           # partial last block of a vector-unfriendly width
    (bp.BF16, 4096, 4096, 32),      # the benchmark's weight
    (bp.BF16, 50, 512, 256),        # 32 lanes per segment
    (bp.F16, 3, 40, 8),             # a partial warp chunk
]


@pytest.mark.parametrize("case", ROW_CASES, ids=lambda c: f"rows_{c[1]}x{c[2]}_bk{c[3]}")
def test_row_penalty_matches_oracle(case):
    dtype, M, K, bk = case
    W = inputs.normal((M, K), 0.05, dtype, seed=5 * M + K)
    check((bp.BLOCK_BASED, dtype, M, K, 1, 1, 4, bk), W, 1e-4, 0.75, groups=bp.GROUPS_ROWS)
