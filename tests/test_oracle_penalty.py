"""Pins of the reweighted-regulariser oracle (Eq. prob_block with Eq. column /
Eq. punched): autograd of an independent grouping of the same objective, a
closed form, partial blocks by brute force.  CPU only."""
import numpy as np
import pytest
import torch

import oracle
from paper_2111_11581_gb300 import inputs

F16, BF16 = 0, 1


def _objective_grad(Wd, scheme, bm, bk, kh, kw, eps, lam):
    """R and dR/dW by autograd, units formed by reshaping (full blocks only)."""
    W = torch.tensor(Wd, dtype=torch.float64, requires_grad=True)
    M, K = W.shape
    if scheme == 0:
        s = (W.reshape(M // bm, bm, K) ** 2).sum(1)                       # (RB, K)
    else:
        KK = kh * kw
        C = K // KK
        W5 = W.reshape(M // bm, bm, C // bk, bk, KK)
        s = (W5 ** 2).sum((1, 3))                                           # (RB, CB, KK)
    alpha = 1.0 / (s.detach() + eps)
    R = lam * (alpha ** 2 * s).sum()
    R.backward()
    return alpha.reshape(-1).numpy(), R.item(), W.grad.numpy()


@pytest.mark.parametrize("scheme,M,K,bm,bk,kh,kw,dtype", [
    (0, 64, 96, 16, 8, 1, 1, F16),
    (0, 32, 48, 32, 48, 1, 1, BF16),       # one block: structured
    (0, 24, 40, 1, 1, 1, 1, F16),          # 1x1 blocks: unstructured
    (1, 32, 16 * 9, 8, 4, 3, 3, BF16),
    (1, 16, 8 * 25, 16, 8, 5, 5, F16),
])
def test_penalty_matches_autograd(scheme, M, K, bm, bk, kh, kw, dtype):
    W = inputs.normal((M, K), 0.05, dtype, seed=M + K)
    Wd = oracle.to_double(W, dtype)
    eps, lam = 1e-3, 0.37
    a, R, g = oracle.reweighted_penalty(W, dtype, scheme, bm, bk, eps, lam, kh, kw)
    a2, R2, g2 = _objective_grad(Wd, scheme, bm, bk, kh, kw, eps, lam)
    np.testing.assert_allclose(a, a2, rtol=1e-13)
    assert R == pytest.approx(R2, rel=1e-12)
    np.testing.assert_allclose(g, g2, rtol=1e-13, atol=0)


def _full_block_layouts(n, seed):
    rng = np.random.default_rng(seed)
    out = []
    for _ in range(n):
        bm = int(rng.choice([1, 2, 4, 8, 16]))
        if rng.random() < 0.5:
            bk = int(rng.choice([1, 3, 8, 16]))
            out.append((0, bm * int(rng.integers(1, 6)), bk * int(rng.integers(1, 8)), bm, bk,
                        1, 1, int(rng.integers(0, 2))))
        else:
            kh, kw = [(1, 1), (3, 3), (2, 5)][int(rng.integers(0, 3))]
            bk = int(rng.choice([1, 2, 4]))
            out.append((1, bm * int(rng.integers(1, 5)), bk * int(rng.integers(1, 6)) * kh * kw,
                        bm, bk, kh, kw, int(rng.integers(0, 2))))
    return out


@pytest.mark.parametrize("scheme,M,K,bm,bk,kh,kw,dtype", _full_block_layouts(25, 13))
def test_penalty_matches_autograd_random_layouts(scheme, M, K, bm, bk, kh, kw, dtype):
    """alpha, R and dR/dW of random full-block layouts (both schemes) equal the
    autograd of the objective with its groups formed by reshaping."""
    W = inputs.normal((M, K), 0.05, dtype, seed=3 * M + K)
    eps, lam = 10.0 ** -int(2 + (M + K) % 4), 0.5 + (M % 3)
    a, R, g = oracle.reweighted_penalty(W, dtype, scheme, bm, bk, eps, lam, kh, kw)
    a2, R2, g2 = _objective_grad(oracle.to_double(W, dtype), scheme, bm, bk, kh, kw, eps, lam)
    np.testing.assert_allclose(a, a2, rtol=1e-13)
    assert R == pytest.approx(R2, rel=1e-12)
    np.testing.assert_allclose(g, g2, rtol=1e-13, atol=0)


def test_penalty_closed_form_single_unit():
    # one column of 4 rows, values 1, 2, 2, 0 (exact in fp16): s = 9
    W = oracle.round_to(np.array([[1.0], [2.0], [2.0], [0.0]]), F16)
    eps, lam = 0.5, 2.0
    a, R, g = oracle.reweighted_penalty(W, F16, 0, 4, 1, eps, lam)
    assert a[0] == 1.0 / 9.5
    assert R == pytest.approx(lam * 9.0 / 9.5 ** 2, rel=1e-15)
    np.testing.assert_allclose(g[:, 0], 2 * lam / 9.5 ** 2 * np.array([1.0, 2.0, 2.0, 0.0]),
                               rtol=1e-15)


def test_penalty_partial_blocks_brute_force():
    # M and C not multiples of the block: units of the last blocks are smaller
    M, C, KK, bm, bk = 10, 7, 9, 4, 3
    W = inputs.normal((M, C * KK), 0.1, BF16, seed=5)
    Wd = oracle.to_double(W, BF16)
    eps, lam = 1e-2, 1.0
    a, R, g = oracle.reweighted_penalty(W, BF16, 1, bm, bk, eps, lam, 3, 3)
    RB, CB = -(-M // bm), -(-C // bk)
    want_g = np.zeros_like(Wd)
    want_R = 0.0
    for rb in range(RB):
        for cb in range(CB):
            for pos in range(KK):
                idx = [(f, c * KK + pos) for f in range(rb * bm, min(M, rb * bm + bm))
                       for c in range(cb * bk, min(C, cb * bk + bk))]
                s = sum(Wd[i] ** 2 for i in idx)
                al = 1.0 / (s + eps)
                assert a[(rb * CB + cb) * KK + pos] == pytest.approx(al, rel=1e-15)
                want_R += al * al * s
                for i in idx:
                    want_g[i] = 2 * lam * al * al * Wd[i]
    assert R == pytest.approx(lam * want_R, rel=1e-13)
    np.testing.assert_allclose(g, want_g, rtol=1e-14)


def test_penalty_rejects_nonpositive_eps():
    W = inputs.normal((8, 8), 0.1, F16, seed=1)
    with pytest.raises(Exception):
        oracle.reweighted_penalty(W, F16, 0, 4, 4, 0.0, 1.0)


def _row_objective_grad(Wd, bk, eps, lam):
    """Eq. row by autograd: the rows of each block (full column blocks)."""
    W = torch.tensor(Wd, dtype=torch.float64, requires_grad=True)
    M, K = W.shape
    s = (W.reshape(M, K // bk, bk) ** 2).sum(2)                              # (M, CB)
    alpha = 1.0 / (s.detach() + eps)
    R = lam * (alpha ** 2 * s).sum()
    R.backward()
    return alpha.reshape(-1).numpy(), R.item(), W.grad.numpy()


@pytest.mark.parametrize("M,K,bk,dtype", [(16, 64, 16, F16), (8, 48, 48, BF16), (12, 20, 1, F16)])
def test_row_penalty_matches_autograd(M, K, bk, dtype):
    W = inputs.normal((M, K), 0.05, dtype, seed=7 * M + K)
    Wd = oracle.to_double(W, dtype)
    eps, lam = 2e-3, 0.6
    a, R, g = oracle.reweighted_penalty(W, dtype, 0, 4, bk, eps, lam, groups="rows")
    a2, R2, g2 = _row_objective_grad(Wd, bk, eps, lam)
    np.testing.assert_allclose(a, a2, rtol=1e-13)
    assert R == pytest.approx(R2, rel=1e-12)
    np.testing.assert_allclose(g, g2, rtol=1e-13, atol=0)


def test_row_penalty_partial_block_and_transpose_duality():
    # a partial last column block sums its real columns only; and the row
    # groups of W are the column groups of W^T with bm = bk (whole-height
    # column blocks of the transpose are its rows' segments)
    M, K, bk = 6, 10, 4
    W = inputs.normal((M, K), 0.05, F16, seed=3)
    Wd = oracle.to_double(W, F16)
    eps, lam = 1e-3, 1.5
    a, R, g = oracle.reweighted_penalty(W, F16, 0, 1, bk, eps, lam, groups="rows")
    CB = 3
    s = np.array([[np.sum(Wd[r, cb * bk:min(K, cb * bk + bk)] ** 2) for cb in range(CB)]
                  for r in range(M)])
    np.testing.assert_allclose(a.reshape(M, CB), 1.0 / (s + eps), rtol=1e-14)
    WT = np.ascontiguousarray(W.T)
    aT, RT, gT = oracle.reweighted_penalty(WT, F16, 0, bk, 1, eps, lam)   # column groups of W^T
    # W^T is K x M: row-blocks of bk rows, unit (rb, column r) = W[r, rb-block]
    np.testing.assert_allclose(aT.reshape(CB, M).T.reshape(-1), a, rtol=1e-14)
    assert RT == pytest.approx(R, rel=1e-14)
    np.testing.assert_allclose(gT.T, g, rtol=1e-14)


def test_row_penalty_rejects_punched():
    W = inputs.normal((8, 18), 0.05, F16, seed=1)
    with pytest.raises(oracle.OracleError):
        oracle.reweighted_penalty(W, F16, 1, 4, 2, 1e-3, 1.0, 3, 3, groups="rows")
