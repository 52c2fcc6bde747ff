"""Pins of the row-pruning oracle (Sec. 4.1.1, independent row and column
pruning of each block; rows of a block are the groups of Eq. row).  CPU only."""
import itertools

import numpy as np
import pytest

import oracle
from paper_2111_11581_gb300 import inputs

F16, BF16 = 0, 1


def _row_scores(Wd, bm, bk):
    M, K = Wd.shape
    CB = -(-K // bk)
    return np.array([[np.sum(Wd[r, cb * bk:min(K, cb * bk + bk)] ** 2) for cb in range(CB)]
                     for r in range(M)])


@pytest.mark.parametrize("M,K,bm,bk,rate,dtype", [
    (64, 96, 16, 8, 4.0, F16), (40, 52, 16, 8, 3.0, BF16),   # partial row- and column-blocks
    (30, 40, 30, 40, 2.5, F16),                                # one block
])
def test_rows_equal_columns_of_the_transpose(M, K, bm, bk, rate, dtype):
    # The rows of the bm x bk blocks of W are the columns of the bk x bm blocks
    # of W^T: on scores without ties the two selections coincide.
    W = inputs.normal((M, K), 0.05, dtype, seed=M * K)
    s = _row_scores(oracle.to_double(W, dtype), bm, bk)
    assert len(np.unique(s)) == s.size           # no ties: the tie orders cannot matter
    m = oracle.prune_rows(W, dtype, bm, bk, rate)
    mT = oracle.prune(np.ascontiguousarray(W.T), dtype, 0, bk, bm, rate)
    np.testing.assert_array_equal(m, mT.T)


def test_rows_counts_and_and_semantics():
    M, K, bm, bk, rate = 48, 64, 16, 16, 4.0
    W = inputs.normal((M, K), 0.05, F16, seed=2)
    cols = oracle.prune(W, F16, 0, bm, bk, 2.0)
    m, keep = oracle.prune_rows(W, F16, bm, bk, rate, mask=cols, return_keep=True)
    CB = K // bk
    # every block keeps floor(16 / 4) = 4 rows and T = M*CB/4 exactly (no extras)
    assert keep.sum() == M * CB // 4
    blocks = keep.reshape(M // bm, CB, bm)
    assert (blocks.sum(2) == 4).all()
    # an element survives iff its column unit and its row unit survive
    rowk = np.zeros((M, K), np.uint8)
    for rb in range(M // bm):
        for cb in range(CB):
            for i in range(bm):
                rowk[rb * bm + i, cb * bk:(cb + 1) * bk] = blocks[rb, cb, i]
    np.testing.assert_array_equal(m, cols & rowk)
    # the kept rows of a block are its highest-norm rows
    s = _row_scores(oracle.to_double(W, F16), bm, bk)
    for rb in range(M // bm):
        for cb in range(CB):
            sc = s[rb * bm:(rb + 1) * bm, cb]
            kept = blocks[rb, cb].astype(bool)
            assert sc[kept].min() > sc[~kept].max()


def test_rows_brute_force_optimum():
    # the selection maximises the kept energy over all row sets with at least
    # floor(P_b / r) rows per block and T rows in total (partial last row-block)
    M, K, bm, bk, rate = 5, 6, 3, 3, 2.5
    W = inputs.normal((M, K), 0.05, F16, seed=9)
    s = _row_scores(oracle.to_double(W, F16), bm, bk)    # (M, CB)
    m, keep = oracle.prune_rows(W, F16, bm, bk, rate, return_keep=True)
    CB = 2
    units, blocks = [], []
    for rb in range(2):
        rows = range(rb * bm, min(M, rb * bm + bm))
        for cb in range(CB):
            blocks.append([(r, cb) for r in rows])
    units = [u for b in blocks for u in b]               # block-major, then row
    T = int(np.floor(len(units) / rate + 0.5))
    best, best_set = -1.0, None
    for comb in itertools.combinations(range(len(units)), T):
        chosen = set(comb)
        ok = all(sum(1 for u in b if units.index(u) in chosen) >= int(np.floor(len(b) / rate))
                 for b in blocks)
        if not ok:
            continue
        e = sum(s[units[i]] for i in comb)
        if e > best:
            best, best_set = e, chosen
    assert keep.sum() == T
    assert sorted(np.flatnonzero(keep)) == sorted(best_set)


def test_rows_special_cases():
    # bm = bk = 1: every element its own block -> global magnitude pruning
    M, K, rate = 12, 10, 4.0
    W = inputs.normal((M, K), 0.05, BF16, seed=4)
    Wd = oracle.to_double(W, BF16)
    m = oracle.prune_rows(W, BF16, 1, 1, rate)
    T = int(np.floor(M * K / rate + 0.5))
    order = np.lexsort((np.arange(M * K), -(Wd.reshape(-1) ** 2)))
    ref = np.zeros(M * K, np.uint8)
    ref[order[:T]] = 1
    np.testing.assert_array_equal(m.reshape(-1), ref)
    # bk = K, bm = M: whole rows, structured row pruning of the layer
    m = oracle.prune_rows(W, BF16, M, K, 3.0)
    assert all(len(set(row)) == 1 for row in m)          # each row all kept or all pruned
    assert m[:, 0].sum() == 4


def test_rows_rejects_bad_rate():
    W = inputs.normal((8, 8), 0.05, F16, seed=1)
    with pytest.raises(oracle.OracleError):
        oracle.prune_rows(W, F16, 4, 4, 0.5)


def _row_layouts(n, seed):
    rng = np.random.default_rng(seed)
    return [(int(rng.integers(1, 150)), int(rng.integers(1, 200)),
             int(rng.choice([1, 2, 5, 8, 16, 32])), int(rng.choice([1, 3, 8, 16, 32])),
             float(rng.choice([1.0, 1.5, 2.0, 8.0 / 3.0, 4.0, 7.0])), int(rng.integers(0, 2)))
            for _ in range(n)]


@pytest.mark.parametrize("M,K,bm,bk,rate,dtype", _row_layouts(30, 77))
def test_rows_satisfy_the_exchange_optimality_conditions(M, K, bm, bk, rate, dtype):
    """The row units (one row of one bm x bk block each, scored by the squared
    norm of its bk weights, computed here from the weights) are selected like
    column units: T = floor(sum P_b / r + 0.5) in total, at least floor(P_b / r)
    per block, maximal kept energy.  Certified by the exchange conditions:
    each block keeps its top rows, and no left-out row outscores a kept row of
    another block above its floor."""
    W = inputs.normal((M, K), 0.05, dtype, seed=M * 31 + K)
    s2 = _row_scores(oracle.to_double(W, dtype), bm, bk)       # [row, column block]
    _, keep = oracle.prune_rows(W, dtype, bm, bk, rate, return_keep=True)
    CB = -(-K // bk)
    blocks, g = [], 0
    for rb in range(-(-M // bm)):
        rows = range(rb * bm, min(M, rb * bm + bm))
        for cb in range(CB):
            blocks.append((list(range(g, g + len(rows))), np.array([s2[r, cb] for r in rows])))
            g += len(rows)
    assert g == keep.size
    T = int(np.floor(sum(len(u) for u, _ in blocks) / rate + 0.5))
    assert int(keep.sum()) == T
    slack = []
    for i, (u, sc) in enumerate(blocks):
        kb = keep[u] == 1
        base = int(np.floor(len(u) / rate))
        assert kb.sum() >= base
        if kb.any() and (~kb).any():
            assert sc[kb].min() >= sc[~kb].max()
        if kb.sum() > base:
            slack.append((sc[kb].min(), i))
    slack.sort()
    for i, (u, sc) in enumerate(blocks):
        out = sc[keep[u] == 0]
        others = [m for m, j in slack[:2] if j != i]
        if out.size and others:
            assert out.max() <= others[0]
