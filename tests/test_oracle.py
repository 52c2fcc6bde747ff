"""Pins of the CPU oracle against facts that do not come from the oracle itself:
exact encodings, brute force on tiny inputs, closed forms, special cases that
reduce to unstructured / structured pruning, the worked BCS example, and
textbook GEMM / convolution (numpy, torch CPU fp64)."""
import itertools
import json
import os
from fractions import Fraction

import numpy as np
import pytest
import torch

import oracle
from paper_2111_11581_gb300 import inputs

F16, BF16 = oracle.F16, oracle.BF16
BB, BP = oracle.BLOCK_BASED, oracle.BLOCK_PUNCHED
HERE = os.path.dirname(os.path.abspath(__file__))


# ------------------------------------------------------------------ encodings
def test_fp16_decode_all_patterns_match_numpy():
    bits = np.arange(1 << 16, dtype=np.uint32).astype(np.uint16)
    ours = oracle.to_double(bits, F16)
    ref = bits.view(np.float16).astype(np.float64)
    same = (ours == ref) | (np.isnan(ours) & np.isnan(ref))
    assert same.all()


def test_bf16_decode_all_patterns_match_fp32_view():
    bits = np.arange(1 << 16, dtype=np.uint32).astype(np.uint16)
    ours = oracle.to_double(bits, BF16)
    ref = (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    same = (ours == ref) | (np.isnan(ours) & np.isnan(ref))
    assert same.all()


def test_fp16_round_matches_numpy_rne():
    rng = np.random.default_rng(1)
    x = np.concatenate([
        rng.normal(0, 1, 20000), rng.normal(0, 1e-5, 5000), rng.normal(0, 3e4, 5000),
        # exact halfway points between neighbouring halves (ties)
        (np.arange(-3000, 3000, dtype=np.float16).astype(np.float64) +
         np.nextafter(np.arange(-3000, 3000, dtype=np.float16), np.float16(np.inf))
         .astype(np.float64)) / 2,
        [65504.0, 65519.99, 65520.0, 1e6, -1e6, 2.0 ** -25, 2.0 ** -24, 3 * 2.0 ** -26, 0.0, -0.0],
    ])
    ours = oracle.round_to(x, F16)
    ref = x.astype(np.float16).view(np.uint16)
    assert (ours == ref).all()


def _bf16_exact(x: float) -> int:
    """Reference RNE to bf16 with rational arithmetic (normal and subnormal)."""
    if x == 0:
        return 0x8000 if np.signbit(x) else 0
    s = 0x8000 if x < 0 else 0
    a = Fraction(abs(x))
    e = a.numerator.bit_length() - a.denominator.bit_length()
    while Fraction(2) ** e > a:
        e -= 1
    while Fraction(2) ** (e + 1) <= a:
        e += 1
    eq = max(e, -126)
    q = Fraction(2) ** (eq - 7)
    n = a / q
    fl = n.numerator // n.denominator
    rem = n - fl
    if rem > Fraction(1, 2) or (rem == Fraction(1, 2) and fl % 2 == 1):
        fl += 1
    r = fl * q
    if r >= Fraction(2) ** 128:
        return s | 0x7f80
    if r < Fraction(2) ** -126:
        return s | int(r / Fraction(2) ** -133)
    e2 = eq if fl < 256 else eq + 1
    mant = int(r / Fraction(2) ** (e2 - 7)) - 128
    return s | ((e2 + 127) << 7) | mant


def test_bf16_round_matches_exact_rational_rne():
    rng = np.random.default_rng(2)
    x = list(rng.normal(0, 1, 3000)) + list(rng.normal(0, 1e-38, 300)) + [
        1 + 2.0 ** -8,                 # tie -> even (1.0)
        1 + 2.0 ** -8 + 2.0 ** -40,    # just above the tie: rounding via fp32 would give 1.0
        1 + 3 * 2.0 ** -8,             # tie -> even (1 + 2^-6)
        -(1 + 2.0 ** -8), 3.0e38, 3.4e38, 2.0 ** -133, 2.0 ** -134, 3 * 2.0 ** -135]
    ours = oracle.round_to(np.array(x), BF16)
    ref = np.array([_bf16_exact(v) for v in x], dtype=np.uint16)
    assert (ours == ref).all()
    assert ours[-8] == 0x3f81      # 1 + 2^-8 + 2^-40 rounds up: one rounding from fp64


# ------------------------------------------------------------------ scores
def _brute_scores(Wd, scheme, bm, bk, kh, kw):
    """Recompute Eq. (column) / Eq. (punched) scores with numpy sums."""
    M = Wd.shape[0]
    Wm = Wd.reshape(M, -1)
    K = Wm.shape[1]
    out = []
    for r0 in range(0, M, bm):
        rows = Wm[r0:r0 + bm]
        if scheme == BB:
            for c0 in range(0, K, bk):
                for j in range(c0, min(K, c0 + bk)):
                    out.append(float(np.sum(rows[:, j] ** 2)))
        else:
            KK = kh * kw
            C = K // KK
            R = rows.reshape(rows.shape[0], C, KK)
            for c0 in range(0, C, bk):
                for pos in range(KK):
                    out.append(float(np.sum(R[:, c0:c0 + bk, pos] ** 2)))
    return np.array(out)


@pytest.mark.parametrize("dtype", [F16, BF16])
@pytest.mark.parametrize("scheme,M,K,kh,kw,bm,bk", [
    (BB, 10, 13, 1, 1, 4, 5),      # partial row- and column-blocks
    (BB, 8, 8, 1, 1, 8, 8),
    (BP, 6, 5 * 9, 3, 3, 4, 2),    # punched 3x3, partial filter and channel blocks
    (BP, 4, 3 * 1, 1, 1, 2, 2),    # punched 1x1
])
def test_scores_exact_on_grid_values(dtype, scheme, M, K, kh, kw, bm, bk):
    # multiples of 2^-4 with |k| <= 32: squares and their sums are exact in fp64,
    # so any summation order gives the same value and a dropped term shows up.
    W = inputs.small_grid((M, K), dtype, seed=11)
    Wd = oracle.to_double(W, dtype)
    s = oracle.scores(W, dtype, scheme, bm, bk, kh, kw)
    ref = _brute_scores(Wd, scheme, bm, bk, kh, kw)
    assert s.shape == ref.shape
    assert (s == ref).all()


def test_scores_hand_example():
    # 2x4 block-based, bm=2, bk=2: columns (1,3), (2,-1), (0,0.5), (4,4)
    Wd = np.array([[1, 2, 0, 4], [3, -1, 0.5, 4]], dtype=np.float64)
    W = oracle.round_to(Wd, F16)
    s = oracle.scores(W, F16, BB, 2, 2)
    assert list(s) == [10.0, 5.0, 0.25, 32.0]
    # punched: F=2, C=2, 1x2 kernels, block 2x2 -> position scores over all 4 kernels
    Wp = np.array([[[[1, 2]], [[3, 0]]], [[[0, 1]], [[1, 1]]]], dtype=np.float64)
    sp = oracle.scores(oracle.round_to(Wp, F16).reshape(2, 4), F16, BP, 2, 2, 1, 2)
    assert list(sp) == [1 + 9 + 0 + 1, 4 + 0 + 1 + 1]


def test_scores_reject_nonfinite():
    W = oracle.round_to(np.array([[1.0, np.inf], [0.0, 1.0]]), F16)
    with pytest.raises(oracle.OracleError):
        oracle.scores(W, F16, BB, 1, 1)


# ------------------------------------------------------------------ counts
@pytest.mark.parametrize("args,expect", [
    # FC 512x512, 16x16 blocks, 4x: every block keeps exactly 4 of 16 columns
    ((BB, 512, 512, 1, 1, 16, 16, 4.0), (32 * 32 * 4, 32 * 32 * 4, 0)),
    # 3x3 punched 128x128, 8x4 blocks, keep 3 of 9
    ((BP, 128, 128 * 9, 3, 3, 8, 4, 3.0), (16 * 32 * 3, 16 * 32 * 3, 0)),
    # 8x with 9 positions: base 1 per block, B/8 extras (B = 16*32 blocks)
    ((BP, 128, 128 * 9, 3, 3, 8, 4, 8.0), (512, 576, 64)),
    # bk=8 at keep 1/16: base 0, all 4096*RB/16 kept units are extras
    ((BB, 4096, 4096, 1, 1, 128, 8, 16.0), (0, 32 * 256, 32 * 256)),
    # partial last column block: K=20, bk=8 -> blocks of 8, 8, 4 at rate 3
    ((BB, 4, 20, 1, 1, 4, 8, 3.0), (2 + 2 + 1, 7, 2)),
])
def test_counts_closed_forms(args, expect):
    assert oracle.counts(*args) == expect


def test_counts_reject_rate_below_one():
    with pytest.raises(oracle.OracleError):
        oracle.counts(BB, 8, 8, 1, 1, 2, 2, 0.5)


# ------------------------------------------------------------------ selection
def _units_of_blocks(scheme, M, K, kh, kw, bm, bk):
    """list of blocks, each a list of unit indices g (unit order of the oracle)."""
    blocks, g = [], 0
    RB = -(-M // bm)
    if scheme == BB:
        CB = -(-K // bk)
        for rb in range(RB):
            for cb in range(CB):
                w = min(bk, K - cb * bk)
                blocks.append(list(range(rb * K + cb * bk, rb * K + cb * bk + w)))
    else:
        KK = kh * kw
        CB = -(-(K // KK) // bk)
        for b in range(RB * CB):
            blocks.append(list(range(b * KK, b * KK + KK)))
    return blocks


def _brute_best(s, blocks, rate, T):
    """Maximum kept energy over all unit sets with |S| = T and >= floor(P_b/r) per block."""
    U = len(s)
    best, best_sets = -1.0, []
    for S in itertools.combinations(range(U), T):
        Sset = set(S)
        if any(sum(u in Sset for u in b) < int(np.floor(len(b) / rate)) for b in blocks):
            continue
        e = sum(s[u] for u in S)
        if e > best + 1e-12:
            best, best_sets = e, [Sset]
        elif abs(e - best) <= 1e-12:
            best_sets.append(Sset)
    return best, best_sets


@pytest.mark.parametrize("scheme,M,K,kh,kw,bm,bk,rate", [
    (BB, 4, 8, 1, 1, 2, 4, 2.0),
    (BB, 4, 8, 1, 1, 2, 4, 4.0),
    (BB, 4, 8, 1, 1, 2, 4, 8.0 / 3.0),   # base 1 per block + global extras
    (BB, 3, 6, 1, 1, 2, 4, 2.5),         # partial row- and column-blocks
    (BP, 2, 2 * 4, 2, 2, 1, 1, 2.0),     # punched 2x2 kernels
    (BP, 3, 3 * 4, 2, 2, 2, 2, 3.0),
])
def test_prune_is_the_unique_energy_optimum(scheme, M, K, kh, kw, bm, bk, rate):
    rng = np.random.default_rng(abs(hash((scheme, M, K, bm, bk, rate))) % 2 ** 32)
    Wd = rng.normal(0, 1, (M, K))
    W = oracle.round_to(Wd, F16)
    s = oracle.scores(W, F16, scheme, bm, bk, kh, kw)
    assert len(set(s.tolist())) == len(s)          # distinct scores -> unique optimum
    mask, keep = oracle.prune(W, F16, scheme, bm, bk, rate, kh, kw, return_keep=True)
    _, T, _ = oracle.counts(scheme, M, K, kh, kw, bm, bk, rate)
    blocks = _units_of_blocks(scheme, M, K, kh, kw, bm, bk)
    best, sets = _brute_best(s, blocks, rate, T)
    assert len(sets) == 1
    assert set(np.nonzero(keep)[0].tolist()) == sets[0]
    assert abs(sum(s[keep == 1]) - best) < 1e-9


def _random_layouts(n, seed):
    rng = np.random.default_rng(seed)
    out = []
    for _ in range(n):
        if rng.random() < 0.5:
            M, K = int(rng.integers(1, 200)), int(rng.integers(1, 300))
            bm = int(rng.choice([1, 2, 3, 8, 16, 32, 64, 128]))
            bk = int(rng.choice([1, 4, 7, 8, 16, 32]))
            rate = float(rng.choice([1.0, 1.5, 2.0, 3.0, 8.0 / 3.0, 4.0, 6.0, 16.0]))
            out.append((BB, M, K, 1, 1, bm, bk, rate))
        else:
            kh, kw = [(1, 1), (3, 3), (2, 3)][int(rng.integers(0, 3))]
            M, C = int(rng.integers(1, 70)), int(rng.integers(1, 40))
            bm = int(rng.choice([1, 4, 8, 16]))
            bk = int(rng.choice([1, 2, 4, 8]))
            rate = float(rng.choice([1.0, 2.0, 3.0, 4.5, 8.0, 9.0]))
            out.append((BP, M, C * kh * kw, kh, kw, bm, bk, rate))
    return out


@pytest.mark.parametrize("scheme,M,K,kh,kw,bm,bk,rate", _random_layouts(40, 2024))
def test_prune_satisfies_the_exchange_optimality_conditions(scheme, M, K, kh, kw, bm, bk, rate):
    """Kept energy is maximal over all unit sets of size T = floor(sum P_b / r + 0.5)
    with at least floor(P_b / r) units per block iff (1) every block keeps its
    highest-scoring units and (2) no unit left out scores above a kept unit of
    another block that holds more than its floor (block energies are concave in
    the count, so single transfers certify the optimum).  Checked on random
    layouts with partial blocks, both schemes and non-integer rates, from the
    scores and the kept set alone."""
    dt = F16 if (M + K) % 2 else BF16
    W = inputs.normal((M, K), 0.05, dt, seed=M * 1000 + K)
    s = oracle.scores(W, dt, scheme, bm, bk, kh, kw)
    _, keep = oracle.prune(W, dt, scheme, bm, bk, rate, kh, kw, return_keep=True)
    blocks = _units_of_blocks(scheme, M, K, kh, kw, bm, bk)
    sizes = [len(b) for b in blocks]
    T = int(np.floor(sum(sizes) / rate + 0.5))
    assert int(keep.sum()) == T
    slack_min = []                                   # (lowest kept score, block) of blocks above floor
    for i, b in enumerate(blocks):
        kb = keep[b] == 1
        base = int(np.floor(len(b) / rate))
        assert kb.sum() >= base
        if kb.any() and (~kb).any():
            assert s[b][kb].min() >= s[b][~kb].max()          # condition (1)
        if kb.sum() > base:
            slack_min.append((s[b][kb].min(), i))
    slack_min.sort()
    for i, b in enumerate(blocks):
        out = s[b][keep[b] == 0]
        if out.size == 0:
            continue
        others = [m for m, j in slack_min[:2] if j != i]
        if others:
            assert out.max() <= others[0]                     # condition (2)


def test_prune_ties_go_to_lower_index():
    W = oracle.round_to(np.ones((4, 8)), F16)     # every score equal
    mask, keep = oracle.prune(W, F16, BB, 2, 4, 8.0 / 3.0, return_keep=True)
    # 4 blocks of 4 units at rate 8/3: base floor(1.5) = 1 per block (its unit 0),
    # T = floor(16 / (8/3) + 0.5) = 6, so E = 2 extras: the lowest-indexed
    # remaining units, which are units 1 and 2 of block 0
    assert np.nonzero(keep)[0].tolist() == [0, 1, 2, 4, 8, 12]


def test_prune_unstructured_special_case():
    """bm = bk = 1: each unit is one weight -> global magnitude pruning (Sec. 4.4)."""
    rng = np.random.default_rng(5)
    M, K, rate = 16, 24, 3.0
    W = oracle.round_to(rng.normal(0, 1, (M, K)), BF16)
    Wd = oracle.to_double(W, BF16)
    mask = oracle.prune(W, BF16, BB, 1, 1, rate)
    T = int(np.floor(M * K / rate + 0.5))
    order = sorted(range(M * K), key=lambda i: (-Wd.flat[i] ** 2, i))
    ref = np.zeros(M * K, np.uint8)
    ref[order[:T]] = 1
    assert (mask.reshape(-1) == ref).all()


def test_prune_structured_special_case():
    """bm = M: one row-block, so each column is kept or pruned whole; with
    bk = K too this is top-T columns by L2 norm (structured pruning, Sec. 4.4)."""
    rng = np.random.default_rng(6)
    M, K = 12, 40
    W = oracle.round_to(rng.normal(0, 1, (M, K)), F16)
    Wd = oracle.to_double(W, F16)
    mask = oracle.prune(W, F16, BB, M, 8, 4.0)
    assert all(mask[:, k].min() == mask[:, k].max() for k in range(K))
    mask2 = oracle.prune(W, F16, BB, M, K, 5.0)
    colnorm = (Wd ** 2).sum(0)
    top = sorted(range(K), key=lambda k: (-colnorm[k], k))[:8]
    assert sorted(np.nonzero(mask2[0])[0].tolist()) == sorted(top)
    assert all(mask2[:, k].min() == mask2[:, k].max() for k in range(K))


@pytest.mark.parametrize("scheme,M,K,kh,kw,bm,bk,rate", [
    (BB, 100, 96, 1, 1, 16, 16, 4.0),
    (BB, 90, 100, 1, 1, 32, 8, 16.0),
    (BP, 40, 24 * 9, 3, 3, 8, 4, 8.0),
    (BP, 33, 10 * 9, 3, 3, 16, 8, 3.0),
])
def test_prune_invariants(scheme, M, K, kh, kw, bm, bk, rate):
    W = inputs.normal((M, K), 0.02, BF16, seed=7)
    mask, keep = oracle.prune(W, BF16, scheme, bm, bk, rate, kh, kw, return_keep=True)
    sb, T, E = oracle.counts(scheme, M, K, kh, kw, bm, bk, rate)
    assert int(keep.sum()) == T
    # every row of a row-block keeps the same columns (BCS occurrence property)
    for r0 in range(0, M, bm):
        rows = mask[r0:r0 + bm]
        assert (rows == rows[0]).all()
    # per block at least floor(P/r)
    for b in _units_of_blocks(scheme, M, K, kh, kw, bm, bk):
        assert keep[b].sum() >= int(np.floor(len(b) / rate))
    # punched: inside a block, the kept positions are the same for every kernel
    if scheme == BP:
        KK = kh * kw
        m3 = mask.reshape(M, K // KK, KK)
        for r0 in range(0, M, bm):
            for c0 in range(0, K // KK, bk):
                blk = m3[r0:r0 + bm, c0:c0 + bk]
                assert (blk == blk[0, 0]).all()
    # achieved rate equals the requested one when sum(P)/r is an integer
    U = keep.size
    if (U / rate) == int(U / rate):
        assert U / keep.sum() == rate


# ------------------------------------------------------------------ storage
def test_bcs_worked_example():
    with open(os.path.join(HERE, "golden", "bcs_example.json")) as f:
        g = json.load(f)
    K, bm = g["K"], g["bm"]
    cols = g["stated_by_paper"]["compact_column_array"]
    Wd = np.zeros((2, K))
    Wd[0, cols] = g["stated_by_paper"]["first_row_weights"]
    Wd[1, cols] = g["row1_weights_chosen_here"]
    W = oracle.round_to(Wd, F16)
    mask = (Wd != 0).astype(np.uint8)
    rb_ptr, col_idx, values = oracle.pack(W, mask, bm)
    assert col_idx.tolist() == cols
    assert rb_ptr.tolist() == g["stated_by_paper"]["column_stride_first_row"]
    assert [0, bm] == g["stated_by_paper"]["occurrence"]
    assert oracle.to_double(values[:3], F16).tolist() == g["stated_by_paper"]["first_row_weights"]


@pytest.mark.parametrize("scheme,M,K,kh,kw,bm,bk,rate", [
    (BB, 70, 50, 1, 1, 16, 8, 4.0),
    (BP, 24, 12 * 9, 3, 3, 8, 4, 3.0),
    (BB, 10, 512, 1, 1, 16, 16, 8.0),
])
def test_pack_roundtrip(scheme, M, K, kh, kw, bm, bk, rate):
    W = inputs.normal((M, K), 1.0, F16, seed=9)
    mask = oracle.prune(W, F16, scheme, bm, bk, rate, kh, kw)
    rb_ptr, col_idx, values = oracle.pack(W, mask, bm)
    W2, mask2 = oracle.unpack(M, K, bm, rb_ptr, col_idx, values)
    assert (mask2 == mask).all()
    assert (W2 == np.where(mask == 1, W, 0)).all()
    assert rb_ptr[-1] == col_idx.size
    for rb in range(len(rb_ptr) - 1):
        seg = col_idx[rb_ptr[rb]:rb_ptr[rb + 1]]
        assert (np.diff(seg) > 0).all()
        # values of row-block rb: bm_rb x K'_rb row-major, starting at bm * rb_ptr[rb]
        rows = W[rb * bm:(rb + 1) * bm]
        kp = seg.size
        blk = values[bm * rb_ptr[rb]: bm * rb_ptr[rb] + rows.shape[0] * kp]
        assert (blk.reshape(rows.shape[0], kp) == rows[:, seg]).all()
        assert (mask[rb * bm:(rb + 1) * bm][:, seg] == 1).all()
        assert mask[rb * bm:(rb + 1) * bm].sum() == rows.shape[0] * kp


@pytest.mark.parametrize("scheme,M,K,kh,kw,bm,bk,rate", _random_layouts(30, 91))
def test_pack_roundtrip_random_layouts(scheme, M, K, kh, kw, bm, bk, rate):
    """The compact storage of random layouts unpacks to the mask and the
    masked weight exactly; each row-block's list is ascending and its values
    are the row-block's rows at those columns."""
    W = inputs.normal((M, K), 1.0, BF16, seed=M + 7 * K)
    mask = oracle.prune(W, BF16, scheme, bm, bk, rate, kh, kw)
    rb_ptr, col_idx, values = oracle.pack(W, mask, bm)
    W2, mask2 = oracle.unpack(M, K, bm, rb_ptr, col_idx, values)
    assert (mask2 == mask).all()
    assert (W2 == np.where(mask == 1, W, 0)).all()
    assert rb_ptr[0] == 0 and rb_ptr[-1] == col_idx.size and len(rb_ptr) == -(-M // bm) + 1
    for rb in range(len(rb_ptr) - 1):
        seg = col_idx[rb_ptr[rb]:rb_ptr[rb + 1]]
        assert (np.diff(seg) > 0).all()
        rows = W[rb * bm:(rb + 1) * bm]
        blk = values[bm * rb_ptr[rb]: bm * rb_ptr[rb] + rows.shape[0] * seg.size]
        assert (blk.reshape(rows.shape[0], seg.size) == rows[:, seg]).all()


def test_pack_rejects_inconsistent_rows():
    W = oracle.round_to(np.ones((4, 4)), F16)
    mask = np.eye(4, dtype=np.uint8)
    with pytest.raises(oracle.OracleError):
        oracle.pack(W, mask, 2)


# ------------------------------------------------------------------ layer outputs
@pytest.mark.parametrize("dtype", [F16, BF16])
def test_masked_gemm_matches_numpy(dtype):
    rng = np.random.default_rng(3)
    M, K, N = 37, 61, 29
    W = oracle.round_to(rng.normal(0, 0.1, (M, K)), dtype)
    X = oracle.round_to(rng.uniform(-1, 1, (K, N)), dtype)
    mask = (rng.random((M, K)) < 0.3).astype(np.uint8)
    bias = rng.normal(0, 0.1, M).astype(np.float32)
    Y, acc = oracle.masked_gemm(W, mask, X, dtype, bias=bias, relu=True, return_acc=True)
    ref = (oracle.to_double(W, dtype) * mask) @ oracle.to_double(X, dtype)
    ref = np.maximum(ref + bias.astype(np.float64)[:, None], 0.0)
    assert np.abs(acc - ref).max() < 1e-12
    assert (Y == oracle.round_to(acc, dtype)).all()


def test_masked_gemm_exact_on_grid_values():
    M, K, N = 9, 20, 7
    W = inputs.small_grid((M, K), F16, seed=1)
    X = inputs.small_grid((K, N), F16, seed=2)
    mask = (np.arange(M * K).reshape(M, K) % 3 == 0).astype(np.uint8)
    _, acc = oracle.masked_gemm(W, mask, X, F16, return_acc=True)
    ref = (oracle.to_double(W, F16) * mask) @ oracle.to_double(X, F16)
    assert (acc == ref).all()          # all partial sums exact -> order-independent


@pytest.mark.parametrize("stride,pad,kh,kw", [(1, 1, 3, 3), (2, 1, 3, 3), (1, 0, 1, 1),
                                              (2, 0, 1, 1), (1, 2, 3, 2), (2, 3, 7, 7)])
def test_masked_conv2d_matches_torch(stride, pad, kh, kw):
    rng = np.random.default_rng(4)
    F, C, Nb, H, Wd = 6, 5, 2, 11, 9
    W = oracle.round_to(rng.normal(0, 0.3, (F, C, kh, kw)), BF16)
    x = oracle.round_to(rng.normal(0, 1, (Nb, C, H, Wd)), BF16)
    mask = (rng.random((F, C * kh * kw)) < 0.5).astype(np.uint8)
    bias = rng.normal(0, 0.1, F).astype(np.float32)
    out, acc = oracle.masked_conv2d(W, mask, x, BF16, pad=(pad, pad), stride=(stride, stride),
                                    bias=bias, relu=True, return_acc=True)
    wt = torch.from_numpy(oracle.to_double(W, BF16) * mask.reshape(F, C, kh, kw))
    xt = torch.from_numpy(oracle.to_double(x, BF16))
    ref = torch.nn.functional.conv2d(xt, wt, torch.from_numpy(bias.astype(np.float64)),
                                     stride=stride, padding=pad).clamp_min(0).numpy()
    assert acc.shape == ref.shape
    assert np.abs(acc - ref).max() < 1e-12
    assert (out == oracle.round_to(acc, BF16)).all()


def _conv_cases(n, seed):
    rng = np.random.default_rng(seed)
    out = []
    for _ in range(n):
        kh, kw = int(rng.integers(1, 6)), int(rng.integers(1, 6))
        sh, sw = int(rng.integers(1, 4)), int(rng.integers(1, 4))
        ph, pw = int(rng.integers(0, 4)), int(rng.integers(0, 4))
        H = int(rng.integers(max(1, kh - 2 * ph), 14))
        W = int(rng.integers(max(1, kw - 2 * pw), 14))
        out.append((int(rng.integers(1, 7)), int(rng.integers(1, 6)), int(rng.integers(1, 3)),
                    H, W, kh, kw, sh, sw, ph, pw))
    return out


@pytest.mark.parametrize("F,C,Nb,H,W,kh,kw,sh,sw,ph,pw", _conv_cases(30, 5))
def test_masked_conv2d_random_shapes_match_torch(F, C, Nb, H, W, kh, kw, sh, sw, ph, pw):
    """Random kernel sizes, unequal strides and paddings, non-square images:
    the fp64 accumulation equals torch's fp64 convolution of the masked weight."""
    rng = np.random.default_rng(F * 1000 + C * 100 + H * 10 + W)
    Wt = oracle.round_to(rng.normal(0, 0.3, (F, C, kh, kw)), F16)
    x = oracle.round_to(rng.normal(0, 1, (Nb, C, H, W)), F16)
    mask = (rng.random((F, C * kh * kw)) < 0.6).astype(np.uint8)
    bias = rng.normal(0, 0.1, F).astype(np.float32)
    out, acc = oracle.masked_conv2d(Wt, mask, x, F16, pad=(ph, pw), stride=(sh, sw), bias=bias,
                                    return_acc=True)
    wt = torch.from_numpy(oracle.to_double(Wt, F16) * mask.reshape(F, C, kh, kw))
    ref = torch.nn.functional.conv2d(torch.from_numpy(oracle.to_double(x, F16)), wt,
                                     torch.from_numpy(bias.astype(np.float64)),
                                     stride=(sh, sw), padding=(ph, pw)).numpy()
    assert acc.shape == ref.shape
    assert np.abs(acc - ref).max() < 1e-12
    assert (out == oracle.round_to(acc, F16)).all()


def test_masked_conv2d_1x1_is_gemm_per_image():
    rng = np.random.default_rng(8)
    F, C, Nb, H, Wd = 8, 12, 3, 5, 4
    W = oracle.round_to(rng.normal(0, 0.3, (F, C)), F16)
    x = oracle.round_to(rng.normal(0, 1, (Nb, C, H, Wd)), F16)
    mask = (rng.random((F, C)) < 0.5).astype(np.uint8)
    _, acc = oracle.masked_conv2d(W.reshape(F, C, 1, 1), mask, x, F16, return_acc=True)
    for b in range(Nb):
        _, g = oracle.masked_gemm(W, mask, x[b].reshape(C, H * Wd), F16, return_acc=True)
        assert np.abs(acc[b].reshape(F, -1) - g).max() == 0.0


def test_oracle_results_do_not_depend_on_thread_count():
    """The parallel loops compute each output in one thread in a fixed order,
    so masks and outputs are identical with one thread and with all."""
    dt = inputs.BF16
    W = inputs.normal((96, 160), 0.05, dt, 41)
    X = inputs.uniform((160, 24), -1.0, 1.0, dt, 42)
    Wc = inputs.normal((12, 6, 3, 3), 0.2, dt, 43)
    x = inputs.normal((2, 6, 9, 7), 1.0, dt, 44)
    n = oracle.max_threads()

    def run():
        m = oracle.prune(W, dt, BB, 32, 16, 3.0)
        y = oracle.masked_gemm(W, m, X, dt)
        mc = oracle.prune(Wc.reshape(12, -1), dt, BP, 4, 2, 3.0, 3, 3)
        yc = oracle.masked_conv2d(Wc, mc, x, dt, pad=(1, 1), stride=(2, 1))
        return m, y, mc, yc

    many = run()
    oracle.set_threads(1)
    try:
        one = run()
    finally:
        oracle.set_threads(n)
    for a, b in zip(many, one):
        assert np.array_equal(a, b)
