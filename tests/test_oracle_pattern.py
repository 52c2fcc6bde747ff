"""Pins of the pattern-based pruning oracle (kernel pattern pruning with a
fixed set of 4-entry 3x3 patterns, plus connectivity pruning; Sec. 2).  CPU
only."""
import itertools

import numpy as np
import pytest

import oracle
from paper_2111_11581_gb300 import inputs

F16, BF16 = 0, 1


def _energies(Wd, pats):
    F, C = Wd.shape[:2]
    sq = (Wd.reshape(F, C, 9) ** 2)
    bits = np.array([[(p >> b) & 1 for b in range(9)] for p in pats], bool)   # (P, 9)
    return np.einsum("fcp,qp->fcq", sq, bits.astype(np.float64))


def test_default_patterns_are_four_entry_and_contain_the_centre():
    for p in oracle.DEFAULT_PATTERNS:
        assert bin(int(p)).count("1") == 4 and (p >> 4) & 1
    assert len(set(int(p) for p in oracle.DEFAULT_PATTERNS)) == 8
    # together they cover all nine positions
    assert np.bitwise_or.reduce(oracle.DEFAULT_PATTERNS) == 0x1ff


@pytest.mark.parametrize("F,C,rate,dtype", [(16, 8, 2.25, F16), (24, 12, 4.0, BF16),
                                            (32, 16, 8.0, F16), (8, 5, 7.3, BF16)])
def test_pattern_choice_and_connectivity(F, C, rate, dtype):
    W = inputs.normal((F, C, 3, 3), 0.05, dtype, seed=F * C)
    Wd = oracle.to_double(W, dtype)
    mask, pat = oracle.prune_pattern(W, dtype, rate, return_patterns=True)
    e = _energies(Wd, oracle.DEFAULT_PATTERNS)                  # (F, C, P)
    # each kernel's pattern maximises its kept energy, ties to the lower index
    np.testing.assert_array_equal(pat.reshape(F, C), np.argmax(e, axis=2))
    best = e.max(axis=2).reshape(-1)
    T = int(np.floor(9 * F * C / (4 * rate) + 0.5))
    order = np.lexsort((np.arange(F * C), -best))
    kept = np.zeros(F * C, bool)
    kept[order[:T]] = True
    ref = np.zeros((F, C, 9), np.uint8)
    for g in np.flatnonzero(kept):
        f, c = divmod(g, C)
        p = int(oracle.DEFAULT_PATTERNS[pat[g]])
        ref[f, c] = [(p >> b) & 1 for b in range(9)]
    np.testing.assert_array_equal(mask, ref.reshape(F, 9 * C))
    assert mask.sum() == 4 * T


def _random_pattern_cases(n, seed):
    rng = np.random.default_rng(seed)
    all4 = [sum(1 << b for b in comb) for comb in itertools.combinations(range(9), 4)]
    out = []
    for _ in range(n):
        k = int(rng.integers(1, 17))
        pats = tuple(int(p) for p in rng.choice(all4, size=k, replace=False))
        out.append((int(rng.integers(1, 40)), int(rng.integers(1, 30)),
                    float(rng.choice([2.25, 3.0, 4.5, 6.0, 8.0, 9.0])), int(rng.integers(0, 2)),
                    pats))
    return out


@pytest.mark.parametrize("F,C,rate,dtype,pats", _random_pattern_cases(25, 8))
def test_pattern_choice_and_connectivity_random_sets(F, C, rate, dtype, pats):
    """Random layers and random pattern sets (1 to 16 distinct 4-entry masks):
    each kernel takes its highest kept-energy pattern (ties to the lower
    index), and the T = floor(9FC / (4r) + 0.5) kernels of highest kept energy
    survive (ties to the lower kernel index)."""
    W = inputs.normal((F, C, 3, 3), 0.05, dtype, seed=F * 100 + C)
    P = np.array(pats, np.uint16)
    mask, pat = oracle.prune_pattern(W, dtype, rate, patterns=P, return_patterns=True)
    e = _energies(oracle.to_double(W, dtype), P)
    np.testing.assert_array_equal(pat.reshape(F, C), np.argmax(e, axis=2))
    best = e.max(axis=2).reshape(-1)
    T = int(np.floor(9 * F * C / (4 * rate) + 0.5))
    kept = np.zeros(F * C, bool)
    kept[np.lexsort((np.arange(F * C), -best))[:T]] = True
    ref = np.zeros((F * C, 9), np.uint8)
    for g in np.flatnonzero(kept):
        ref[g] = [(int(P[pat[g]]) >> b) & 1 for b in range(9)]
    np.testing.assert_array_equal(mask, ref.reshape(F, C, 9).reshape(F, 9 * C))


def test_all_patterns_keep_the_four_largest_weights():
    # with every 4-entry pattern allowed, a kernel keeps its 4 largest magnitudes
    pats = np.array([sum(1 << b for b in comb) for comb in itertools.combinations(range(9), 4)],
                    np.uint16)
    W = inputs.normal((6, 5, 3, 3), 0.05, F16, seed=3)
    Wd = oracle.to_double(W, F16).reshape(6, 5, 9)
    mask = oracle.prune_pattern(W, F16, 2.25, patterns=pats).reshape(6, 5, 9)
    for f in range(6):
        for c in range(5):
            top = np.argsort(-(Wd[f, c] ** 2), kind="stable")[:4]
            assert set(np.flatnonzero(mask[f, c])) == set(top)


def test_hand_example():
    # one kernel: centre 4, N 3, E 2, S 1, corners 0.5; the T shape N,E,S + centre
    # (pattern 1) holds 16 + 9 + 4 + 1 = 30, more than any other default pattern
    k = np.zeros((1, 1, 3, 3), np.float32)
    k[0, 0] = [[0.5, 3, 0.5], [0, 4, 2], [0.5, 1, 0.5]]
    bits = k.astype(np.float16).view(np.uint16)
    mask, pat = oracle.prune_pattern(bits, F16, 2.25, return_patterns=True)
    assert pat[0] == 1
    np.testing.assert_array_equal(mask.reshape(3, 3), [[0, 1, 0], [0, 1, 1], [0, 1, 0]])


def test_rejections():
    W = inputs.normal((4, 2, 3, 3), 0.05, F16, seed=1)
    with pytest.raises(oracle.OracleError):
        oracle.prune_pattern(W, F16, 2.0)                       # below 9/4
    with pytest.raises(oracle.OracleError):
        oracle.prune_pattern(W, F16, 3.0, patterns=np.array([0b111], np.uint16))   # 3 entries
