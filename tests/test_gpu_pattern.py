"""GPU parity of bp_prune_pattern (kernel patterns + connectivity pruning of
3x3 layers) against the oracle, bit for bit, and of the convolution of a
pattern-pruned layer (packed with one list per filter) against the oracle."""
import numpy as np
import pytest
import torch

import oracle
from paper_2111_11581_gb300 import bp, inputs
from tests._util import assert_close, dev16, host_bits

pytestmark = pytest.mark.gpu
PUN = bp.BLOCK_PUNCHED

CASES = [
    # dtype, F, C, rate, patterns
    (bp.F16, 64, 32, 2.25, None),                 # patterns only, every kernel kept
    (bp.BF16, 128, 128, 4.0, None),
    (bp.F16, 96, 40, 8.0, None),
    (bp.BF16, 130, 70, 12.0, None),               # odd sizes, T not a round fraction
    (bp.F16, 32, 16, 5.0, (0b000011011, 0b110110000, 0b101010001, 0b100010101)),
]


@pytest.mark.parametrize("case", CASES, ids=lambda c: f"d{c[0]}_{c[1]}x{c[2]}_r{c[3]:g}_p{0 if c[4] is None else len(c[4])}")
def test_prune_pattern_bit_exact(case):
    dtype, F, C, rate, pats = case
    pats = bp.DEFAULT_PATTERNS if pats is None else pats
    W = inputs.normal((F, C, 3, 3), 0.05, dtype, seed=F + 7 * C)
    lay = bp.layout(PUN, dtype, F, C * 9, 8, 4, 3, 3)
    mask = bp.prune_pattern(lay, dev16(W.reshape(F, -1), dtype), rate, pats)
    torch.cuda.synchronize()
    ref = oracle.prune_pattern(W, dtype, rate, np.array(pats, np.uint16))
    got = mask.cpu().numpy()
    assert (got == ref).all(), f"{int((got != ref).sum())} mask bytes differ"


def test_default_patterns_match_the_oracle_set():
    assert list(bp.DEFAULT_PATTERNS) == [int(p) for p in oracle.DEFAULT_PATTERNS]


@pytest.mark.parametrize("rate", [4.0, 8.0])
def test_pattern_pruned_conv(rate):
    dtype, Nb, C, F, H = bp.F16, 4, 32, 48, 12
    W = inputs.normal((F, C, 3, 3), 0.1, dtype, seed=21)
    x = inputs.normal((Nb, C, H, H), 1.0, dtype, seed=22)
    b = inputs.bias(F, 0.1, 23)
    lay = bp.layout(PUN, dtype, F, C * 9, 8, 4, 3, 3)
    Wd = dev16(W.reshape(F, -1), dtype)
    mask = bp.prune_pattern(lay, Wd, rate)
    # filters keep different (channel, position) columns: one list per filter
    pw = bp.pack(bp.layout(PUN, dtype, F, C * 9, 1, 1, 3, 3), Wd, mask)
    y = bp.conv2d(pw, dev16(x, dtype), pad=(1, 1), bias=torch.from_numpy(b).cuda(), relu=True)
    torch.cuda.synchronize()
    assert bp.device_status() == bp.OK
    ref = oracle.masked_conv2d(W, mask.cpu().numpy(), x, dtype, pad=(1, 1),
                               bias=b, relu=True)
    assert_close(host_bits(y), ref, dtype, "bp_conv2d on a pattern mask")
