"""GPU parity of bp_prune_rows (row units of each block, ANDed into a mask)
against the oracle, bit for bit, and of the product of a row + column pruned
layer (packed with one list per row) against the oracle's masked GEMM."""
import numpy as np
import pytest
import torch

import oracle
from paper_2111_11581_gb300 import bp, inputs
from tests._util import assert_close, dev16, host_bits

pytestmark = pytest.mark.gpu
BB = bp.BLOCK_BASED

CASES = [
    # dtype, M, K, bm, bk, column rate, row rate
    (bp.F16, 256, 256, 16, 16, 2.0, 2.0),
    (bp.BF16, 100, 96, 16, 10, 8.0 / 3.0, 3.0),      # partial row- and column-blocks, extras
    (bp.BF16, 384, 512, 128, 32, 2.0, 2.0),          # the benchmark's block shape
    (bp.F16, 64, 80, 1, 1, 1.0, 4.0),                # 1x1 blocks: global magnitude pruning
    (bp.BF16, 48, 256, 48, 256, 1.0, 3.0),           # one block: whole rows
    (bp.F16, 130, 200, 64, 8, 4.0, 8.0),             # bk * keep < 1 for rows: extras only
]


def _ids(c):
    return f"d{c[0]}_{c[1]}x{c[2]}_b{c[3]}x{c[4]}_rc{c[5]:.3g}_rr{c[6]:.3g}"


@pytest.mark.parametrize("case", CASES, ids=_ids)
def test_prune_rows_bit_exact(case):
    dtype, M, K, bm, bk, rc, rr = case
    W = inputs.normal((M, K), 0.05, dtype, seed=M * 3 + K)
    lay = bp.layout(BB, dtype, M, K, bm, bk)
    Wd = dev16(W, dtype)
    mask = bp.prune(lay, Wd, rc)
    mask = bp.prune_rows(lay, Wd, rr, mask)
    torch.cuda.synchronize()
    ref = oracle.prune_rows(W, dtype, bm, bk, rr, mask=oracle.prune(W, dtype, 0, bm, bk, rc))
    got = mask.cpu().numpy()
    assert (got == ref).all(), f"{int((got != ref).sum())} mask bytes differ"
    # rows alone (an all-ones mask in)
    m2 = bp.prune_rows(lay, Wd, rr)
    torch.cuda.synchronize()
    assert (m2.cpu().numpy() == oracle.prune_rows(W, dtype, bm, bk, rr)).all()


@pytest.mark.parametrize("case", [(bp.BF16, 384, 512, 300, 128, 32, 2.0, 2.0),
                                  (bp.F16, 100, 96, 70, 16, 10, 8.0 / 3.0, 3.0)],
                         ids=lambda c: f"{c[1]}x{c[2]}x{c[3]}_b{c[4]}x{c[5]}")
def test_row_and_column_pruned_gemm(case):
    dtype, M, K, N, bm, bk, rc, rr = case
    W = inputs.normal((M, K), 0.05, dtype, seed=11 + M)
    X = inputs.uniform((K, N), -1.0, 1.0, dtype, seed=12 + M)
    b = inputs.bias(M, 0.1, 13)
    lay = bp.layout(BB, dtype, M, K, bm, bk)
    Wd = dev16(W, dtype)
    mask = bp.prune_rows(lay, Wd, rr, bp.prune(lay, Wd, rc))
    # rows of a row-block now keep different columns: one list per row
    pw = bp.pack(bp.layout(BB, dtype, M, K, 1, bk), Wd, mask)
    Y = bp.gemm(pw, dev16(X, dtype, pad_last_to=8), bias=torch.from_numpy(b).cuda(), relu=True)
    torch.cuda.synchronize()
    assert bp.device_status() == bp.OK
    ref = oracle.masked_gemm(W, mask.cpu().numpy(), X, dtype, bias=b, relu=True)
    assert_close(host_bits(Y), ref, dtype, "bp_gemm on a row + column mask")
