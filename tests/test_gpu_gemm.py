"""GPU parity of bp_gemm against the CPU oracle (element by element, within
max |err| <= 1e-2 * max(1, |ref|)), on layers spanning several tiles with
ragged tails, both operand orientations, both dtypes, bias / ReLU, plus the
full-size FC layer and sampled rows of the full-size sweep shapes."""
import numpy as np
import pytest
import torch

import oracle
from paper_2111_11581_gb300 import bp, inputs
from tests._util import assert_close, dev16, host_bits

pytestmark = pytest.mark.gpu
BB = bp.BLOCK_BASED


def _layer(M, K, N, bm, bk, rate, dtype, seed, bias=False, relu=False):
    W = inputs.normal((M, K), 0.05, dtype, seed)
    X = inputs.uniform((K, N), -1.0, 1.0, dtype, seed + 1)
    b = inputs.bias(M, 0.1, seed + 2) if bias else None
    lay = bp.layout(BB, dtype, M, K, bm, bk)
    Wd = dev16(W, dtype)
    mask = bp.prune(lay, Wd, rate)
    pw = bp.pack(lay, Wd, mask)
    return W, X, b, mask.cpu().numpy(), pw


CASES = [
    # M, K, N, bm, bk, rate, dtype, bias, relu
    (64, 96, 64, 16, 16, 4.0, bp.F16, False, False),
    (100, 200, 130, 8, 8, 8.0 / 3.0, bp.BF16, True, True),      # ragged M, K, N; extras
    (256, 512, 300, 32, 32, 2.0, bp.F16, True, False),
    (200, 384, 257, 64, 16, 4.0, bp.BF16, False, True),
    (300, 256, 513, 128, 32, 4.0, bp.BF16, True, True),         # weight-as-A, partial row-block
    (256, 320, 1000, 128, 8, 16.0, bp.F16, False, False),       # extras only, weight-as-A
    (512, 256, 96, 256, 16, 2.0, bp.BF16, True, False),         # bm = 256 (two slabs)
    (160, 128, 200, 256, 32, 2.0, bp.F16, False, False),        # one partial 256-row block
    (72, 136, 33, 24, 8, 3.0, bp.BF16, True, True),             # bm not a power of two
    (33, 70, 7, 1, 1, 4.0, bp.F16, False, False),               # unstructured, N < 8
    (48, 512, 256, 48, 8, 8.0, bp.BF16, False, False),          # structured (bm = M)
    (128, 64, 1, 16, 16, 1.0, bp.F16, True, False),             # N = 1, nothing pruned
    # 16 row-blocks x 11 column tiles = 176 tiles: more than one wave of CTAs,
    # and the last column tile is ragged (100 of 256 tokens)
    (2048, 512, 2660, 128, 32, 4.0, bp.BF16, True, True),
]


@pytest.mark.parametrize("case", CASES, ids=lambda c: f"{c[0]}x{c[1]}x{c[2]}_b{c[3]}x{c[4]}_r{c[5]:.3g}_d{c[6]}")
def test_gemm_matches_oracle(case):
    M, K, N, bm, bk, rate, dtype, has_bias, relu = case
    W, X, b, mask, pw = _layer(M, K, N, bm, bk, rate, dtype, seed=M + K + N, bias=has_bias,
                               relu=relu)
    Xd = dev16(X, dtype, pad_last_to=8)
    bd = torch.from_numpy(b).cuda() if b is not None else None
    Y = bp.gemm(pw, Xd, bias=bd, relu=relu)
    torch.cuda.synchronize()
    assert bp.device_status() == bp.OK
    ref = oracle.masked_gemm(W, mask, X, dtype, bias=b, relu=relu)
    assert_close(host_bits(Y), ref, dtype, "bp_gemm")


def test_gemm_all_pruned_is_bias_only():
    M, K, N = 48, 64, 40
    W = inputs.normal((M, K), 1.0, bp.F16, 9)
    lay = bp.layout(BB, bp.F16, M, K, 16, 16)
    Wd = dev16(W, bp.F16)
    pw = bp.pack(lay, Wd, torch.zeros((M, K), dtype=torch.uint8, device="cuda"))
    X = dev16(inputs.uniform((K, N), -1, 1, bp.F16, 10), bp.F16)
    b = torch.linspace(-1, 1, M, device="cuda", dtype=torch.float32)
    Y = bp.gemm(pw, X, bias=b, relu=True)
    ref = torch.relu(b)[:, None].expand(M, N).to(torch.float16)
    assert torch.equal(Y, ref)


@pytest.mark.parametrize("dtype", [bp.F16, bp.BF16])
def test_fc512_full_size(dtype):
    """Single FC layer 512x512, 16x16 blocks keeping 4 of 16 columns, X 512x64."""
    L = inputs.fc512()
    W = inputs.layer_weight(L, dtype)
    X = inputs.layer_input(L, dtype)
    lay = bp.layout(BB, dtype, L.M, L.K, L.bm, L.bk)
    Wd = dev16(W, dtype)
    mask = bp.prune(lay, Wd, L.rate)
    pw = bp.pack(lay, Wd, mask)
    Y = bp.gemm(pw, dev16(X, dtype))
    ref = oracle.masked_gemm(W, mask.cpu().numpy(), X, dtype)
    assert_close(host_bits(Y), ref, dtype, "fc512")
    assert int(mask.sum()) == L.M * L.K // 4


def _uneven_mask(M, K, bm, bk, seed):
    """Block-based mask whose row-blocks keep different numbers of columns per
    block (0 .. bk), so K' differs from row-block to row-block."""
    rng = np.random.default_rng(seed)
    mask = np.zeros((M, K), dtype=np.uint8)
    for rb in range(0, M, bm):
        keep = (rb // bm * 3) % (bk + 1)
        for c in range(0, K, bk):
            w = min(bk, K - c)
            cols = rng.choice(w, size=min(keep, w), replace=False)
            mask[rb:rb + bm, c + cols] = 1
    return mask


SMALL_CASES = [
    # M, K, N, bm, bk, dtype, uneven: layers of the short CUDA-core path
    # (bm <= 32, at most 2^24 kept multiply-adds)
    (96, 320, 72, 16, 16, bp.F16, True),        # row-blocks keep 0 .. 16 columns per block
    (100, 1000, 45, 32, 8, bp.BF16, True),      # ragged M and N, K just under the staged limit
    (64, 2048, 40, 32, 32, bp.BF16, False),     # K past the staged limit: rows gathered by index
    (50, 1536, 33, 8, 16, bp.F16, True),        # K past the limit, uneven counts
]


@pytest.mark.parametrize("case", SMALL_CASES, ids=lambda c: f"{c[0]}x{c[1]}x{c[2]}_b{c[3]}x{c[4]}_u{int(c[6])}")
def test_short_path_matches_oracle(case):
    M, K, N, bm, bk, dtype, uneven = case
    W = inputs.normal((M, K), 0.05, dtype, M + K)
    X = inputs.uniform((K, N), -1.0, 1.0, dtype, N)
    b = inputs.bias(M, 0.1, 7)
    lay = bp.layout(BB, dtype, M, K, bm, bk)
    Wd = dev16(W, dtype)
    if uneven:
        mask = torch.from_numpy(_uneven_mask(M, K, bm, bk, M * N)).cuda()
    else:
        mask = bp.prune(lay, Wd, 8.0)
    pw = bp.pack(lay, Wd, mask)
    assert pw.c.nnz_vals * N <= 1 << 24
    Y = bp.gemm(pw, dev16(X, dtype, pad_last_to=8), bias=torch.from_numpy(b).cuda(), relu=True)
    torch.cuda.synchronize()
    assert bp.device_status() == bp.OK
    ref = oracle.masked_gemm(W, mask.cpu().numpy(), X, dtype, bias=b, relu=True)
    assert_close(host_bits(Y), ref, dtype, "short path")


SWEEP_SAMPLES = [
    # M, K, N, bm, bk, rate, dtype
    (4096, 4096, 4096, 128, 32, 4.0, bp.BF16),
    (4096, 4096, 4096, 8, 8, 16.0, bp.F16),
    (3072, 768, 8192, 16, 128, 2.0, bp.BF16),
    (768, 3072, 8192, 64, 16, 8.0, bp.F16),
]


@pytest.mark.parametrize("case", SWEEP_SAMPLES, ids=lambda c: f"{c[0]}x{c[1]}x{c[2]}_bm{c[3]}_bk{c[4]}_r{c[5]:g}")
def test_sweep_full_size_sampled_rows(case):
    """Full-size sweep shapes in the launch configuration of the benchmark; the
    oracle recomputes a sample of whole output rows (first, last, random)."""
    M, K, N, bm, bk, rate, dtype = case
    L = inputs.gemm_point(M, K, N, bm, bk, rate, dtype)
    W = inputs.layer_weight(L, dtype)
    X = inputs.layer_input(L, dtype)
    lay = bp.layout(BB, dtype, M, K, bm, bk)
    Wd = dev16(W, dtype)
    mask = bp.prune(lay, Wd, rate)
    pw = bp.pack(lay, Wd, mask)
    Xd = dev16(X, dtype)
    Y = bp.gemm(pw, Xd)
    torch.cuda.synchronize()
    assert bp.device_status() == bp.OK
    rng = np.random.default_rng(M + bm)
    rows = np.unique(np.concatenate([[0, M - 1, bm - 1, bm], rng.integers(0, M, 28)]))
    m_np = mask.cpu().numpy()
    ref = oracle.masked_gemm(W[rows], m_np[rows], X, dtype)
    got = host_bits(Y)[rows]
    assert_close(got, ref, dtype, "sweep rows")
    # the whole output against a second witness: cuBLAS on the masked weight (fp32)
    Wm = (Wd.float() * mask.float())
    ref2 = (Wm @ Xd.float())
    err = (Y.float() - ref2).abs()
    assert bool((err <= 1e-2 * ref2.abs().clamp_min(1.0)).all())


@pytest.mark.parametrize("case", [
    # few items, many chunks: every item split along k (8 items x 8 units)
    (512, 4096, 512, 128, 32, 4.0, bp.BF16, True, True),
    # 4 slabs x 1 column tile, small bm: the union lists are long
    (512, 2048, 200, 16, 8, 8.0, bp.F16, False, False),
], ids=lambda c: f"{c[0]}x{c[1]}x{c[2]}_b{c[3]}x{c[4]}")
def test_split_k_matches_oracle_and_unsplit(case):
    """The k-split product (fp32 partial sums added into an accumulator tile
    in the workspace) and the unsplit one both match the oracle, and a second
    split call on the same workspace does too (the kernel left its tiles and
    counters at zero)."""
    M, K, N, bm, bk, rate, dtype, has_bias, relu = case
    W, X, b, mask, pw = _layer(M, K, N, bm, bk, rate, dtype, seed=7 * M + K, bias=has_bias,
                               relu=relu)
    Xd = dev16(X, dtype, pad_last_to=8)
    bd = torch.from_numpy(b).cuda() if b is not None else None
    ws = bp.gemm_workspace(pw, N)
    assert ws is not None, "this shape should split"
    Ys = bp.gemm(pw, Xd, bias=bd, relu=relu, ws=ws)
    Yu = bp.gemm(pw, Xd, bias=bd, relu=relu, split=False)
    Ys2 = bp.gemm(pw, Xd, bias=bd, relu=relu, ws=ws)     # tiles and counters were reset
    torch.cuda.synchronize()
    assert bp.device_status() == bp.OK
    assert not ws.any(), "the kernel left the split workspace non-zero"
    ref = oracle.masked_gemm(W, mask, X, dtype, bias=b, relu=relu)
    assert_close(host_bits(Ys), ref, dtype, "split")
    assert_close(host_bits(Yu), ref, dtype, "unsplit")
    assert_close(host_bits(Ys2), ref, dtype, "split, second call")
