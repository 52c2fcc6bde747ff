"""GPU parity of bp_prune / bp_pack_size / bp_pack against the CPU oracle:
masks, rb_ptr, col_idx and values must match bit for bit, and the tiled
device image must decode back to the same weights and column lists."""
import numpy as np
import pytest
import torch

import oracle
from paper_2111_11581_gb300 import bp, inputs
from tests._util import dev16

pytestmark = pytest.mark.gpu
BB, BP_ = bp.BLOCK_BASED, bp.BLOCK_PUNCHED

CASES = [
    # scheme, dtype, M, K, kh, kw, bm, bk, rate
    (BB, bp.F16, 512, 512, 1, 1, 16, 16, 4.0),            # FC 512x512, keep 4 of 16
    (BP_, bp.F16, 128, 128 * 9, 3, 3, 8, 4, 3.0),         # 3x3 CONV, keep 3 of 9
    (BP_, bp.F16, 256, 128 * 9, 3, 3, 8, 4, 8.0),         # VGG layer: base 1 + extras
    (BP_, bp.BF16, 64, 64 * 9, 3, 3, 16, 8, 8.0),         # ResNet 3x3 blocks
    (BB, bp.BF16, 256, 64, 1, 1, 32, 32, 8.0),            # ResNet 1x1 reduce
    (BB, bp.BF16, 10, 512, 1, 1, 16, 16, 8.0),            # FC 512->10, one partial row-block
    (BB, bp.BF16, 1000, 2048, 1, 1, 32, 32, 6.0),         # FC 2048->1000, partial last block
    (BB, bp.BF16, 768, 3072, 1, 1, 128, 8, 16.0),         # bk*keep < 1: all kept units are extras
    (BB, bp.F16, 100, 96, 1, 1, 16, 10, 8.0 / 3.0),       # partial row/col blocks, base + extras
    (BB, bp.F16, 64, 80, 1, 1, 1, 1, 3.0),                # unstructured special case
    (BB, bp.BF16, 48, 256, 1, 1, 48, 8, 4.0),             # structured special case (bm = M)
    (BB, bp.BF16, 384, 256, 1, 1, 128, 32, 2.0),          # bm = 128 (weight-as-A tiles)
    (BB, bp.F16, 512, 192, 1, 1, 256, 16, 4.0),           # bm = 256
    (BP_, bp.F16, 24, 5 * 49, 7, 7, 8, 2, 5.0),           # 7x7 kernels, partial channel block
]


def _ids(c):
    return f"s{c[0]}_d{c[1]}_{c[2]}x{c[3]}_k{c[4]}{c[5]}_b{c[6]}x{c[7]}_r{c[8]:.3g}"


@pytest.mark.parametrize("case", CASES, ids=_ids)
def test_prune_and_pack_bit_exact(case):
    scheme, dtype, M, K, kh, kw, bm, bk, rate = case
    W = inputs.normal((M, K), 0.05, dtype, seed=M * 7 + K)
    lay = bp.layout(scheme, dtype, M, K, bm, bk, kh, kw)
    Wd = dev16(W, dtype)
    mask = bp.prune(lay, Wd, rate)
    torch.cuda.synchronize()
    ref_mask = oracle.prune(W, dtype, scheme, bm, bk, rate, kh, kw)
    got = mask.cpu().numpy()
    assert (got == ref_mask).all(), f"{int((got != ref_mask).sum())} mask bytes differ"

    pw = bp.pack(lay, Wd, mask)
    rb_ptr, col_idx, values = oracle.pack(W, ref_mask, bm)
    assert (pw.rb_ptr.cpu().numpy() == rb_ptr).all()
    assert (pw.col_idx.cpu().numpy() == col_idx).all()
    assert (pw.values.cpu().view(torch.int16).numpy().view(np.uint16) == values).all()
    _check_device_image(pw, ref_mask.astype(bool), W, M, K)


def _sw128(row, k):
    return (row >> 3) * 1024 + (row & 7) * 128 + (((k >> 3) ^ (row & 7)) << 4) + (k & 7) * 2


def _plan(l, bound=None):
    """Expected load plan of a chunk list: tile loads of 8 << lg rows for runs of
    8-position groups whose live entries are consecutive columns (a group with
    no live entry, padding, continues any run)."""
    w = np.zeros(16, np.int32)
    live = np.concatenate([[True], l[1:] != l[:-1]])
    first = l[::8]
    for g in range(8):
        for i in range(1, 8):
            q = 8 * g + i
            if live[q] and l[q] != first[g] + i:
                return w
    boxes, g = [], 0
    while g < 8:
        run = 1
        while g + run < 8 and (first[g + run] == first[g] + 8 * run or not live[8 * (g + run)]):
            run += 1
        lg = 3 if run >= 8 else 2 if run >= 4 else 1 if run >= 2 else 0
        if bound is not None and int(first[g]) + (8 << lg) > bound:
            return w                      # a load would pass the last listed row: gather
        boxes.append((int(first[g]), g | (lg << 4)))
        g += 1 << lg
    w[0] = len(boxes)
    desc = 0
    for b, (y, d) in enumerate(boxes):
        w[1 + b] = y
        desc |= d << (8 * b)
    w[9:11] = np.array([desc & 0xffffffff, desc >> 32], np.uint32).view(np.int32)
    # the loads cover the 64 list positions in order, and every live entry is
    # its load's first column plus its offset
    pos = 0
    for b, (y, d) in enumerate(boxes):
        assert (d & 7) == pos // 8
        rows = 8 << (d >> 4)
        seg = slice(pos, pos + rows)
        assert (l[seg][live[seg]] == (y + np.arange(rows))[live[seg]]).all()
        pos += rows
    assert pos == 64
    return w


def _check_section3(img, off, pw, mask, W, M, K):
    """The implicit convolution's section, from the mask and weights alone: per
    slab, the K-groups (64 channels c64*64 .. at kernel position (i, j)) any row
    keeps, listed position-major, one per chunk; records (c64 << 16 | i << 8 |
    j, TMA word); weight tiles K-major 128-byte swizzled with column u =
    channel 64 c64 + u (zero for channels past C and pruned weights)."""
    kh, kw = pw.lay.kh, pw.lay.kw
    khw = kh * kw
    C = K // khw
    C64 = -(-C // 64)
    S = -(-M // 128)
    cmax = S * C64 * khw
    tiles = off + (8 * (S + 1) + 255) // 256 * 256
    meta = tiles + cmax * 16384
    assert img.size == meta + cmax * 320
    kc3 = img[off: off + 8 * (S + 1)].view(np.int64)
    assert kc3[0] == 0
    offs = _sw128(np.arange(128)[:, None], np.arange(64)[None, :])
    for s in range(S):
        r0, r1 = 128 * s, min(128 * s + 128, M)
        keep = mask[r0:r1].reshape(r1 - r0, C, khw)
        groups = [(c64, pos // kw, pos % kw) for pos in range(khw) for c64 in range(C64)
                  if keep[:, 64 * c64: 64 * c64 + 64, pos].any()]
        assert kc3[s + 1] - kc3[s] == len(groups), (s, kc3[s + 1] - kc3[s], len(groups))
        rows = np.arange(r0, r1)
        for c, (c64, i, j) in enumerate(groups):
            rec = img[meta + (kc3[s] + c) * 320: meta + (kc3[s] + c + 1) * 320].view(np.int32)
            assert rec[0] == (c64 << 16) | (i << 8) | j and rec[64] == 1, (s, c)
            tw = np.zeros((128, 64), np.uint16)
            for u in range(64):
                ch = 64 * c64 + u
                if ch < C:
                    k = ch * khw + i * kw + j
                    tw[:r1 - r0, u] = np.where(mask[rows, k], W[rows, k], 0)
            base = tiles + (kc3[s] + c) * 16384
            dec = img[base: base + 16384].view(np.uint16)[offs // 2]
            assert (dec == tw).all(), (s, c)


def _check_device_image(pw, mask, W, M, K):
    """Decode the device image on the host, from the mask and weights alone:
    per 128-row slab, aligned 64-column blocks whose union of kept columns has
    at least 48 entries are listed whole, the other union columns follow in
    ascending order 64 per chunk (a partial last chunk repeats its last index);
    each chunk's 128 x 64 weight tile is K-major 128-byte swizzled and holds
    W where the row keeps the column (first occurrence of an index only)."""
    img = pw.dev.cpu().numpy()
    S = -(-M // 128)
    hdr = img[:8 * (S + 2)].view(np.int64)
    kc_ptr, Kc = hdr[:S + 1], int(hdr[S + 1])
    off = (8 * (S + 2) + 255) // 256 * 256
    tile_bytes = 128 * 128
    C = int(kc_ptr[-1])
    meta_off = off + C * tile_bytes
    meta2_off = meta_off + C * 320
    qmap_off = meta2_off + C * 320
    assert kc_ptr[0] == 0
    end = qmap_off + (4 * K + 15) // 16 * 16
    kh, kw = pw.lay.kh, pw.lay.kw
    if kh * kw > 1:
        _check_section3(img, (end + 255) // 256 * 256, pw, mask, W, M, K)
    else:
        assert img.size == end
    qmap = img[qmap_off: qmap_off + 4 * K].view(np.int32)
    offs = _sw128(np.arange(128)[:, None], np.arange(64)[None, :])
    listed = np.zeros(K, bool)
    all_lists = []
    for s in range(S):
        r0, r1 = 128 * s, min(128 * s + 128, M)
        union = mask[r0:r1].any(axis=0)
        lists = []
        for k0 in range(0, K, 64):
            if k0 + 64 <= K and union[k0:k0 + 64].sum() >= 48:
                lists.append(np.arange(k0, k0 + 64, dtype=np.int32))
        dense = np.zeros(K, bool)
        for l in lists:
            dense[l] = True
        rest = np.flatnonzero(union & ~dense).astype(np.int32)
        for c in range(0, rest.size, 64):
            l = np.full(64, rest[min(c + 63, rest.size - 1)], np.int32)
            seg = rest[c:c + 64]
            l[:seg.size] = seg
            lists.append(l)
        assert kc_ptr[s + 1] - kc_ptr[s] == len(lists), s
        for l in lists:
            listed[l] = True
        all_lists += [(int(kc_ptr[s]) + i, l) for i, l in enumerate(lists)]
        for i, l in enumerate(lists):
            c = int(kc_ptr[s]) + i
            base = off + c * tile_bytes
            rec = meta_off + c * 320
            assert (img[rec: rec + 256].view(np.int32) == l).all(), (s, i)
            plan = img[rec + 256: rec + 320].view(np.int32)
            assert (plan == _plan(l)).all(), (s, i, plan[:11], _plan(l)[:11])
            live = np.concatenate([[True], l[1:] != l[:-1]])
            want = np.zeros((128, 64), np.uint16)
            rows = np.arange(r0, r1)
            keep = mask[rows][:, l] & live[None, :]
            want[:r1 - r0] = np.where(keep, W[rows][:, l], 0)
            dec = img[base:base + tile_bytes].view(np.uint16)[offs // 2]
            assert (dec == want).all(), (s, i)
    # compacted coordinates: rank of each listed column; records with ranked lists
    want_q = np.where(listed, np.cumsum(listed) - 1, -1).astype(np.int32)
    assert Kc == int(listed.sum())
    assert (qmap == want_q).all()
    for c, l in all_lists:
        rec = meta2_off + c * 320
        l2 = want_q[l]
        assert (img[rec: rec + 256].view(np.int32) == l2).all(), c
        assert (img[rec + 256: rec + 320].view(np.int32) == _plan(l2, bound=Kc)).all(), c


def test_prune_ties_resolved_like_oracle():
    # every weight equal: all scores tie, so only the tie rule decides
    M, K = 64, 96
    W = oracle.round_to(np.full((M, K), 0.25), bp.F16)
    for scheme, kh, kw, bm, bk, rate in [(BB, 1, 1, 16, 16, 2.5), (BB, 1, 1, 1, 1, 7.0),
                                         (BP_, 3, 3, 8, 4, 8.0)]:
        Kx = K if scheme == BB else 8 * 9
        Wx = W[:, :Kx].copy()
        lay = bp.layout(scheme, bp.F16, M, Kx, bm, bk, kh, kw)
        mask = bp.prune(lay, dev16(Wx, bp.F16), rate).cpu().numpy()
        assert (mask == oracle.prune(Wx, bp.F16, scheme, bm, bk, rate, kh, kw)).all()


def test_prune_rejects_nonfinite():
    W = inputs.normal((32, 32), 1.0, bp.F16, seed=3)
    W[5, 7] = 0x7c00                     # +inf
    lay = bp.layout(BB, bp.F16, 32, 32, 8, 8)
    with pytest.raises(bp.BpError) as e:
        bp.prune(lay, dev16(W, bp.F16), 2.0)
    assert e.value.status == bp.ERR_NONFINITE


def test_pack_rejects_rows_that_disagree():
    lay = bp.layout(BB, bp.F16, 32, 32, 8, 8)
    mask = torch.ones((32, 32), dtype=torch.uint8, device="cuda")
    mask[3, 5] = 0                        # row 3 differs from row 0 of its row-block
    rb_ptr = torch.empty(5, dtype=torch.int64, device="cuda")
    st, *_ = bp.bp_pack_size(lay, mask.data_ptr(), rb_ptr.data_ptr(), 0)
    assert st == bp.ERR_INVALID_ARG


def test_rate_one_keeps_everything_and_all_pruned_layer():
    W = inputs.normal((40, 24), 1.0, bp.BF16, seed=4)
    lay = bp.layout(BB, bp.BF16, 40, 24, 8, 8)
    assert bp.prune(lay, dev16(W, bp.BF16), 1.0).cpu().numpy().all()
    # rate so high that T rounds to 0: nothing kept, every K'_rb = 0
    mask = bp.prune(lay, dev16(W, bp.BF16), 1e9)
    assert int(mask.sum()) == 0
    pw = bp.pack(lay, dev16(W, bp.BF16), mask)
    assert int(pw.c.nnz_cols) == 0
