"""GPU parity of bp_conv2d against the CPU oracle's masked direct convolution."""
import numpy as np
import pytest
import torch

import oracle
from paper_2111_11581_gb300 import bp, inputs
from tests._util import assert_close, dev16, host_bits

pytestmark = pytest.mark.gpu
BB, BPU = bp.BLOCK_BASED, bp.BLOCK_PUNCHED


def _run(F, C, kh, kw, Nb, H, W_, pad, stride, scheme, bm, bk, rate, dtype, seed, bias=True,
         relu=True, oracle_images=None):
    Wt = inputs.normal((F, C, kh, kw), inputs.kaiming_std(C * kh * kw), dtype, seed)
    x = inputs.normal((Nb, C, H, W_), 1.0, dtype, seed + 1)
    b = inputs.bias(F, 0.01, seed + 2) if bias else None
    lay = bp.layout(scheme, dtype, F, C * kh * kw, bm, bk, kh, kw)
    Wd = dev16(Wt.reshape(F, -1), dtype)
    mask = bp.prune(lay, Wd, rate)
    pw = bp.pack(lay, Wd, mask)
    xd = dev16(x, dtype)
    bd = torch.from_numpy(b).cuda() if b is not None else None
    out = bp.conv2d(pw, xd, pad=(pad, pad), stride=(stride, stride), bias=bd, relu=relu)
    torch.cuda.synchronize()
    assert bp.device_status() == bp.OK
    m = mask.cpu().numpy()
    nb = Nb if oracle_images is None else oracle_images
    ref = oracle.masked_conv2d(Wt, m, x[:nb], dtype, pad=(pad, pad), stride=(stride, stride),
                               bias=b, relu=relu)
    assert_close(host_bits(out)[:nb], ref, dtype, "bp_conv2d")
    return out, Wd, mask, xd, bd


CASES = [
    # F, C, kh, kw, Nb, H, W, pad, stride, scheme, bm, bk, rate, dtype
    (16, 8, 3, 3, 2, 8, 8, 1, 1, BPU, 8, 4, 3.0, bp.F16),
    (24, 12, 3, 3, 3, 11, 9, 1, 2, BPU, 8, 4, 8.0, bp.BF16),     # stride 2, odd sizes, extras
    (40, 20, 3, 3, 2, 14, 14, 1, 1, BPU, 16, 8, 8.0, bp.BF16),   # partial filter/channel blocks
    (64, 32, 1, 1, 2, 7, 7, 0, 1, BB, 32, 32, 8.0, bp.BF16),     # 1x1 as block-based
    (64, 48, 1, 1, 2, 14, 14, 0, 2, BB, 32, 32, 6.0, bp.F16),    # 1x1 stride 2 (downsample)
    (16, 3, 7, 7, 2, 20, 20, 3, 2, BPU, 8, 2, 4.0, bp.BF16),     # 7x7 stride 2
    (20, 8, 3, 3, 1, 5, 6, 2, 1, BB, 4, 16, 2.0, bp.F16),        # block-based on a 3x3 view
    (128, 16, 3, 3, 2, 9, 9, 1, 1, BPU, 128, 4, 3.0, bp.BF16),   # bm = 128 filters
    (8, 8, 3, 3, 4, 4, 4, 1, 1, BPU, 8, 4, 9.0, bp.F16),         # keep 1 of 9
    # plane-staged 3x3 im2col: several channels per block with a partial last
    # group (4x4: 128 channels per block, 200 = 128 + 72; 8x8: 32 per block)
    (32, 200, 3, 3, 3, 4, 4, 1, 1, BPU, 8, 4, 4.0, bp.BF16),
    (24, 40, 3, 3, 2, 8, 8, 1, 1, BPU, 8, 8, 3.0, bp.F16),
    (16, 12, 3, 3, 2, 28, 28, 1, 1, BPU, 8, 4, 2.0, bp.F16),     # pixel groups cross rows
    # TMA box stores of the NCHW output: two filter slabs, the second partial
    # (boxes clipped at F); 28x28 = 784 pixels, some 32-pixel groups cross images
    (200, 16, 3, 3, 3, 8, 8, 1, 1, BPU, 8, 4, 3.0, bp.BF16),
    (96, 64, 1, 1, 2, 28, 28, 0, 1, BB, 32, 32, 2.0, bp.BF16),
    # im2col with threads along the rows: stride-1 planes under 32 pixels
    (16, 8, 3, 3, 3, 5, 5, 1, 1, BPU, 8, 4, 3.0, bp.F16),
    (32, 16, 3, 3, 5, 2, 2, 1, 1, BPU, 8, 4, 8.0, bp.BF16),
    # planes of 32-127 pixels, H*W not a multiple of 8: image groups staged in
    # shared memory, 8-column groups spanning two images, a partial last group
    (24, 16, 3, 3, 11, 7, 7, 1, 1, BPU, 8, 4, 3.0, bp.BF16),
    (16, 24, 3, 3, 10, 6, 6, 1, 1, BPU, 8, 4, 3.0, bp.F16),
    # Ho*Wo dividing 32: each 32-pixel output group holds whole images, written
    # as 16-byte runs of 32 channels x Ho*Wo; few items, so the launches split
    (256, 64, 3, 3, 40, 2, 2, 1, 1, BPU, 8, 4, 8.0, bp.BF16),   # 2x2, two slabs
    (160, 32, 3, 3, 33, 1, 1, 1, 1, BPU, 8, 4, 3.0, bp.F16),    # 1x1 outputs, 32-row second slab
    (64, 24, 3, 3, 50, 1, 2, 1, 1, BPU, 8, 4, 3.0, bp.BF16),    # 1x2
    (96, 16, 3, 3, 45, 2, 4, 1, 1, BPU, 16, 8, 4.0, bp.F16),    # 2x4
]


@pytest.mark.parametrize("case", CASES, ids=lambda c: f"F{c[0]}C{c[1]}k{c[2]}s{c[8]}_b{c[10]}x{c[11]}_r{c[12]:g}")
def test_conv_matches_oracle(case):
    F, C, kh, kw, Nb, H, W_, pad, stride, scheme, bm, bk, rate, dtype = case
    _run(F, C, kh, kw, Nb, H, W_, pad, stride, scheme, bm, bk, rate, dtype, seed=F * C + H)


def test_conv3x3_full_size():
    """3x3 CONV, N=128, C=F=128, 16x16, pad 1, blocks 8 filters x 4 channels keep 3
    of 9 positions, bias, ReLU.  The oracle recomputes 16 of the 128 images; the
    whole batch is also checked against cuDNN on the masked weight."""
    L = inputs.conv3x3_128()
    out, Wd, mask, xd, bd = _run(L.M, L.C, 3, 3, L.N, L.H, L.W, 1, 1, BPU, L.bm, L.bk, L.rate,
                                 bp.F16, seed=L.seed, oracle_images=16)
    wm = (Wd.float() * mask.float()).reshape(L.M, L.C, 3, 3)
    ref = torch.relu(torch.nn.functional.conv2d(xd.float(), wm, bd, padding=1))
    err = (out.float() - ref).abs()
    assert bool((err <= 1e-2 * ref.abs().clamp_min(1.0)).all())
