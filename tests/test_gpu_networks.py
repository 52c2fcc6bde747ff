"""GPU parity of the network workloads' pruned layers at their own shapes.

Selected layers of the VGG-16 workload (CIFAR-10 shape, batch 256, fp16) and
of the ResNet-50 workload (ImageNet shape, batch 64, bf16) are pruned, packed
and run through bp_conv2d / bp_gemm on their whole batch, as the workload
benchmark runs them.  Masks and column lists must equal the oracle's; the
outputs of the first and the last image (all outputs of the FC layers) must
match the oracle's masked direct convolution / masked GEMM within tolerance.

The layers cover every im2col path: plane-staged 3x3 (32x32 .. 4x4 planes),
image-group 3x3 (14x14 and 7x7 planes), threads along the rows (2x2 planes,
stride-2 3x3, 1x1 on small planes and strided 1x1), the per-plane 1x1 copy
(56x56), and both FC layers (a partial row-block, a partial last block).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2111_11581_gb300 import bp, inputs
from tests._util import assert_close, dev16, host_bits

pytestmark = pytest.mark.gpu

_VGG = {l.name: l for l in inputs.vgg16_cifar()}
_RN = {l.name: l for l in inputs.resnet50_imagenet()}

LAYERS = [("vgg16", _VGG[n], bp.F16) for n in ("conv2", "conv4", "conv7", "conv8", "conv12",
                                                "fc")] + \
         [("resnet50", _RN[n], bp.BF16) for n in ("s1b1_1x1a", "s1b1_3x3", "s2b1_3x3",
                                                   "s2b1_down", "s3b2_3x3", "s3b2_1x1a",
                                                   "s4b2_3x3", "s4b1_1x1b", "fc")]


@pytest.mark.parametrize("net,layer,dtype", LAYERS, ids=[f"{n}_{l.name}" for n, l, _ in LAYERS])
def test_network_layer_matches_oracle(net, layer, dtype):
    W = inputs.layer_weight(layer, dtype)
    x = inputs.layer_input(layer, dtype)
    b = inputs.layer_bias(layer)
    lay = bp.layout(layer.scheme, dtype, layer.M, layer.K, layer.bm, layer.bk, layer.kh, layer.kw)
    Wd = dev16(W.reshape(layer.M, -1), dtype)
    mask = bp.prune(lay, Wd, layer.rate)
    torch.cuda.synchronize()
    ref_mask = oracle.prune(W.reshape(layer.M, -1), dtype, layer.scheme, layer.bm, layer.bk,
                            layer.rate, layer.kh, layer.kw)
    got_mask = mask.cpu().numpy()
    assert (got_mask == ref_mask).all(), f"{int((got_mask != ref_mask).sum())} mask bytes differ"
    pw = bp.pack(lay, Wd, mask)
    _, col_idx, _ = oracle.pack(W.reshape(layer.M, -1), ref_mask, layer.bm)
    assert (pw.col_idx.cpu().numpy() == col_idx).all()
    bd = torch.from_numpy(b).cuda() if b is not None else None
    xd = dev16(x, dtype)
    if layer.kind == "conv":
        pad, stride = (layer.pad, layer.pad), (layer.stride, layer.stride)
        out = bp.conv2d(pw, xd, pad=pad, stride=stride, bias=bd, relu=layer.relu)
        torch.cuda.synchronize()
        assert bp.device_status() == bp.OK
        idx = [0, layer.N - 1]
        ref = oracle.masked_conv2d(W, ref_mask, x[idx], dtype, pad=pad, stride=stride, bias=b,
                                   relu=layer.relu)
        assert_close(host_bits(out)[idx], ref, dtype, f"{net} {layer.name}")
    else:
        out = bp.gemm(pw, xd, bias=bd, relu=layer.relu)
        torch.cuda.synchronize()
        assert bp.device_status() == bp.OK
        ref = oracle.masked_gemm(W, ref_mask, x, dtype, bias=b, relu=layer.relu)
        assert_close(host_bits(out), ref, dtype, f"{net} {layer.name}")
