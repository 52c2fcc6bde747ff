"""GPU parity of every pruned layer of the two network workloads at its own shape.

All 13 pruned layers of the VGG-16 workload (CIFAR-10 shape, batch 256, fp16:
12 block-punched 3x3 CONVs and the block-based FC 512 -> 10) and all 53
pruned layers of the ResNet-50 workload (ImageNet shape, batch 64, bf16:
block-punched 3x3 CONVs, block-based 1x1 CONVs, downsample CONVs and the FC)
are pruned, packed and run through bp_conv2d / bp_gemm on their whole batch,
as the workload benchmark runs them.  Per layer:

* the mask, rb_ptr, col_idx and the compact weight values equal the oracle's
  bit for bit (Sec. 4.1 pruning rule, Sec. 4.3 storage);
* the outputs of three images (the first, the last and one drawn from a
  seeded generator) of a CONV layer, and all outputs of an FC layer, match
  the oracle's masked direct convolution / masked GEMM within
  max |err| <= 1e-2 * max(1, |ref|).

The dense first layers (VGG conv1, the ResNet stem) are not pruned by the
workloads and have no library call to check.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2111_11581_gb300 import bp, inputs
from tests._util import assert_close, dev16, host_bits

pytestmark = pytest.mark.gpu

LAYERS = [("vgg16", l, bp.F16) for l in inputs.vgg16_cifar() if l.scheme >= 0] + \
         [("resnet50", l, bp.BF16) for l in inputs.resnet50_imagenet() if l.scheme >= 0]


def test_every_pruned_layer_is_listed():
    assert sum(1 for n, _, _ in LAYERS if n == "vgg16") == 13
    assert sum(1 for n, _, _ in LAYERS if n == "resnet50") == 53


@pytest.mark.parametrize("net,layer,dtype", LAYERS, ids=[f"{n}_{l.name}" for n, l, _ in LAYERS])
def test_network_layer_matches_oracle(net, layer, dtype):
    W = inputs.layer_weight(layer, dtype)
    Wg = W.reshape(layer.M, -1)
    lay = bp.layout(layer.scheme, dtype, layer.M, layer.K, layer.bm, layer.bk, layer.kh, layer.kw)
    Wd = dev16(Wg, dtype)
    mask = bp.prune(lay, Wd, layer.rate)
    pw = bp.pack(lay, Wd, mask)
    torch.cuda.synchronize()
    ref_mask = oracle.prune(Wg, dtype, layer.scheme, layer.bm, layer.bk, layer.rate, layer.kh,
                            layer.kw)
    got_mask = mask.cpu().numpy()
    assert (got_mask == ref_mask).all(), f"{int((got_mask != ref_mask).sum())} mask bytes differ"
    rb_ptr, col_idx, values = oracle.pack(Wg, ref_mask, layer.bm)
    assert (pw.rb_ptr.cpu().numpy() == rb_ptr).all(), "rb_ptr differs"
    assert (pw.col_idx.cpu().numpy() == col_idx).all(), "col_idx differs"
    assert (host_bits(pw.values) == values).all(), "packed values differ"

    x = inputs.layer_input(layer, dtype)
    b = inputs.layer_bias(layer)
    bd = torch.from_numpy(b).cuda() if b is not None else None
    xd = dev16(x, dtype, pad_last_to=8 if layer.kind == "fc" else 1)
    if layer.kind == "conv":
        pad, stride = (layer.pad, layer.pad), (layer.stride, layer.stride)
        out = bp.conv2d(pw, xd, pad=pad, stride=stride, bias=bd, relu=layer.relu)
        torch.cuda.synchronize()
        assert bp.device_status() == bp.OK
        rng = np.random.default_rng(layer.seed)
        idx = sorted({0, layer.N - 1, int(rng.integers(1, layer.N - 1))})
        ref = oracle.masked_conv2d(W, ref_mask, x[idx], dtype, pad=pad, stride=stride, bias=b,
                                   relu=layer.relu)
        assert_close(host_bits(out)[idx], ref, dtype, f"{net} {layer.name}")
    else:
        out = bp.gemm(pw, xd, bias=bd, relu=layer.relu)
        torch.cuda.synchronize()
        assert bp.device_status() == bp.OK
        ref = oracle.masked_gemm(W, ref_mask, x, dtype, bias=b, relu=layer.relu)
        assert_close(host_bits(out), ref, dtype, f"{net} {layer.name}")
