"""Seeded synthetic inputs and workload shapes.

This module is shared by the tests, the benchmark, the CUDA path and the CPU
oracle, so it holds NO arithmetic of the method: it only draws random
tensors (as 16-bit float bit patterns in numpy uint16 arrays, plus fp32
biases) and lists layer shapes and pruning settings.

The paper's datasets (CIFAR-10, ImageNet, BERT token streams) and trained
weights are not available; these generators stand in for them with tensors of
the same shapes and the distributions stated for each workload:

* FC layer 512x512: W ~ N(0, 0.02), bm = bk = 16, keep 4 of 16; X 512x64 ~ U(-1, 1).
* 3x3 CONV: input 128x128x16x16 ~ N(0, 1), F = 128, Kaiming-normal weights
  (std sqrt(2 / fan_in)), bias ~ N(0, 0.01), ReLU, blocks 8 filters x 4
  channels, keep 3 of 9 positions.
* VGG-16 on 32x32x3 (CIFAR-10 shape), batch 256, fp16.
* ResNet-50 on 224x224x3 (ImageNet shape), batch 64, bf16.
* GEMM sweep 4096^3 and BERT-base FC shapes (3072x768, 768x3072, N = 8192).

Seeds follow s = 1000 * workload_number + layer_index (+ an offset per tensor).
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np
import torch

F16, BF16 = 0, 1
BLOCK_BASED, BLOCK_PUNCHED = 0, 1
_TORCH_DT = {F16: torch.float16, BF16: torch.bfloat16}


def dtype_name(dtype: int) -> str:
    return "bf16" if dtype == BF16 else "f16"


def _bits(t: torch.Tensor) -> np.ndarray:
    return t.contiguous().view(torch.int16).numpy().view(np.uint16)


def normal(shape, std: float, dtype: int, seed: int, mean: float = 0.0) -> np.ndarray:
    """Bit patterns of N(mean, std^2) samples rounded to fp16/bf16."""
    g = torch.Generator().manual_seed(int(seed))
    t = torch.empty(tuple(shape), dtype=torch.float32).normal_(mean, std, generator=g)
    return _bits(t.to(_TORCH_DT[dtype]))


def uniform(shape, lo: float, hi: float, dtype: int, seed: int) -> np.ndarray:
    """Bit patterns of U(lo, hi) samples rounded to fp16/bf16."""
    g = torch.Generator().manual_seed(int(seed))
    t = torch.empty(tuple(shape), dtype=torch.float32).uniform_(lo, hi, generator=g)
    return _bits(t.to(_TORCH_DT[dtype]))


def bias(n: int, std: float, seed: int) -> np.ndarray:
    g = torch.Generator().manual_seed(int(seed))
    return torch.empty(n, dtype=torch.float32).normal_(0.0, std, generator=g).numpy()


def kaiming_std(fan_in: int) -> float:
    """He initialisation scale for ReLU layers: sqrt(2 / fan_in)."""
    return math.sqrt(2.0 / fan_in)


def small_grid(shape, dtype: int, seed: int, scale_log2: int = 4, vmax: int = 32) -> np.ndarray:
    """Values k * 2^-scale_log2 with integer |k| <= vmax: their squares and sums
    of squares are exact in fp64 (for exact-arithmetic pins)."""
    g = torch.Generator().manual_seed(int(seed))
    k = torch.randint(-vmax, vmax + 1, tuple(shape), generator=g).to(torch.float32)
    return _bits((k * 2.0 ** -scale_log2).to(_TORCH_DT[dtype]))


def as_torch(bits: np.ndarray, dtype: int) -> torch.Tensor:
    """View uint16 bit patterns as a torch fp16/bf16 tensor (no copy of values)."""
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(_TORCH_DT[dtype])


# --------------------------------------------------------------------- workloads
@dataclass
class Layer:
    """One prunable layer of a workload (GEMM view M x K; conv if kh/kw/H given)."""
    name: str
    kind: str                 # "fc" or "conv"
    scheme: int               # BLOCK_BASED / BLOCK_PUNCHED / -1 = left dense
    M: int                    # out features / filters
    C: int                    # in features / channels
    kh: int = 1
    kw: int = 1
    bm: int = 1
    bk: int = 1
    rate: float = 1.0
    stride: int = 1
    pad: int = 0
    H: int = 0                # input spatial size (conv)
    W: int = 0
    N: int = 0                # tokens (fc) or batch (conv)
    seed: int = 0
    relu: bool = True
    has_bias: bool = True

    @property
    def K(self) -> int:
        return self.C * self.kh * self.kw

    @property
    def Ho(self) -> int:
        return (self.H + 2 * self.pad - self.kh) // self.stride + 1

    @property
    def Wo(self) -> int:
        return (self.W + 2 * self.pad - self.kw) // self.stride + 1

    @property
    def gemm_n(self) -> int:
        return self.N * self.Ho * self.Wo if self.kind == "conv" else self.N


def fc512() -> Layer:
    """Single FC layer 512x512, block-based 16x16, keep 4 of 16 (4x), X 512x64."""
    return Layer("fc512", "fc", BLOCK_BASED, 512, 512, bm=16, bk=16, rate=4.0, N=64,
                 seed=1000, relu=False, has_bias=False)


def conv3x3_128() -> Layer:
    """Single 3x3 CONV, N=128, C=F=128, 16x16, pad 1, punched 8x4, keep 3 of 9."""
    return Layer("conv3x3", "conv", BLOCK_PUNCHED, 128, 128, kh=3, kw=3, bm=8, bk=4, rate=3.0,
                 stride=1, pad=1, H=16, W=16, N=128, seed=2000)


def vgg16_cifar(batch: int = 256) -> list[Layer]:
    """VGG-16 on 32x32x3: 13 3x3 CONVs (first dense, rest punched 8f x 4c at 8x),
    2x2 max-pools after layers 2, 4, 7, 10, 13, FC 512->10 block-based 16x16 at 8x."""
    plan = [64, 64, "M", 128, 128, "M", 256, 256, 256, "M", 512, 512, 512, "M", 512, 512, 512,
            "M"]
    layers, c, hw, i = [], 3, 32, 0
    for v in plan:
        if v == "M":
            hw //= 2
            continue
        i += 1
        dense = i == 1
        layers.append(Layer(f"conv{i}", "conv", -1 if dense else BLOCK_PUNCHED, v, c, kh=3,
                            kw=3, bm=8, bk=4, rate=1.0 if dense else 8.0, stride=1, pad=1, H=hw,
                            W=hw, N=batch, seed=3000 + i))
        c = v
    layers.append(Layer("fc", "fc", BLOCK_BASED, 10, 512, bm=16, bk=16, rate=8.0, N=batch,
                        seed=3000 + 14, relu=False))
    return layers


VGG_POOL_AFTER = {"conv2", "conv4", "conv7", "conv10", "conv13"}


def resnet50_imagenet(batch: int = 64) -> list[Layer]:
    """ResNet-50 (v1.5 strides) on 224x224x3.  Stem 7x7/2 dense + 3x3/2 max-pool.
    3x3 CONVs block-punched 16 filters x 8 channels; 1x1 CONVs and the FC
    block-based 32x32.  Rates: 1x1 reduce 8x, 3x3 8x, 1x1 expand 2x,
    downsample 6x, FC 6x (mean over the 53 pruned layers = 6x)."""
    layers = [Layer("stem", "conv", -1, 64, 3, kh=7, kw=7, stride=2, pad=3, H=224, W=224,
                    N=batch, seed=4000)]
    cin, hw, idx = 64, 56, 0
    for si, (nblk, w) in enumerate(zip((3, 4, 6, 3), (64, 128, 256, 512))):
        for b in range(nblk):
            s = 2 if (b == 0 and si > 0) else 1
            pre = f"s{si + 1}b{b + 1}"
            idx += 1
            layers.append(Layer(pre + "_1x1a", "conv", BLOCK_BASED, w, cin, bm=32, bk=32,
                                rate=8.0, H=hw, W=hw, N=batch, seed=4000 + 10 * idx + 1))
            layers.append(Layer(pre + "_3x3", "conv", BLOCK_PUNCHED, w, w, kh=3, kw=3, bm=16,
                                bk=8, rate=8.0, stride=s, pad=1, H=hw, W=hw, N=batch,
                                seed=4000 + 10 * idx + 2))
            hwo = hw // s
            layers.append(Layer(pre + "_1x1b", "conv", BLOCK_BASED, 4 * w, w, bm=32, bk=32,
                                rate=2.0, H=hwo, W=hwo, N=batch, seed=4000 + 10 * idx + 3,
                                relu=False))
            if b == 0:
                layers.append(Layer(pre + "_down", "conv", BLOCK_BASED, 4 * w, cin, bm=32,
                                    bk=32, rate=6.0, stride=s, H=hw, W=hw, N=batch,
                                    seed=4000 + 10 * idx + 4, relu=False))
            cin, hw = 4 * w, hwo
    layers.append(Layer("fc", "fc", BLOCK_BASED, 1000, 2048, bm=32, bk=32, rate=6.0, N=batch,
                        seed=4999, relu=False))
    return layers


GEMM_SHAPES = ((4096, 4096, 4096), (3072, 768, 8192), (768, 3072, 8192))
SWEEP_BM = (8, 16, 32, 64, 128)
SWEEP_BK = (8, 16, 32, 128)
SWEEP_KEEP = (2, 4, 8, 16)      # keep fraction 1/x, i.e. rate x


def gemm_point(M, K, N, bm, bk, rate, dtype, seed=5000) -> Layer:
    return Layer(f"gemm{M}x{K}x{N}_bm{bm}_bk{bk}_r{rate:g}_{dtype_name(dtype)}", "fc",
                 BLOCK_BASED, M, K, bm=bm, bk=bk, rate=float(rate), N=N, seed=seed,
                 relu=False, has_bias=False)


def layer_weight(layer: Layer, dtype: int) -> np.ndarray:
    """Weight bits: GEMM view M x K (conv weights are OIHW, same memory)."""
    if layer.kind == "conv":
        std = kaiming_std(layer.K)
        return normal((layer.M, layer.C, layer.kh, layer.kw), std, dtype, layer.seed)
    if layer.name == "fc512" or layer.name.startswith("gemm"):
        return normal((layer.M, layer.K), 0.02, dtype, layer.seed)
    return normal((layer.M, layer.K), kaiming_std(layer.K), dtype, layer.seed)


def layer_input(layer: Layer, dtype: int) -> np.ndarray:
    """Activation bits: conv NCHW ~ N(0,1); FC/GEMM K x N ~ U(-1, 1)."""
    if layer.kind == "conv":
        return normal((layer.N, layer.C, layer.H, layer.W), 1.0, dtype, layer.seed + 500)
    return uniform((layer.K, layer.N), -1.0, 1.0, dtype, layer.seed + 500)


def layer_bias(layer: Layer):
    return bias(layer.M, 0.01, layer.seed + 700) if layer.has_bias else None
