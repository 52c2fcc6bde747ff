"""Rule-based pruning-scheme mapping on GB300 (Sec. 5.2): an offline latency
model measured with this library's own kernels, and the block-size rule.

Latency model (Sec. 5.2.1): for each layer setting (layer type -- 1x1, 3x3
and 5x5 CONV, FC -- filters, channels, feature-map size, compression rate)
and each candidate block size, a test model of 10 cascaded layers with that
setting is built from seeded synthetic weights (`bp_prune`, `bp_pack`) and
timed on the GPU (`bp_conv2d` / `bp_gemm`), L2 flushed before every run, the
median over the runs divided by 10; the entry is that latency divided by the
layer's dense MACs (the paper's normalisation).  Layers whose filters equal
their channels are truly cascaded (each layer reads the previous one's
output); the others read the same input.  Structured pruning -- the block that
spans the whole weight (all filters x all channels for block-punched, all
rows x all columns for block-based) -- is measured the same way as the
reference point.

Block-size rule (Sec. 5.2.2): given a latency threshold beta (0.2 in the
paper), the smallest block (by bm * bk, then bm) whose normalised latency is
at most (1 + beta) times the structured one is chosen; when none is, the
structured block is.

Scheme mapping (Fig. decision tree): depthwise 3x3 CONV layers are not pruned;
3x3 CONV layers get block-punched pruning (pattern-based pruning, the
alternative for large datasets, is `bp_prune_pattern`); the other layers get
the general scheme: block-punched for kernels larger than 1x1 (5x5), block-based
for 1x1 CONV and FC layers (their GEMM view).

The selection logic is plain host code (tested on CPU with given tables); only
`measure_setting` / `build_model` launch kernels.
"""
from __future__ import annotations

import dataclasses
import json
import statistics

STRUCTURED = (-1, -1)   # placeholder block size: the whole weight

# Candidate block sizes (bm, bk): filters x channels for block-punched,
# rows x columns for block-based.
PUNCHED_BLOCKS = [(4, 4), (8, 4), (8, 8), (16, 8), (16, 16), (32, 16), (32, 32), (64, 32),
                  (128, 32)]
BASED_BLOCKS = [(8, 8), (16, 16), (32, 32), (64, 32), (128, 32), (128, 64)]


@dataclasses.dataclass(frozen=True)
class Setting:
    """One layer setting of the latency model."""
    kind: str          # "conv1x1", "conv3x3", "conv5x5", "fc", "dw3x3"
    filters: int       # M (output channels / out-features)
    channels: int      # C (input channels / in-features)
    fmap: int          # feature-map height = width (CONV), tokens (FC)
    rate: float        # compression rate
    batch: int = 1

    def key(self) -> str:
        return f"{self.kind}:{self.filters}x{self.channels}:{self.fmap}:b{self.batch}:r{self.rate:g}"

    def macs(self) -> float:
        if self.kind == "fc":
            return float(self.filters) * self.channels * self.fmap
        return float(self.filters) * self.channels * ksize(self.kind) ** 2 * self.fmap * \
            self.fmap * self.batch


def ksize(kind: str) -> int:
    """Kernel height = width of a CONV layer type (1 for FC)."""
    return {"conv3x3": 3, "dw3x3": 3, "conv5x5": 5}.get(kind, 1)


def scheme_for(kind: str) -> str | None:
    """Pruning regularity for a layer type (decision tree of Sec. 5.2)."""
    if kind == "dw3x3":
        return None                     # depthwise 3x3: not pruned
    if kind in ("conv3x3", "conv5x5"):
        return "punched"
    return "based"


def candidates(kind: str, filters: int, channels: int) -> list[tuple[int, int]]:
    """Candidate blocks for a layer: those that fit inside the weight, plus the
    structured block."""
    sch = scheme_for(kind)
    if sch is None:
        return []
    k = ksize(kind) ** 2
    cols = channels * (k if sch == "based" else 1)
    blocks = PUNCHED_BLOCKS if sch == "punched" else BASED_BLOCKS
    return [(bm, bk) for bm, bk in blocks if bm <= filters and bk <= cols] + [STRUCTURED]


def select_block(table: dict, setting: Setting, beta: float = 0.2) -> tuple[int, int] | None:
    """The rule: smallest block (bm*bk, then bm) whose normalised latency is
    within (1 + beta) of structured pruning's; structured if none is; None for
    layers that are not pruned.  `table` maps setting keys to
    {"bm x bk" or "structured": normalised latency}."""
    if scheme_for(setting.kind) is None:
        return None
    row = table[setting.key()]
    ref = row["structured"]
    ok = []
    for name, lat in row.items():
        if name == "structured":
            continue
        bm, bk = (int(v) for v in name.split("x"))
        if lat <= (1.0 + beta) * ref:
            ok.append((bm * bk, bm, bk))
    if not ok:
        return STRUCTURED
    _, bm, bk = min(ok)
    return (bm, bk)


def block_name(b: tuple[int, int]) -> str:
    return "structured" if b == STRUCTURED else f"{b[0]}x{b[1]}"


# ------------------------------------------------------------------ measurement (GPU)
def measure_setting(setting: Setting, blocks=None, reps: int = 100, seed: int = 0,
                    depth: int = 10) -> dict:
    """Normalised latency (seconds per dense MAC) of each candidate block for
    one setting: a test model of `depth` layers with the setting (seeded
    N(0, 0.05) weights pruned at setting.rate and packed), cascaded when the
    layer keeps its channel count; per run L2 is flushed (a 256 MiB write read
    back) and the `depth` launches are timed with CUDA events; the median over
    `reps` runs (after 3 warm-up runs), divided by `depth`, then by the
    layer's dense MACs.  Returns {"bm x bk" / "structured": latency / MACs}."""
    import torch

    from . import bp, inputs

    dt = bp.BF16
    sch = scheme_for(setting.kind)
    kk = ksize(setting.kind)
    M, C = setting.filters, setting.channels
    K = C * kk * kk
    pad = (kk // 2, kk // 2)
    blocks = candidates(setting.kind, M, C) if blocks is None else blocks
    Ws = [inputs.as_torch(inputs.normal((M, K), 0.05, dt, seed + 17 * i), dt).cuda()
          for i in range(depth)]
    if setting.kind == "fc":
        x = inputs.as_torch(inputs.uniform((K, setting.fmap), -1.0, 1.0, dt, seed + 1), dt).cuda()
    else:
        x = inputs.as_torch(inputs.normal((setting.batch, C, setting.fmap, setting.fmap), 1.0, dt,
                                          seed + 1), dt).cuda()
    cascade = M == C
    flush = torch.empty(64 << 20, dtype=torch.float32, device="cuda")
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    out = {}
    for b in blocks:
        if b == STRUCTURED:
            bm, bk = M, (C if sch == "punched" else K)
        else:
            bm, bk = b
        if sch == "punched":
            lay = bp.layout(bp.BLOCK_PUNCHED, dt, M, K, bm, bk, kk, kk)
        else:
            lay = bp.layout(bp.BLOCK_BASED, dt, M, K, bm, bk)
        pws = [bp.pack(lay, W, bp.prune(lay, W, setting.rate)) for W in Ws]
        if setting.kind == "fc":
            wss = [bp.gemm_workspace(pw, setting.fmap) for pw in pws]
            ys = [bp.gemm(pw, x, ws=ws, split=ws is not None) for pw, ws in zip(pws, wss)]

            def run():
                h = x
                for pw, ws, y in zip(pws, wss, ys):
                    bp.gemm(pw, h, out=y, ws=ws, split=ws is not None)
                    h = y if cascade else x
        else:
            wss = [bp.conv2d_workspace(pw, tuple(x.shape), pad) for pw in pws]
            ys = [bp.conv2d(pw, x, pad=pad, ws=ws) for pw, ws in zip(pws, wss)]

            def run():
                h = x
                for pw, ws, y in zip(pws, wss, ys):
                    bp.conv2d(pw, h, pad=pad, out=y, ws=ws)
                    h = y if cascade else x
        for _ in range(3):
            run()
        ts = []
        for _ in range(reps):
            flush.zero_()
            flush.sum()
            ev[0].record()
            run()
            ev[1].record()
            torch.cuda.synchronize()
            ts.append(ev[0].elapsed_time(ev[1]) * 1e-3 / depth)
        if bp.device_status() != bp.OK:
            raise RuntimeError("kernel watchdog fired while measuring " + setting.key())
        out[block_name(b)] = statistics.median(ts) / setting.macs()
        del pws, ys
    return out


def build_model(settings, reps: int = 100, depth: int = 10) -> dict:
    """The latency model: {setting key: {block: normalised latency}}."""
    return {s.key(): measure_setting(s, reps=reps, depth=depth) for s in settings}


def default_settings() -> list[Setting]:
    """The grid: 1x1, 3x3 and 5x5 CONV layers on ResNet-like (feature map,
    channels) pairs 56/64, 28/128, 14/256, 7/512 (batch 32; 1x1 layers expand
    4x, the others keep their channels), and the FC shapes of the workloads
    (ResNet-50's 2048 -> 1000 over 64 images, BERT-base's 768 -> 3072 over 8192
    tokens), each at compression rates 2x, 4x and 8x (the workloads' rates)."""
    s = []
    for rate in (2.0, 4.0, 8.0):
        for fm, ch in ((56, 64), (28, 128), (14, 256), (7, 512)):
            s.append(Setting("conv3x3", ch, ch, fm, rate, batch=32))
            s.append(Setting("conv5x5", ch, ch, fm, rate, batch=32))
            s.append(Setting("conv1x1", 4 * ch, ch, fm, rate, batch=32))
        s.append(Setting("fc", 1000, 2048, 64, rate))
        s.append(Setting("fc", 3072, 768, 8192, rate))
    return s


def save(model: dict, path: str):
    with open(path, "w") as f:
        json.dump(model, f, indent=1, sort_keys=True)
