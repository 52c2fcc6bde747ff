"""Rule-based pruning-scheme mapping on GB300 (Sec. 5.2): an offline latency
model measured with this library's own kernels, and the block-size rule.

Latency model (Sec. 5.2.1): for each layer setting (layer type, filters,
channels, feature-map size, compression rate) and each candidate block size,
prune a seeded synthetic weight with `bp_prune`, pack it, and time the layer
(`bp_conv2d` or `bp_gemm`) on the GPU; the entry is the latency divided by the
layer's dense MACs (the paper's normalisation).  Structured pruning -- the
block that spans the whole weight (all filters x all channels for
block-punched, all rows x all columns for block-based) -- is measured the
same way as the reference point.

Block-size rule (Sec. 5.2.2): given a latency threshold beta (0.2 in the
paper), the smallest block (by bm * bk, then bm) whose normalised latency is
at most (1 + beta) times the structured one is chosen; when none is, the
structured block is.

Scheme mapping (Fig. decision tree): depthwise 3x3 CONV layers are not pruned;
3x3 CONV layers get block-punched pruning (pattern-based pruning, the
alternative for large datasets, is not built); every other CONV and FC layer
gets block-based pruning.

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
    kind: str          # "conv3x3", "conv1x1", "fc", "dw3x3"
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
        k = 9 if self.kind == "conv3x3" else 1
        return float(self.filters) * self.channels * k * self.fmap * self.fmap * self.batch


def scheme_for(kind: str) -> str | None:
    """Pruning regularity for a layer type (decision tree of Sec. 5.2)."""
    if kind == "dw3x3":
        return None                     # depthwise 3x3: not pruned
    if kind == "conv3x3":
        return "punched"
    return "based"


def candidates(kind: str, filters: int, channels: int) -> list[tuple[int, int]]:
    """Candidate blocks for a layer: those that fit inside the weight, plus the
    structured block."""
    sch = scheme_for(kind)
    if sch is None:
        return []
    k = (9 if kind == "conv3x3" else 1)
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
def measure_setting(setting: Setting, blocks=None, reps: int = 10, seed: int = 0) -> dict:
    """Normalised latency (seconds per dense MAC) of each candidate block for
    one setting: prune a seeded N(0, 0.05) weight at setting.rate, pack, and
    time the layer call (CUDA events, median of `reps` after 3 warm-ups).
    Returns {"bm x bk" / "structured": latency / MACs}."""
    import torch

    from . import bp, inputs

    dt = bp.BF16
    sch = scheme_for(setting.kind)
    k = 9 if setting.kind == "conv3x3" else 1
    M, C = setting.filters, setting.channels
    K = C * k
    blocks = candidates(setting.kind, M, C) if blocks is None else blocks
    W = inputs.normal((M, K), 0.05, dt, seed)
    Wd = inputs.as_torch(W, dt).cuda()
    if setting.kind == "fc":
        x = inputs.as_torch(inputs.uniform((K, setting.fmap), -1.0, 1.0, dt, seed + 1), dt).cuda()
    else:
        x = inputs.as_torch(inputs.normal((setting.batch, C, setting.fmap, setting.fmap), 1.0, dt,
                                          seed + 1), dt).cuda()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    out = {}
    for b in blocks:
        if b == STRUCTURED:
            bm, bk = M, (C if sch == "punched" else K)
        else:
            bm, bk = b
        if sch == "punched":
            lay = bp.layout(bp.BLOCK_PUNCHED, dt, M, K, bm, bk, 3, 3)
        else:
            lay = bp.layout(bp.BLOCK_BASED, dt, M, K, bm, bk)
        mask = bp.prune(lay, Wd, setting.rate)
        pw = bp.pack(lay, Wd, mask)
        if setting.kind == "fc":
            ws = bp.gemm_workspace(pw, setting.fmap)
            y = bp.gemm(pw, x, ws=ws, split=ws is not None)
            fn = lambda: bp.gemm(pw, x, out=y, ws=ws, split=ws is not None)  # noqa: E731
        else:
            pad = (1, 1) if setting.kind == "conv3x3" else (0, 0)
            ws = bp.conv2d_workspace(pw, tuple(x.shape), pad)
            y = bp.conv2d(pw, x, pad=pad, ws=ws)
            fn = lambda: bp.conv2d(pw, x, pad=pad, out=y, ws=ws)  # noqa: E731
        for _ in range(3):
            fn()
        ts = []
        for _ in range(reps):
            ev[0].record()
            fn()
            ev[1].record()
            torch.cuda.synchronize()
            ts.append(ev[0].elapsed_time(ev[1]) * 1e-3)
        if bp.device_status() != bp.OK:
            raise RuntimeError("kernel watchdog fired while measuring " + setting.key())
        out[block_name(b)] = statistics.median(ts) / setting.macs()
    return out


def build_model(settings, reps: int = 10) -> dict:
    """The latency model: {setting key: {block: normalised latency}}."""
    return {s.key(): measure_setting(s, reps=reps) for s in settings}


def default_settings() -> list[Setting]:
    """The grid of the paper's E2 latency study on ResNet-like shapes (Sec. 6.2):
    1x1 and 3x3 CONV at feature maps 56/28/14/7 with 64-512 channels, plus FC
    shapes; compression rate 8x (6x-8x are the rates of the workloads)."""
    s = []
    for fm, ch in ((56, 64), (28, 128), (14, 256), (7, 512)):
        s.append(Setting("conv3x3", ch, ch, fm, 8.0, batch=32))
        s.append(Setting("conv1x1", 4 * ch, ch, fm, 8.0, batch=32))
    s.append(Setting("fc", 1000, 2048, 64, 8.0))
    s.append(Setting("fc", 3072, 768, 8192, 8.0))
    return s


def save(model: dict, path: str):
    with open(path, "w") as f:
        json.dump(model, f, indent=1, sort_keys=True)
