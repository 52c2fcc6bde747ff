"""Measurement builds of libbp: pipeline variants behind build switches, and the
per-stage timeline of the tensor-core product.

    python -m paper_2111_11581_gb300.variants time NAME:[DEFINE,...] ...
        builds one library per NAME with the given -D switches (e.g.
        `base: balance:BP_BALANCE`) and times each on
        the same workloads, every build in a process of its own:
        4096^3 bf16 at 128 x 32 blocks, keep 1/4 (the benchmark's layer),
        4096^3 at 8 x 64 blocks, keep 1/2 (whole 64-column blocks: TMA tile
        loads instead of gathers) and BERT-base 3072 x 768 over 8192 tokens at
        64 x 16 blocks, keep 1/8; four rotating activation sets, 400 launches.

    python -m paper_2111_11581_gb300.variants latency NAME:[DEFINE,...] ...
        the same builds, each timing single launches as the workload benchmark
        does (L2 flushed by a 256 MiB write, read back, then CUDA events around
        one call; median of 10): the 512 x 512 FC layer, the 3x3 CONV layer,
        two ResNet-50 1x1 layers and the 4096^3 layer.

    python -m paper_2111_11581_gb300.variants probe
        builds and runs probes/tc_rates.cu: tcgen05.mma 128 x N x 16 issued
        back to back from one thread (cycles per instruction for N = 256, 128,
        64, 16), TMA bulk copies from 1, 2 and 4 threads per SM (bytes per
        cycle an SM ingests), the stage ring without data (cycles per 64-column
        chunk for 2-6 stages, with and without the per-stage fences),
        back-to-back MMAs while other warps copy into shared memory (bulk or
        cp.async rows), and groups of four MMAs and a commit with the
        tensor-core thread's per-chunk work placed between them (barrier
        probes, fences, loads, descriptor arithmetic; other warps polling or
        copying meanwhile).

    python -m paper_2111_11581_gb300.variants trace [gemm|gemm8|conv3x3|resnet50:LAYER|vgg16:LAYER|fc512][+warm] [DEFINE ...]
        builds with BP_TRACE and prints CTA 0's clock64 timeline of one launch,
        L2 flushed before it, of the 4096^3 layer (bm=128 bk=32 at 4x; gemm8:
        bm=8 bk=64 at 2x; or of the 3x3 CONV layer: N=128, C=F=128, 16x16, or
        of one ResNet-50 / VGG-16 layer by name); with +warm, of the last of
        three back-to-back launches instead: per pipeline stage when the control
        thread and a gather group found it free, when the gather was issued,
        when the tensor-core thread saw the stage loaded and committed; per
        window when the control thread and the gather warps had its records;
        per item when the tensor-core thread had a free accumulator and when
        the epilogue saw it finished and had stored it; and the global-timer
        start and end of every CTA.

The switches (all off in the library `build()` makes): BP_TRACE (timeline),
BP_BALANCE (whole-item waves, then equal chunk ranges per CTA with fp32
partial tiles), BP_EPI_DIRECT (output boxes written back from shared memory
with plain stores instead of TMA stores), BP_NO_PDL (ordinary launches
instead of programmatic dependent ones).  Builds go to _build/variants/NAME next to the library.
"""
from __future__ import annotations

import concurrent.futures as cf
import ctypes
import os
import subprocess
import sys

from . import build as B

OUT = os.path.join(B.HERE, "_build", "variants")


def build_variant(name: str, defines) -> str:
    """libbp.so built with -D<define> for each define, into _build/variants/name."""
    out = os.path.join(OUT, name)
    os.makedirs(out, exist_ok=True)
    cc = B.nvcc()
    flags = B.ARCH + ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC",
                      "-I" + os.path.join(B.ROOT, "include"), "--expt-relaxed-constexpr"]
    flags += ["-D" + d for d in defines if d]

    def one(src):
        obj = os.path.join(out, os.path.basename(src) + ".o")
        r = subprocess.run([cc, *flags, "-c", src, "-o", obj], capture_output=True, text=True)
        if r.returncode:
            raise RuntimeError(f"nvcc failed on {src}:\n{r.stderr}")
        return obj

    with cf.ThreadPoolExecutor(max_workers=min(8, os.cpu_count() or 1)) as ex:
        objs = list(ex.map(one, B._sources()))
    lib = os.path.join(out, "libbp.so")
    subprocess.run([cc, *B.ARCH, "-shared", "-o", lib, *objs], check=True)
    return lib


TIME_CASES = [(4096, 4096, 4096, 128, 32, 4.0, "bf16"), (4096, 4096, 4096, 8, 64, 2.0, "bf16"),
              (3072, 768, 8192, 64, 16, 8.0, "f16")]


def _time_in_process(lib: str):
    import torch

    from . import bp, inputs
    bp.load(lib)
    res = []
    for (M, K, N, bm, bk, rate, d) in TIME_CASES:
        dt = bp.BF16 if d == "bf16" else bp.F16
        L = inputs.gemm_point(M, K, N, bm, bk, rate, dt)
        W = inputs.as_torch(inputs.layer_weight(L, dt), dt).cuda()
        sets = [torch.empty((K, N), dtype=W.dtype, device="cuda").uniform_(-1, 1)
                for _ in range(4)]
        lay = bp.layout(bp.BLOCK_BASED, dt, M, K, bm, bk)
        mask = bp.prune(lay, W, rate)
        pw = bp.pack(lay, W, mask)
        ws = bp.gemm_workspace(pw, N)
        Ys = [bp.gemm(pw, X, ws=ws) for X in sets]
        ref = (W.float() * mask.float()) @ sets[0].float()
        ok = bool(((Ys[0].float() - ref).abs() <= 1e-2 * ref.abs().clamp_min(1)).all())
        for i in range(20):
            bp.gemm(pw, sets[i % 4], out=Ys[i % 4], ws=ws)
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        n = 400
        e0.record()
        for i in range(n):
            bp.gemm(pw, sets[i % 4], out=Ys[i % 4], ws=ws)
        e1.record()
        torch.cuda.synchronize()
        us = e0.elapsed_time(e1) * 1000 / n
        res.append(f"{M}x{K}x{N} bm{bm} bk{bk} r{rate:g}: {us:.2f} us "
                   f"{2.0 * int(mask.sum()) * N / us * 1e-6:.1f} TFLOP/s ok={ok}")
    print(" | ".join(res), flush=True)


LATENCY_CASES = ["fc512", "conv3x3", "resnet50:s1b1_1x1b", "resnet50:s3b2_1x1a", "gemm"]


def _layer_call(workload: str):
    """(run, note) for one launch of a named layer, operands on the device."""
    import torch

    from . import bp, inputs
    if workload == "fc512":
        L, dt = inputs.fc512(), bp.F16
        W = inputs.as_torch(inputs.layer_weight(L, dt), dt).cuda()
        X = inputs.as_torch(inputs.layer_input(L, dt), dt).cuda()
        lay = bp.layout(bp.BLOCK_BASED, dt, L.M, L.K, L.bm, L.bk)
        pw = bp.pack(lay, W, bp.prune(lay, W, L.rate))
        Y = bp.gemm(pw, X)
        return lambda: bp.gemm(pw, X, out=Y)
    if workload == "gemm":
        dt = bp.BF16
        L = inputs.gemm_point(4096, 4096, 4096, 128, 32, 4.0, dt)
        W = inputs.as_torch(inputs.layer_weight(L, dt), dt).cuda()
        X = inputs.as_torch(inputs.layer_input(L, dt), dt).cuda()
        lay = bp.layout(bp.BLOCK_BASED, dt, L.M, L.K, L.bm, L.bk)
        pw = bp.pack(lay, W, bp.prune(lay, W, L.rate))
        ws = bp.gemm_workspace(pw, L.N)
        Y = bp.gemm(pw, X, ws=ws)
        return lambda: bp.gemm(pw, X, out=Y, ws=ws)
    if workload == "conv3x3":
        L, dt = inputs.conv3x3_128(), bp.F16
    else:
        name = workload.split(":", 1)[1]
        L, dt = [l for l in inputs.resnet50_imagenet() if l.name == name][0], bp.BF16
    W = inputs.as_torch(inputs.layer_weight(L, dt).reshape(L.M, -1), dt).cuda()
    X = inputs.as_torch(inputs.layer_input(L, dt), dt).cuda()
    lay = bp.layout(L.scheme, dt, L.M, L.K, L.bm, L.bk, L.kh, L.kw)
    pw = bp.pack(lay, W, bp.prune(lay, W, L.rate))
    pad, st = (L.pad, L.pad), (L.stride, L.stride)
    ws = bp.conv2d_workspace(pw, X.shape, pad, st)
    Y = bp.conv2d(pw, X, pad=pad, stride=st, ws=ws)
    return lambda: bp.conv2d(pw, X, pad=pad, stride=st, out=Y, ws=ws)


def _latency_in_process(lib: str):
    import statistics

    import torch

    from . import bp
    bp.load(lib)
    flush = torch.empty(256 * 2 ** 20 // 4, dtype=torch.float32, device="cuda")
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    res = []
    for w in LATENCY_CASES:
        run = _layer_call(w)
        ts = []
        for _ in range(12):
            flush.zero_()
            flush.sum()
            ev[0].record()
            run()
            ev[1].record()
            torch.cuda.synchronize()
            ts.append(ev[0].elapsed_time(ev[1]) * 1e3)
        res.append(f"{w}: {statistics.median(ts[2:]):.2f} us")
    print(" | ".join(res), flush=True)


def _trace_in_process(lib: str, workload: str):
    import numpy as np
    import torch

    # WORKLOAD+warm: the last of three back-to-back launches, no flush (code,
    # parameters and the packed image in L2, the start overlapping the previous
    # launch as in a timing loop)
    warm = workload.endswith("+warm")
    workload = workload.removesuffix("+warm")

    from . import bp, inputs
    L_ = bp.load(lib)
    L_.bp_debug_trace_read.restype = ctypes.c_int
    L_.bp_debug_trace_read.argtypes = [ctypes.c_void_p, ctypes.c_int]
    L_.bp_debug_trace_clear.restype = ctypes.c_int
    if workload == "fc512":
        L, dt = inputs.fc512(), bp.F16
        W = inputs.as_torch(inputs.layer_weight(L, dt), dt).cuda()
        X = inputs.as_torch(inputs.layer_input(L, dt), dt).cuda()
        lay = bp.layout(bp.BLOCK_BASED, dt, L.M, L.K, L.bm, L.bk)
        pw = bp.pack(lay, W, bp.prune(lay, W, L.rate))
        Y = bp.gemm(pw, X)
        run = lambda: bp.gemm(pw, X, out=Y)  # noqa: E731
    elif workload == "conv3x3" or workload.startswith(("resnet50:", "vgg16:")):
        if workload == "conv3x3":
            L, dt = inputs.conv3x3_128(), bp.F16
        elif workload.startswith("vgg16:"):
            name = workload.split(":", 1)[1]
            L, dt = [l for l in inputs.vgg16_cifar() if l.name == name][0], bp.F16
        else:
            name = workload.split(":", 1)[1]
            L, dt = [l for l in inputs.resnet50_imagenet() if l.name == name][0], bp.BF16
        W = inputs.as_torch(inputs.layer_weight(L, dt).reshape(L.M, -1), dt).cuda()
        X = inputs.as_torch(inputs.layer_input(L, dt), dt).cuda()
        lay = bp.layout(L.scheme, dt, L.M, L.K, L.bm, L.bk, L.kh, L.kw)
        pw = bp.pack(lay, W, bp.prune(lay, W, L.rate))
        pad, st = (L.pad, L.pad), (L.stride, L.stride)
        ws = bp.conv2d_workspace(pw, X.shape, pad, st)
        Y = bp.conv2d(pw, X, pad=pad, stride=st, ws=ws)
        run = lambda: bp.conv2d(pw, X, pad=pad, stride=st, out=Y, ws=ws)  # noqa: E731
    else:
        dt = bp.BF16
        L = (inputs.gemm_point(4096, 4096, 4096, 8, 64, 2.0, dt) if workload == "gemm8" else
             inputs.gemm_point(4096, 4096, 4096, 128, 32, 4.0, dt))
        W = inputs.as_torch(inputs.layer_weight(L, dt), dt).cuda()
        X = inputs.as_torch(inputs.layer_input(L, dt), dt).cuda()
        lay = bp.layout(bp.BLOCK_BASED, dt, L.M, L.K, L.bm, L.bk)
        pw = bp.pack(lay, W, bp.prune(lay, W, L.rate))
        ws = bp.gemm_workspace(pw, L.N)
        Y = bp.gemm(pw, X, ws=ws)
        run = lambda: bp.gemm(pw, X, out=Y, ws=ws)  # noqa: E731
    for _ in range(20):
        run()
    torch.cuda.synchronize()
    # as the workload benchmark times a launch: L2 flushed (a 256 MiB write,
    # read back) just before it
    flush = torch.empty(256 * 2 ** 20 // 4, dtype=torch.float32, device="cuda")
    flush.zero_()
    flush.sum()
    torch.cuda.synchronize()
    L_.bp_debug_trace_clear()
    if warm:
        for _ in range(3):
            run()
    else:
        flush.zero_()
        flush.sum()
        run()
    torch.cuda.synchronize()
    if workload == "fc512":
        # the short CUDA-core path: per CTA clock64 at its start, loads issued,
        # row-block range arrived, data landed, product done, end
        L_.bp_debug_small_trace_read.restype = ctypes.c_int
        L_.bp_debug_small_trace_read.argtypes = [ctypes.c_void_p, ctypes.c_int]
        sb = (ctypes.c_ulonglong * (256 * 8))()
        assert L_.bp_debug_small_trace_read(sb, 256 * 8) == 256 * 8
        st = np.frombuffer(sb, dtype=np.uint64).reshape(256, 8).astype(np.int64)
        st = st[st[:, 5] > 0]
        d = np.diff(st[:, :6], axis=1)
        print(f"short path, {len(st)} CTAs: median cycles issue {np.median(d[:, 0]):.0f}, "
              f"range {np.median(d[:, 1]):.0f}, data {np.median(d[:, 2]):.0f}, product "
              f"{np.median(d[:, 3]):.0f}, epilogue {np.median(d[:, 4]):.0f}; total "
              f"{np.median(st[:, 5] - st[:, 0]):.0f}")
        g0 = st[:, 6].min()
        print(f"global timer (us after the first CTA start): starts {(st[:, 6] - g0).min() / 1e3:.2f}"
              f"..{(st[:, 6] - g0).max() / 1e3:.2f}, ends {(st[:, 7] - g0).min() / 1e3:.2f}.."
              f"{(st[:, 7] - g0).max() / 1e3:.2f}")
        return
    n = 1024 * 8
    buf = (ctypes.c_ulonglong * n)()
    assert L_.bp_debug_trace_read(buf, n) == n
    t = np.frombuffer(buf, dtype=np.uint64).reshape(1024, 8).astype(np.int64)
    stages = t[:256]
    valid = stages[:, 5] > 0
    # cycles after CTA 0 passed the grid dependency wait
    t0 = t[511, 0]
    rel = np.where(stages > 0, stages - t0, -1)[valid]
    print("stage ctrl_wait ctrl_free ctrl_arr ctrl_w gath_free gath_iss mma_w commit  (clock64 "
          "cycles after CTA 0's start; control: waits for the stage, has it, arrived, weight "
          "tile issued)")
    for i, r in enumerate(rel):
        print(f"{i:5d} {r[4]:9d} {r[0]:9d} {r[6]:8d} {r[7]:6d} {r[1]:9d} {r[2]:8d} {r[3]:6d} {r[5]:6d}")
    c = rel[:, 5]
    if len(c) > 1:
        print(f"median commit interval {np.median(np.diff(c)):.0f} cycles")
    wins = t[256:384]
    wv = wins[:, 2] > 0
    if wv.any():
        print("window ctrl_top ctrl_recs ctrl_next gath_recs  (control: loop top, this window's "
              "records landed, next window requested; gather warp 0: records landed)")
        for i, r in enumerate(wins[wv]):
            print(f"{i:6d} {r[0] - t0:8d} {r[2] - t0:9d} {r[1] - t0:9d} {r[3] - t0:9d}")
    items = t[384:448]
    iv = items[:, 6] > 0
    print("item acc_free epi_saw epi_done")
    for i, r in enumerate(items[iv]):
        print(f"{i:4d} {r[4] - t0:8d} {r[5] - t0:7d} {r[6] - t0:8d}")
    print(f"CTA 0 exit {t[511, 1] - t0} cycles after its start")
    grp = t[512:1024]
    gv = (grp[:, 4] > 0) & (grp[:, 5] > 0) & (grp[:, 3] > 0)
    if gv.any():
        g = grp[gv]
        print(f"epilogue groups of warp 0 (32 columns each): {int(gv.sum())}; median cycles: "
              f"convert {np.median(g[:, 0] - g[:, 4]):.0f}, box free {np.median(g[:, 1] - g[:, 0]):.0f}, "
              f"write+fence {np.median(g[:, 2] - g[:, 1]):.0f}, store issue {np.median(g[:, 3] - g[:, 2]):.0f}, "
              f"next load wait {np.median(g[:, 5] - g[:, 3]):.0f}, group {np.median(g[:, 5] - g[:, 4]):.0f}")
        print("first groups: start, convert, load issue, to store, box free, write, issue, load wait "
              "(cycles after CTA 0's start / durations)")
        for k, r in enumerate(g[:8]):
            print(f"  {k}: {r[4] - t0:7d} {r[6] - r[4]:5d} {r[7] - r[6]:5d} {r[0] - r[7]:5d} "
                  f"{r[1] - r[0]:5d} {r[2] - r[1]:5d} {r[3] - r[2]:5d} {r[5] - r[3]:5d}")
    sp = t[1000:1004]
    if (sp[:, 3] > 0).any():
        print("split epilogue per quadrant, CTA 0 (cycles after its start): reductions start, "
              "issued, fenced, counted; item 0's last arrival (cycles after its sums landed): "
              "output stores start, stored + tile zeroed, each group stored")
        for q, r in enumerate(sp):
            line = f"  q{q}: " + " ".join(f"{v - t0:7d}" if v > 0 else "      -" for v in r[:4])
            if r[4] > 0:
                gs = t[1004 + q]
                line += " | " + " ".join(f"{v - r[4]:7d}" for v in list(r[5:7]) + list(gs) if v > 0)
            print(line)
    g = rel[rel[:, 4] >= 0]
    if len(g):
        print(f"median gather issue -> tensor cores see the rows {np.median(g[:, 4] - g[:, 2]):.0f}")
    ends = t.reshape(-1)[448 * 8: 448 * 8 + 2 * 248].reshape(248, 2)
    ends = ends[ends[:, 1] > 0]
    if len(ends):
        s0 = ends[:, 0].min()
        e = (ends[:, 1] - s0) / 1000.0
        print(f"CTA end (us after the first start): min {e.min():.1f} median "
              f"{np.median(e):.1f} max {e.max():.1f}")


def main(argv):
    if len(argv) >= 1 and argv[0] == "_time":
        _time_in_process(argv[1])
        return
    if len(argv) >= 1 and argv[0] == "_latency":
        _latency_in_process(argv[1])
        return
    if len(argv) >= 1 and argv[0] == "_trace":
        _trace_in_process(argv[1], argv[2])
        return
    if argv and argv[0] == "probe":
        src = os.path.join(B.HERE, "probes", "tc_rates.cu")
        os.makedirs(OUT, exist_ok=True)
        exe = os.path.join(OUT, "tc_rates")
        subprocess.run([B.nvcc(), *B.ARCH, "-O3", "-std=c++17", "-I" + os.path.join(B.ROOT, "include"),
                        src, "-o", exe, "-lcuda"], check=True)
        rc = 0
        for args in (["0", "512", "256"], ["0", "512", "128"], ["0", "512", "64"],
                     ["0", "512", "16"], ["1", "512", "256", "1"], ["1", "512", "256", "2"],
                     ["1", "512", "256", "4"],
                     # stage ring without data: stages, fences
                     ["2", "4096", "256", "4", "0"], ["2", "4096", "256", "4", "1"],
                     ["2", "4096", "256", "4", "3"], ["2", "4096", "256", "6", "1"],
                     ["2", "4096", "256", "2", "1"], ["2", "4096", "256", "4", "5"],
                     ["2", "2048", "256", "4", "2049"],
                     ["2", "2048", "256", "4", "2053"], ["2", "4096", "128", "4", "1"],
                     # what a commit costs: groups of 2 / 4 / 8 MMAs
                     ["4", "2048", "256", "4", "2"], ["4", "2048", "256", "4", "0"],
                     ["4", "2048", "256", "4", "1"], ["4", "4096", "256", "2", "0"],
                     ["4", "1024", "256", "8", "0"], ["4", "1024", "256", "8", "1"],
                     # the row gather alone against its footprint (MB) and row pitch (KB)
                     ["5", "2048", "16", "8", "0"], ["5", "2048", "16", "8", "8"],
                     ["5", "2048", "64", "8", "8"], ["5", "2048", "256", "8", "8"],
                     ["5", "2048", "64", "4", "8"], ["5", "2048", "64", "2", "8"],
                     # gathers beside a bulk-copy stream (the product's mix, no tensor core)
                     ["6", "2048", "64", "6", "0"], ["6", "2048", "64", "6", "1"],
                     ["6", "2048", "64", "6", "2"], ["6", "2048", "64", "4", "0"],
                     ["6", "2048", "64", "4", "2"],
                     # what per-group work between MMA groups costs the issue stream
                     ["8", "2048", "256", "1", "0"], ["8", "2048", "256", "2", "1"],
                     ["8", "2048", "256", "3", "2"], ["8", "2048", "256", "4", "4"],
                     ["8", "2048", "256", "5", "8"], ["8", "2048", "256", "6", "16"],
                     ["8", "2048", "256", "9", "0"], ["8", "2048", "256", "10", "0"],
                     ["8", "2048", "256", "1", "8192"], ["8", "2048", "256", "1", "9216"],
                     ["8", "2048", "256", "1", "10240"], ["8", "2048", "256", "1", "1028"],
                     ["8", "2048", "256", "1", "2052"],
                     # the product's stage ring with its data, no tensor core
                     ["7", "4096", "256", "4", "0"], ["7", "4096", "256", "4", "1"],
                     ["7", "4096", "256", "4", "2"], ["7", "4096", "256", "4", "3"],
                     ["7", "4096", "256", "4", "4"], ["7", "4096", "256", "4", "8"],
                     ["7", "4096", "128", "4", "0"], ["7", "4096", "256", "3", "0"],
                     ["7", "4096", "256", "4", "17"], ["7", "4096", "256", "8", "33"],
                     ["7", "4096", "256", "8", "49"], ["7", "4096", "256", "8", "32"],
                     ["7", "4096", "256", "6", "33"], ["7", "4096", "128", "4", "1"],
                     ["7", "4096", "256", "4", "65"], ["7", "4096", "256", "4", "129"],
                     ["7", "4096", "256", "4", "64"], ["7", "4096", "256", "8", "97"],
                     ["7", "4096", "256", "4", "256"], ["7", "4096", "256", "4", "257"],
                     ["7", "4096", "256", "8", "289"],
                     # MMAs against concurrent copies: bulk, then cp.async rows
                     ["3", "512", "256", "1", "0"], ["3", "512", "256", "2", "0"],
                     ["3", "512", "256", "2", "4"], ["3", "512", "256", "4", "4"],
                     ["3", "512", "256", "6", "4"]):
            rc |= subprocess.run([exe, *args]).returncode
        sys.exit(rc)
    if not argv or argv[0] not in ("time", "latency", "trace"):
        print(__doc__)
        sys.exit(2)
    if argv[0] in ("time", "latency"):
        variants = []
        for a in argv[1:]:
            name, _, fl = a.partition(":")
            variants.append((name, [f for f in fl.split(",") if f]))
        libs = {n: build_variant(n, f) for n, f in variants}
        for n, _ in variants:
            r = subprocess.run([sys.executable, "-m", "paper_2111_11581_gb300.variants",
                                "_" + argv[0], libs[n]], capture_output=True, text=True, cwd=B.ROOT)
            print(f"[{n}] {r.stdout.strip()} {r.stderr.strip()[-400:] if r.returncode else ''}",
                  flush=True)
    else:
        wl = argv[1] if len(argv) > 1 else "gemm"
        extra = [d for d in argv[2:] if d]
        lib = build_variant("trace" + "".join("_" + d.lower() for d in extra), ["BP_TRACE"] + extra)
        r = subprocess.run([sys.executable, "-m", "paper_2111_11581_gb300.variants", "_trace", lib,
                            wl], cwd=B.ROOT)
        sys.exit(r.returncode)


if __name__ == "__main__":
    main(sys.argv[1:])
