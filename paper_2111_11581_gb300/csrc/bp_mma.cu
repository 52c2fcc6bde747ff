// Block-sparse product on the sm_103a tensor cores (bp_gemm, and bp_conv2d:
// the implicit GEMM over an NHWC copy of the input, the NCHW planes in place
// for 1 x 1 layers, or an im2col matrix).
//
// The packed weight is a sequence of 128-row slabs; a slab's column list is
// the union of its rows' kept columns (Sec. 4.3: the rows of a row-block keep
// the same columns, so for bm a multiple of 128 the list is the row-block's
// own).  A work unit is one slab times one tile of 256 activation columns
// (tokens / pixels).  Per k-chunk of 64 listed columns a pipeline stage holds
// the chunk's pre-swizzled weight tile (the MMA's A operand, K-major) and the
// 64 activation rows the chunk names (the B operand, MN-major, 128-byte
// swizzle), so columns no row of the slab keeps never enter the product:
//
//   warps 0-7   gather: for chunks without a load plan, the activation rows,
//               16-byte cp.async straight into the swizzled layout (one
//               512-byte row segment per warp instruction), signalled with
//               cp.async.mbarrier.arrive.noinc so no thread blocks on them;
//   warp 8      control (one thread): per chunk, once its stage is free, sets
//               the stage's flags, copies its weight tile (TMA bulk), and when
//               the chunk's list is made of runs of consecutive columns (its
//               plan, built at pack time) loads the activation rows of each
//               run with TMA tile loads;
//   warp 9      MMA issuer: tcgen05.mma 128 x 256 x 16 into one of two fp32
//               accumulators in tensor memory (the epilogue of a tile
//               overlaps the MMAs of the next), following the stage flags;
//   warps 10-13 epilogue: tcgen05.ld, + bias, ReLU, round to fp16/bf16, then
//               TMA tensor stores of 32 x 32 boxes staged in shared memory
//               (GEMM), or direct stores into the NCHW output (convolution);
//   warp 14     scheduler (one thread): the only role that decodes work
//               units; copies the chunks' records (index list + load plan)
//               into shared memory a window of kWin chunks at a time, with a
//               descriptor the control thread and the gather warps follow,
//               up to two windows ahead (TMA bulk copies).
//
// One mbarrier per stage says that the stage is loaded (the control thread's
// arrival with the TMA byte count, and the gather group's arrivals); the
// tensor-core thread's commit frees it.
//
// Every wait is bounded (see mbar_wait); on expiry the kernel records
// kDevTimeout in the device status word, drains its own copies and tensor
// core work, frees tensor memory and returns.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <cstdint>
#include <mutex>

#include "bp_common.cuh"

// BP_TRACE (off by default; a build for measurement only): CTA 0 records
// clock64() at fixed points of each of its first kTraceChunks pipeline stages,
// read back with bp_debug_trace_read().  Events per stage: 0 control thread
// found the stage free, 1 gather group found it free, 2 gather group issued
// its copies, 3 MMA thread saw the stage loaded, 4 control thread started
// waiting for the stage, 5 MMA thread committed the stage, 6 and 7 control
// thread before / after issuing the weight copy.  Per window w (entries 256 +
// w): 0 control thread at the window, 2 it saw the window's records, 3 gather
// warp 0 saw them; per item i (entries 384 + i): 4 MMA thread holds a
// free accumulator, 5 the first epilogue warp saw the finished accumulator, 6
// it issued the item's last store.  Entries 448 .. hold the global-timer start
// and end of each of the first 248 CTAs; entry 511: CTA 0's clock64() after
// the grid dependency wait (0) and at exit (1).  Per 32-column output group g
// of the first epilogue warp (entries 512 + g): 4 group start, 6 converted, 7
// next group's tensor-memory load issued, 0 store entered, 1 its staging box
// free, 2 box written and fenced, 3 store issued, 5 the next load landed.
// Split launches, per epilogue warp of quadrant q (entries 1000 + q): 0 its
// reductions start, 1 issued, 2 fenced, 3 arrival counted (CTA 0), and for
// the last arrival of split item 0 (any CTA, its own clock): 4 the sums
// landed in shared memory, 5 the output stores start, 6 the output stored and
// the tile zeroed; entries 1004 + q: each column group stored.
#ifdef BP_TRACE
namespace bp {
constexpr int kTraceChunks = 1024;
constexpr int kTraceEvents = 8;
__device__ unsigned long long g_trace[kTraceChunks * kTraceEvents];
}  // namespace bp
#define BP_TR(seq, ev)                                                                   \
    do {                                                                                 \
        if (blockIdx.x == 0 && (seq) < bp::kTraceChunks)                                 \
            bp::g_trace[(seq) * bp::kTraceEvents + (ev)] = clock64();                    \
    } while (0)
#else
#define BP_TR(seq, ev) \
    do {               \
    } while (0)
#endif

namespace bp {
namespace {

constexpr uint64_t kDrainNs = 1000000000ull;
constexpr int kMaxStages = 8;
constexpr int kWin = 16;               // chunk records per shared-memory window
constexpr int kWinBufs = 3;            // windows in shared memory (one being filled ahead)
constexpr uint32_t kWinBytes = kWin * kMetaBytes;
constexpr uint32_t kCwinBytes = 256;        // one Window record (size checked below)
constexpr int kWmeta = 6;                   // int64 words of a window descriptor
// Window descriptor flags (Smem::wmeta word 3).
constexpr uint32_t kWinFirst = 1;       // the window starts its unit
constexpr uint32_t kWinLast = 2;        // the window ends its unit
constexpr uint32_t kWinFinal = 4;       // the unit is the CTA's final one
// Stage flags (Smem::sflag): how the stage's activations were loaded and where
// its chunk sits in its work unit.  Only the scheduler warp decodes work units
// (into window descriptors, Smem::wmeta, which the control thread and the
// gather warps follow); the tensor-core thread follows the stage flags the
// control thread sets.
constexpr uint32_t kStageTma = 1;       // activations loaded by TMA (no proxy fence needed)
constexpr uint32_t kStageFirst = 2;     // first chunk of its unit: a fresh accumulator
constexpr uint32_t kStageLast = 4;      // last chunk of its unit: the accumulator is complete
constexpr uint32_t kStageFinal = 8;     // last chunk of the CTA's final unit
constexpr uint32_t kStageEnd = 16;      // no more chunks: the stage holds nothing
constexpr int64_t kMaxCachedKc = 2048; // kc_ptr entries kept in shared memory at most
constexpr int64_t kMaxSmem = 232448;   // dynamic shared memory per CTA (227 KB)
constexpr int kNT = 256;               // activation columns per tile at most (the MMA's N)
constexpr uint32_t kWTileBytes = kSlab * kBK * 2;   // 16 KB
constexpr uint32_t kXTileBytes = kNT * kBK * 2;     // 32 KB

// Warp roles.
constexpr int kGatherWarps = 8;
constexpr int kCtrlWarp = 8;
constexpr int kMmaWarp = 9;
constexpr int kEpiWarp0 = 10;
constexpr int kSchedWarp = kEpiWarp0 + 4;   // decodes the windows ahead (lane 0)
constexpr int kThreads = (kSchedWarp + 1) * 32;
// The gather warps form kGatherGroups groups that take turns: group g
// gathers the chunks whose sequence number is g modulo kGatherGroups, so one
// group issues copies while another waits for its next stage.
constexpr int kGatherGroups = 2;
constexpr int kGroupWarps = kGatherWarps / kGatherGroups;
constexpr int kRowsPerWarp = 64 / kGroupWarps;      // list positions per warp and chunk
constexpr uint32_t kGroupThreads = kGroupWarps * 32;
// One barrier per stage tells the tensor-core thread that the stage is
// loaded: the control thread arrives once (with the stage's TMA byte count)
// and the chunk's gather group kGroupThreads times, each thread when its
// copies have landed, or lane 0 of each warp for its warp when the chunk has
// a load plan (TMA brings its rows).  A second barrier for the gathered rows
// costs the tensor-core thread another wait per chunk, 100-150 cycles even
// when its phase has already completed.
constexpr uint32_t kStageArrivals = kGroupThreads + 1;

struct Params {
    CUtensorMap ymap;       // output, box 32 x 32 (x 1), 64-byte swizzle: GEMM Y as a 2-D
                            // tensor (N, M); NCHW output as a 3-D tensor (Ho*Wo, M, Nb)
    CUtensorMap ymap64;     // the same tensor, box 64 x 32 (x 1), 128-byte swizzle
    CUtensorMap xmap[4];    // activations X (N inner, K rows), boxes 64 x (8 << i), 128-byte swizzle
    int dtype;
    int relu;
    int conv;               // 1: Y is the NCHW output of a convolution
    int ytma;               // 1: output boxes are written with TMA stores through ymap
    int yvec;               // convolution: Ho*Wo % 8 == 0 (BP_EPI_DIRECT: 8 pixels per 16-byte store)
    int64_t M, num_slabs;
    int64_t N;              // tokens (GEMM) or Nb*Ho*Wo pixels (conv)
    int nt;                 // activation columns per tile: a multiple of 32, 64 .. 256
    int xboxes;             // 64-column TMA boxes per activation row: ceil(nt / 64)
    int64_t num_items;      // (slab, column tile) items
    int64_t full_items;     // the first full_items items are single work units
    int split;              // units per later item (k-chunk ranges)
    int64_t num_units;      // full_items + (num_items - full_items) * split
    float *part;            // split items: one fp32 accumulator tile per item, [item][128][256];
                            // balanced launches: one partial tile per CTA
    int32_t *cnt;           // split items: arrivals per (item, row quadrant); balanced
                            // launches: per (CTA, row quadrant) "partial written" flags
    // implicit convolution (stride 1): X is the NHWC input with channels padded
    // to 8 (imap: 4-D (C8, W, H, Nb), boxes of 64 channels x Wo x hbox x nbox);
    // a chunk's B operand is one box: per output pixel a K-major row of 64
    // channels at one kernel position (128-byte swizzle)
    int impl;
    CUtensorMap imap;
    int64_t i_ipt, i_rpt, i_tpi, i_HoWo, i_Wo, i_Ho, i_Nb;
    int i_ph, i_pw;
    int i_s;                // stride 1, or 2: imap holds the input's four phases
    // 1 x 1 stride-1 convolution read in place: the activation row of channel c
    // for pixel n = b*HW + hw is X + b*d_CHW + c*ldx + hw (ldx = HW), no load plans
    int direct;
    int64_t d_CHW;
    uint32_t i_box_bytes;
    int sk;                 // 1: balanced launch (whole items in full waves, then each CTA
                            // one equal range of the remaining items' chunks)
    int64_t sk_i0;          // balanced launch: first item of the ranges
    int64_t sk_total;       // balanced launch: chunks of all items (tiles x kc_total)
    int64_t kc_total;       // chunks of one column tile (all slabs)
    int64_t stages;
    uint32_t tmem_cols, acc_cols, ystage_bytes;
    const int64_t *kc_ptr;
    int64_t kc_cached;      // entries of kc_ptr copied to shared memory (0 = none)
    const uint8_t *tiles;   // k-chunk weight tiles (16 KB each)
    const uint8_t *meta;    // k-chunk records: index list + load plan (kMetaBytes each)
    const uint16_t *X;
    int64_t ldx;
    uint16_t *Y;
    int64_t ldy;
    int64_t HoWo;           // conv: output pixels per image
    const float *bias;
    uint64_t watchdog_ns;
    int64_t drop_stage;     // fault injection: CTA 0 never fills this stage (-1 = off)
    unsigned *status;
};

// Two fp32 values to one 16-bit pair (a low, b high), round to nearest even,
// negative values to zero when kRelu (one cvt instruction).
template <bool kBf16, bool kRelu>
__device__ __forceinline__ uint32_t cvt_pair(float a, float b) {
    uint32_t d;
    if (kBf16) {
        if (kRelu) asm("cvt.rn.relu.bf16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(b), "f"(a));
        else asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(b), "f"(a));
    } else {
        if (kRelu) asm("cvt.rn.relu.f16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(b), "f"(a));
        else asm("cvt.rn.f16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(b), "f"(a));
    }
    return d;
}

template <bool kBf16, bool kRelu>
__device__ __forceinline__ void cvt_group(const uint32_t (&r)[32], float bv, uint32_t (&pk)[16]) {
#pragma unroll
    for (int e = 0; e < 16; ++e)
        pk[e] = cvt_pair<kBf16, kRelu>(__uint_as_float(r[2 * e]) + bv, __uint_as_float(r[2 * e + 1]) + bv);
}

// bias + ReLU + cast of a 32-column group, one branch per group
__device__ __forceinline__ void cvt_any(const Params &p, const uint32_t (&r)[32], float bv,
                                        uint32_t (&pk)[16]) {
    if (p.dtype == BP_BF16) {
        if (p.relu) cvt_group<true, true>(r, bv, pk);
        else cvt_group<true, false>(r, bv, pk);
    } else {
        if (p.relu) cvt_group<false, true>(r, bv, pk);
        else cvt_group<false, false>(r, bv, pk);
    }
}

// Whole images of an NCHW output: lane r (channel row) of a 32-column group
// holds Ho*Wo consecutive values of each of `imgs` images (packed pairs in pk,
// Ho*Wo a power of two below 32) and writes them at yl + i * istride (its
// channel's place in image i's run of 32 channels x Ho*Wo pixels), so that
// every warp store is one contiguous piece of 64 Ho*Wo bytes.  Loops are
// unrolled to their bound so that pk stays in registers.
__device__ __forceinline__ void store_images(uint16_t *yl, int64_t istride, uint32_t HW, int imgs,
                                             const uint32_t (&pk)[16]) {
    if (HW == 1u) {
#pragma unroll
        for (int i = 0; i < 32; ++i)
            if (i < imgs) yl[i * istride] = (uint16_t)(pk[i >> 1] >> (16 * (i & 1)));
    } else if (HW == 2u) {
#pragma unroll
        for (int i = 0; i < 16; ++i)
            if (i < imgs) *reinterpret_cast<uint32_t *>(yl + i * istride) = pk[i];
    } else if (HW == 4u) {
#pragma unroll
        for (int i = 0; i < 8; ++i)
            if (i < imgs) *reinterpret_cast<uint2 *>(yl + i * istride) = make_uint2(pk[2 * i], pk[2 * i + 1]);
    } else if (HW == 8u) {
#pragma unroll
        for (int i = 0; i < 4; ++i)
            if (i < imgs)
                *reinterpret_cast<uint4 *>(yl + i * istride) =
                    make_uint4(pk[4 * i], pk[4 * i + 1], pk[4 * i + 2], pk[4 * i + 3]);
    } else {
#pragma unroll
        for (int i = 0; i < 2; ++i)
            if (i < imgs) {
                uint4 *d = reinterpret_cast<uint4 *>(yl + i * istride);
                d[0] = make_uint4(pk[8 * i], pk[8 * i + 1], pk[8 * i + 2], pk[8 * i + 3]);
                d[1] = make_uint4(pk[8 * i + 4], pk[8 * i + 5], pk[8 * i + 6], pk[8 * i + 7]);
            }
    }
}

struct Smem {
    uint8_t *w;          // stages x kWTileBytes
    uint8_t *x;          // stages x kXTileBytes
    uint8_t *ystage;     // GEMM: 4 epilogue warps x 2 buffers x 2 KB
    uint64_t *wfull;     // [stages] the stage is loaded: weight tile, TMA-loaded activations
                         // and gathered rows (kStageArrivals arrivals + the TMA bytes)
    uint64_t *empty;     // [stages] tensor cores done with the stage
    uint64_t *tfull;     // [2] accumulator ready for the epilogue
    uint64_t *tempty;    // [2] accumulator drained
    uint64_t *drain;     // [1]
    uint64_t *fixbar;    // [4] balanced launch: a partial tile's quadrant landed (per epilogue warp)
    uint64_t *ffull;     // the CTA's final item's accumulator is complete (single use)
    uint64_t *pfull;     // [kWinBufs] a window of chunk records landed (TMA byte count)
    uint64_t *pempty;    // [kWinBufs] the gather warps and the control thread are done with it
    uint32_t *sflag;     // [stages] what the stage holds (kStage* bits), set by the control
                         // thread before its arrival on wfull
    uint32_t *tmem_base;
    int *abort_flag;
    int64_t *gprog;      // [kGatherWarps + 1] per gather warp: 1 + the sequence number of the
                         // last chunk it arrived for; [kGatherWarps]: warps out of their loop
    int64_t *skv;        // [4] balanced launch: chunk position of item sk_i0, chunks from
                         // there on, this CTA's range [lo, hi) (set in the prologue)
    int64_t *wmeta;      // [kWinBufs][kWmeta] per window buffer, written before the
                         // arrival on pfull: chunks in the window (0: no more windows),
                         // the tile's first token column, the window's first chunk
                         // position, kWin* flags, and the implicit convolution's first
                         // output row and image
    uint8_t *cwin;       // [sizeof(Window)] window 1, decoded before the dependency wait
    int *pre;            // weight tiles requested before the dependency wait (-1: the
                         // first window was not requested then)
    uint8_t *win;        // [kWinBufs][kWinBytes] chunk records of the current windows
    int64_t *kc;         // [kc_cached] copy of kc_ptr, or nullptr
};

__device__ __forceinline__ Smem carve(uint8_t *raw, const Params &p) {
    Smem s;
    uint8_t *base = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(raw) + 1023) & ~static_cast<uintptr_t>(1023));
    s.w = base;
    s.x = base + p.stages * kWTileBytes;
    s.ystage = s.x + p.stages * kXTileBytes;
    uint8_t *b = s.ystage + p.ystage_bytes;
    s.wfull = reinterpret_cast<uint64_t *>(b);
    s.empty = s.wfull + p.stages;
    s.tfull = s.empty + p.stages;
    s.tempty = s.tfull + 2;
    s.drain = s.tempty + 2;
    s.fixbar = s.drain + 1;
    s.ffull = s.fixbar + 4;
    s.pfull = s.ffull + 1;
    s.pempty = s.pfull + kWinBufs;
    s.sflag = reinterpret_cast<uint32_t *>(s.pempty + kWinBufs);
    s.tmem_base = s.sflag + p.stages;
    s.abort_flag = reinterpret_cast<int *>(s.tmem_base + 1);
    s.gprog = reinterpret_cast<int64_t *>(
        (reinterpret_cast<uintptr_t>(s.abort_flag + 1) + 7) & ~static_cast<uintptr_t>(7));
    s.skv = s.gprog + kGatherWarps + 1;
    s.wmeta = s.skv + 4;
    s.cwin = reinterpret_cast<uint8_t *>(s.wmeta + kWmeta * kWinBufs);
    s.pre = reinterpret_cast<int *>(s.cwin + kCwinBytes);
    // TMA bulk copies need a 16-byte-aligned destination: round up to 128 bytes
    const uintptr_t after = reinterpret_cast<uintptr_t>(s.pre + 2);
    s.win = reinterpret_cast<uint8_t *>((after + 127) & ~static_cast<uintptr_t>(127));
    s.kc = p.kc_cached ? reinterpret_cast<int64_t *>(s.win + kWinBufs * kWinBytes) : nullptr;
    return s;
}

size_t smem_bytes(int64_t stages, uint32_t ystage_bytes, int64_t kc_cached) {
    return 1024 + (size_t)stages * (kWTileBytes + kXTileBytes) + ystage_bytes +
           (2 * (size_t)stages + 10 + 2 * kWinBufs) * 8 + 4 * (size_t)stages + 8 + 8 +
           8 * (kGatherWarps + 1) + 32 + 8 * kWmeta * kWinBufs + kCwinBytes + 8 + 128 +
           (size_t)kWinBufs * kWinBytes + 8 * (size_t)kc_cached;
}

__device__ __forceinline__ void raise_timeout(const Params &p, const Smem &s) {
    *reinterpret_cast<volatile int *>(s.abort_flag) = 1;
    atomicOr(p.status, kDevTimeout);
}

struct Item {
    int64_t slab, n0, kc0, nkc, rows;   // rows = real rows of the slab
    int64_t j;                          // split item index (-1: whole item)
    int s, S;                           // unit s of S of the item
    // balanced launches: 0 the whole item, 1 its first chunks (this CTA adds
    // the partial tiles of the CTAs that own the rest and writes the output),
    // 2 a later range of its chunks (this CTA writes a partial tile)
    int role;
    int64_t gpos, nitem;                // first chunk of the item (global position), its chunks
    int64_t ncols;                      // output columns (pixels) of the tile
    int64_t img0, h0;                   // implicit convolution: first image and row of the tile
};

// Work unit u -> (slab, column tile) item, slab fastest, and its k-chunk
// range: the whole item for u < full_items, else unit s of `split` equal
// shares of the item's chunks.  Unit, item and slab counts are below 2^31
// (checked at launch), so the divisions are 32-bit: 64-bit divisions by a
// runtime value cost hundreds of cycles, and the control thread decodes units
// on its issue path.
__device__ __forceinline__ Item decode(const Params &p, const int64_t *kc, int64_t u) {
    Item t;
    uint32_t it = (uint32_t)u;
    t.role = 0;
    t.gpos = 0;
    t.j = -1;
    t.s = 0;
    t.S = 1;
    if (u >= p.full_items) {
        const uint32_t v = (uint32_t)(u - p.full_items), sp = (uint32_t)p.split;
        const uint32_t jj = v / sp;
        t.j = jj;
        t.s = (int)(v - jj * sp);
        t.S = p.split;
        it = (uint32_t)p.full_items + jj;
    }
    const uint32_t ns = (uint32_t)p.num_slabs;
    const uint32_t tile = it / ns;
    t.slab = it - tile * ns;
    t.n0 = (int64_t)tile * p.nt;
    t.ncols = min((int64_t)p.nt, p.N - t.n0);
    t.img0 = t.h0 = 0;
    if (p.impl) {
        // tiles of whole output rows: ipt images, or rpt rows of one image
        if (p.i_ipt > 0) {
            t.img0 = (int64_t)tile * p.i_ipt;
            t.n0 = t.img0 * p.i_HoWo;
            t.ncols = min(p.i_ipt, p.i_Nb - t.img0) * p.i_HoWo;
        } else {
            const uint32_t tpi = (uint32_t)p.i_tpi;
            const uint32_t img = tile / tpi;
            t.img0 = img;
            t.h0 = (int64_t)(tile - img * tpi) * p.i_rpt;
            t.n0 = t.img0 * p.i_HoWo + t.h0 * p.i_Wo;
            t.ncols = min(p.i_rpt, p.i_Ho - t.h0) * p.i_Wo;
        }
    }
    const int64_t c0 = kc[t.slab], nc = kc[t.slab + 1] - c0;
    if (t.S == 1) {
        t.kc0 = c0;
        t.nkc = nc;
    } else {
        const int64_t kb = nc * t.s / t.S, ke = nc * (t.s + 1) / t.S;
        t.kc0 = c0 + kb;
        t.nkc = ke - kb;
    }
    t.rows = min((int64_t)kSlab, p.M - t.slab * kSlab);
    t.nitem = t.nkc;
    return t;
}

// Balanced launches: CTA c first runs whole items c, c + gridDim.x, ... below
// item sk_i0 (full waves: the same count for every CTA), then the chunks of
// items sk_i0 .. in item order (column tile, then slab) are cut into
// gridDim.x equal ranges, CTA c taking the c-th.  An item cut by a range
// boundary is finished by the CTA that computes its first chunks (the last
// thing that CTA does); the CTAs that compute its later chunks do so first
// thing in their range and leave fp32 partial tiles.  Every CTA thus runs the
// same number of chunks, instead of a last wave that leaves most SMs idle, and
// the whole-item waves keep the working set of the first waves as small as a
// plain launch's (a few column tiles at a time).
// first chunk position (relative to the ranges' start) of CTA c's range; T =
// chunks of the ranges
__device__ __forceinline__ int64_t sk_lo(int64_t T, int64_t c) { return c * T / gridDim.x; }
// the CTA whose range holds chunk position g (absolute); skv as in Smem
__device__ __forceinline__ int64_t sk_owner(const int64_t *skv, int64_t g) {
    const int64_t T = skv[1], r = g - skv[0];
    const int64_t G = gridDim.x;
    int64_t c = r * G / T;
    while (c + 1 < G && sk_lo(T, c + 1) <= r) ++c;
    while (c > 0 && sk_lo(T, c) > r) --c;
    return c;
}
// The part of the item holding chunk position u that lies in [u, end).
__device__ __forceinline__ Item sk_decode(const Params &p, const int64_t *kc, int64_t u,
                                          int64_t end) {
    Item t;
    t.j = -1;
    t.s = 0;
    t.S = 1;
    const uint32_t kct = (uint32_t)p.kc_total;
    const uint32_t tile = (uint32_t)u / kct;      // positions are below 2^31 (checked at launch)
    const int64_t o = u - (int64_t)tile * kct;
    // the slab whose chunks hold o: the last s with kc[s] <= o (o < kc[num_slabs])
    int64_t lo = 0, hi = p.num_slabs;
    while (hi - lo > 1) {
        const int64_t mid = (lo + hi) >> 1;
        if (kc[mid] <= o) lo = mid;
        else hi = mid;
    }
    t.slab = lo;
    t.n0 = (int64_t)tile * p.nt;
    const int64_t klo = o - kc[lo];
    t.nitem = kc[lo + 1] - kc[lo];
    const int64_t khi = min(t.nitem, klo + (end - u));
    t.kc0 = kc[lo] + klo;
    t.nkc = khi - klo;
    t.gpos = u - klo;
    t.role = klo > 0 ? 2 : (khi < t.nitem ? 1 : 0);
    t.rows = min((int64_t)kSlab, p.M - t.slab * kSlab);
    t.ncols = min((int64_t)p.nt, p.N - t.n0);
    t.img0 = t.h0 = 0;
    return t;
}

// This CTA's work units in order: items (or split units) blockIdx.x, + gridDim.x,
// ...; in balanced launches those below sk_i0, then the item parts of its
// chunk range.
struct UnitIter {
    int64_t u, end;
    bool ranged;         // in the chunk range of a balanced launch
    const int64_t *skv;
    __device__ __forceinline__ void enter_range() {
        ranged = true;
        u = skv[2];
        end = skv[3];
    }
    __device__ __forceinline__ void init(const Params &p, const int64_t *skv_) {
        skv = skv_;
        ranged = false;
        u = blockIdx.x;
        end = p.sk ? p.sk_i0 : p.num_units;
        if (p.sk && u >= end) enter_range();
    }
    __device__ __forceinline__ bool valid() const { return u < end; }
    __device__ __forceinline__ Item get(const Params &p, const int64_t *kc) const {
        return ranged ? sk_decode(p, kc, u, end) : decode(p, kc, u);
    }
    __device__ __forceinline__ void step(const Params &p, const Item &t) {
        if (ranged) {
            u += t.nkc;
        } else {
            u += gridDim.x;
            if (p.sk && u >= end) enter_range();
        }
    }
};

// Walks this CTA's windows: runs of up to kWin consecutive k-chunks of one
// work unit, in the order the CTA processes them (units with no chunk skipped).
struct Window {
    UnitIter ui;         // work unit
    int64_t k0, cnt;     // first chunk of the window within the unit, chunks in it
    Item t;
    __device__ __forceinline__ void first(const Params &p, const int64_t *kcp, const int64_t *skv) {
        k0 = 0;
        for (ui.init(p, skv); ui.valid(); ui.step(p, t)) {
            t = ui.get(p, kcp);
            if (t.nkc > 0) break;
        }
        cnt = valid(p) ? min((int64_t)kWin, t.nkc) : 0;
    }
    __device__ __forceinline__ void next(const Params &p, const int64_t *kcp) {
        k0 += kWin;
        if (k0 >= t.nkc) {
            k0 = 0;
            for (ui.step(p, t); ui.valid(); ui.step(p, t)) {
                t = ui.get(p, kcp);
                if (t.nkc > 0) break;
            }
        }
        cnt = valid(p) ? min((int64_t)kWin, t.nkc - k0) : 0;
    }
    __device__ __forceinline__ bool valid(const Params &) const { return ui.valid(); }
};
static_assert(sizeof(Window) <= kCwinBytes, "window record");

// The CTA's final item: its last work unit, when it has chunks and the launch
// splits nothing.  By the time its accumulator is complete every pipeline
// stage is idle, and the gather warps share its epilogue with the epilogue
// warps (each warp can read the tensor-memory lanes of quadrant warp % 4).
__device__ __forceinline__ bool final_unit(const Params &p, const UnitIter &ui, const Item &t) {
    if (p.split > 1 || p.sk || t.nkc == 0) return false;
    UnitIter nx = ui;
    nx.step(p, t);
    return !nx.valid();
}

// Load plan of a chunk record (see DevLayout): number of tile loads.
__device__ __forceinline__ int plan_loads(const uint8_t *rec) {
    return *reinterpret_cast<const volatile int32_t *>(rec + kListBytes);
}

// ------------------------------------------------------------------ gather warps
__device__ void gather_warps(const Params &p, const Smem &s) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    volatile int *abort_flag = s.abort_flag;
    const int group = warp / kGroupWarps, gw = warp % kGroupWarps;
    const int nst = (int)p.stages;
    constexpr int kStep = kGatherGroups;
    constexpr int rbase = 0;
    int gst = group;            // stage of this group's next chunk (sequence number group + 2i)
    uint32_t gph = 0;
    int64_t count = 0, wseq = 0;
    bool ok = true;
    for (;; ++wseq) {
        const int buf = (int)(wseq % kWinBufs);
        // outcomes of waits are made warp-uniform, so the warp leaves the loop as one
        ok = __all_sync(0xffffffffu, mbar_wait(&s.pfull[buf], (uint32_t)((wseq / kWinBufs) & 1),
                                              p.watchdog_ns, abort_flag));
        if (!ok) break;
        if (warp == 0 && lane == 0) BP_TR(256 + wseq, 3);
        // the window's descriptor, written by the control thread before its
        // arrival on pfull
        const int64_t wcnt = s.wmeta[kWmeta * buf], wn0 = s.wmeta[kWmeta * buf + 1];
        if (wcnt == 0) break;       // no more windows
        const uint8_t *recs = s.win + buf * kWinBytes;
        // the tile's token columns: 16 bytes (8 columns) per lane, lanes past
        // the tile's width idle
        const int64_t n = wn0 + lane * 8;
        const uint32_t nb =
            (lane * 8 < p.nt && n < p.N) ? (uint32_t)min((int64_t)16, (p.N - n) * 2) : 0u;
        const uint16_t *xcol = p.X;
        if (nb && p.direct) {
            const int64_t b = n / p.ldx;
            xcol = p.X + b * p.d_CHW + (n - b * p.ldx);
        } else if (nb) {
            xcol = p.X + n;
        }
        // This warp's list positions of its next chunk are read from shared
        // memory before the current chunk's copies are issued: the copies fill
        // the load/store queue, and reads issued behind them would wait for it.
        int32_t idx[kRowsPerWarp];
        bool tma = false;
        auto fetch = [&](int64_t j, int32_t (&ix)[kRowsPerWarp], bool &planned) {
            const uint8_t *rec = recs + j * kMetaBytes;
            planned = plan_loads(rec) > 0 && !p.direct;
            const int32_t *l = reinterpret_cast<const int32_t *>(rec);
#pragma unroll
            for (int i = 0; i < kRowsPerWarp; ++i) ix[i] = l[rbase + gw + kGroupWarps * i];
        };
        const int64_t base = count;         // sequence number of the window's first chunk
        int64_t j = (group - base % kGatherGroups + kGatherGroups) % kGatherGroups;
        if (j < wcnt) fetch(j, idx, tma);
        for (; j < wcnt; j += kStep) {
            int32_t nidx[kRowsPerWarp];
            bool ntma = false;
            if (j + kStep < wcnt) fetch(j + kStep, nidx, ntma);
            const int64_t seq = base + j;
            // stage = seq mod stages, phase = its ring pass parity (kept
            // incrementally: a 64-bit division per chunk sits on the issue path)
            const int stage = gst;
            const uint32_t phase = gph;
            gst += kStep;
            if (gst >= nst) {
                gst -= nst;
                gph ^= 1u;
            }
            const bool drop = blockIdx.x == 0 && seq == p.drop_stage;
            // A planned chunk is loaded by the control thread; the group still
            // waits for its stage (lane 0 alone) and arrives on it, lane 0 for
            // the warp, which keeps it at most one phase of the stage barriers
            // ahead of the tensor cores.
            ok = __all_sync(0xffffffffu,
                            (!tma || lane == 0)
                                ? mbar_wait(&s.empty[stage], phase ^ 1u, p.watchdog_ns, abort_flag)
                                : true);
            if (!ok) break;
            if (gw == 0 && lane == 0) BP_TR(seq, 1);
            if (tma && !drop && lane == 0) mbar_arrive_cnt(&s.wfull[stage], 32);
            if (!tma && !drop) {
                // 64 rows x nt columns: one warp instruction per row segment
                const uint32_t xs = smem_u32(s.x + stage * kXTileBytes);
                const int cn = lane >> 3, jj = lane & 7;
                if (lane * 8 < p.nt) {
                    // lanes whose 8 columns are all inside N copy without the
                    // zero-fill operand
                    if (nb == 16u) {
#pragma unroll
                        for (int i = 0; i < kRowsPerWarp; ++i) {
                            const int r = rbase + gw + kGroupWarps * i;
                            cp_async_16_full(xs + cn * 8192 + r * 128 + ((jj ^ (r & 7)) << 4),
                                             xcol + (int64_t)idx[i] * p.ldx);
                        }
                    } else {
#pragma unroll
                        for (int i = 0; i < kRowsPerWarp; ++i) {
                            const int r = rbase + gw + kGroupWarps * i;
                            cp_async_16(xs + cn * 8192 + r * 128 + ((jj ^ (r & 7)) << 4),
                                        xcol + (int64_t)idx[i] * p.ldx, nb);
                        }
                    }
                }
                // Arrive on the stage once this thread's copies have landed, without
                // blocking.  The tile was written through the generic proxy; the
                // tensor-core thread orders it before its async-proxy reads with a
                // proxy fence after acquiring the barrier.
                cp_async_arrive_noinc(&s.wfull[stage]);
                if (gw == 0 && lane == 0) BP_TR(seq, 2);
            }
            // progress for the control thread's unwinding (after the arrivals)
            if (lane == 0) *reinterpret_cast<volatile int64_t *>(&s.gprog[warp]) = seq + 1;
#pragma unroll
            for (int i = 0; i < kRowsPerWarp; ++i) idx[i] = nidx[i];
            tma = ntma;
        }
        count = base + wcnt;
        if (!ok) break;
        __syncwarp();        // the lanes' reads of the window precede lane 0's release
        if (lane == 0) mbar_arrive(&s.pempty[buf]);
    }
    if (!ok) raise_timeout(p, s);
    cp_async_wait_all();
    __syncwarp();
    if (lane == 0) {
        __threadfence_block();
        atomicAdd(reinterpret_cast<unsigned long long *>(&s.gprog[kGatherWarps]), 1ull);
    }
}

// ------------------------------------------------------------------ control thread
struct WindowFiller {
    Window ahead;        // next window to copy into shared memory (decoded)
    int64_t filled;      // windows copied so far
    // Requests window `filled` (= ahead) into its buffer with its descriptor;
    // past the last window, the end marker (a descriptor of 0 chunks).  Then
    // decodes the window after it.
    __device__ __forceinline__ void fill(const Params &p, const Smem &s, const int64_t *kcp) {
        const int buf = (int)(filled % kWinBufs);
        int64_t *wm = s.wmeta + kWmeta * buf;
        ++filled;
        if (!ahead.valid(p)) {
            wm[0] = 0;
            mbar_arrive(&s.pfull[buf]);
            return;
        }
        wm[0] = ahead.cnt;
        wm[1] = ahead.t.n0;
        wm[2] = ahead.t.kc0 + ahead.k0;
        wm[3] = (ahead.k0 == 0 ? kWinFirst : 0u) | (ahead.k0 + ahead.cnt == ahead.t.nkc ? kWinLast : 0u) |
                (final_unit(p, ahead.ui, ahead.t) ? kWinFinal : 0u);
        wm[4] = ahead.t.h0;
        wm[5] = ahead.t.img0;
        const uint32_t bytes = (uint32_t)ahead.cnt * kMetaBytes;
        mbar_arrive_expect_tx(&s.pfull[buf], bytes);
        bulk_g2s(smem_u32(s.win + buf * kWinBytes),
                 p.meta + (ahead.t.kc0 + ahead.k0) * kMetaBytes, bytes, &s.pfull[buf]);
        ahead.next(p, kcp);
    }
    // the CTA is unwinding: let the window copies that may be in flight land first
    __device__ __forceinline__ void drain(const Params &p, const Smem &s) {
        for (int64_t q = filled > kWinBufs ? filled - kWinBufs : 0; q < filled; ++q)
            if (!mbar_wait(&s.pfull[q % kWinBufs], (uint32_t)((q / kWinBufs) & 1), kDrainNs,
                           nullptr))
                atomicOr(p.status, kDevTimeout);
    }
};

// Before the grid dependency wait, while the previous kernel in the stream may
// still run: the chunk records of the first window and the weight tiles of the
// first chunks come from the packed image (written by bp_pack, which
// synchronises), not from anything a kernel in flight writes, so they are
// requested now, and window 1 is decoded (kept in cwin for the scheduler
// warp).  A weight tile only adds its bytes to its stage barrier; the control
// thread arrives once the stage's activation loads are issued.
// Returns the number of weight tiles requested, or -1 when the window was not
// copied (balanced launches, whose ranges are set after the wait).
__device__ int control_prefetch(const Params &p, const Smem &s) {
    if (p.sk) return -1;
    const int64_t *kcp = s.kc ? s.kc : p.kc_ptr;
    WindowFiller wf;
    wf.ahead.first(p, kcp, s.skv);
    wf.filled = 0;
    if (!wf.ahead.valid(p)) return -1;
    const Window win = wf.ahead;
    wf.fill(p, s, kcp);
    *reinterpret_cast<Window *>(s.cwin) = wf.ahead;
    const int n = (int)min((int64_t)p.stages, win.cnt);
    for (int j = 0; j < n; ++j) {
        if (blockIdx.x == 0 && j == p.drop_stage) return j;
        mbar_expect_tx(&s.wfull[j], kWTileBytes);
        bulk_g2s(smem_u32(s.w + j * kWTileBytes), p.tiles + (win.t.kc0 + win.k0 + j) * (int64_t)kWTileBytes,
                 kWTileBytes, &s.wfull[j]);
    }
    return n;
}

// The scheduler warp's lane 0: requests the CTA's windows of chunk records in
// order, each with its descriptor, as the buffers come free (the window after
// the last one is the end marker).  It is the only role that decodes work
// units, and it runs up to kWinBufs - 1 windows ahead of the others, so the
// decoding (cold code, run once per window) stays off their paths.
__device__ void scheduler_thread(const Params &p, const Smem &s) {
    const int64_t *kcp = s.kc ? s.kc : p.kc_ptr;
    volatile int *abort_flag = s.abort_flag;
    WindowFiller wf;
    if (*s.pre >= 0) {          // window 0 was requested before the dependency wait
        wf.ahead = *reinterpret_cast<const Window *>(s.cwin);
        wf.filled = 1;
    } else {
        wf.ahead.first(p, kcp, s.skv);
        wf.filled = 0;
    }
    bool ok = true;
    for (;;) {
        // window `filled` goes to the buffer released by window filled - kWinBufs
        const int64_t prev = wf.filled - kWinBufs;
        if (prev >= 0 && !mbar_wait(&s.pempty[prev % kWinBufs], (uint32_t)((prev / kWinBufs) & 1),
                                    p.watchdog_ns, abort_flag)) {
            ok = false;
            break;
        }
        const bool end = !wf.ahead.valid(p);
        wf.fill(p, s, kcp);
        if (end) break;
    }
    if (!ok) raise_timeout(p, s);
    // the last window copies land before the CTA can exit, whether or not a
    // consumer reached them
    wf.drain(p, s);
}

// The control thread follows the window descriptors: per chunk it waits for
// the stage, sets the stage's flags and issues its TMA loads.  After the last
// chunk a stage flagged kStageEnd tells the tensor-core thread to stop.
__device__ void control_thread(const Params &p, const Smem &s, int pre) {
    volatile int *abort_flag = s.abort_flag;
    const int64_t npre = pre > 0 ? pre : 0;     // chunks whose weight tile is requested
    int stage = 0;
    uint32_t phase = 0;
    bool ok = true;
    int64_t count = 0;
    for (int64_t wseq = 0;; ++wseq) {
        const int buf = (int)(wseq % kWinBufs);
        BP_TR(256 + wseq, 0);
        if (!mbar_wait(&s.pfull[buf], (uint32_t)((wseq / kWinBufs) & 1), p.watchdog_ns,
                       abort_flag)) {
            ok = false;
            break;
        }
        BP_TR(256 + wseq, 2);
        const int64_t *wm = s.wmeta + kWmeta * buf;
        const int64_t wcnt = wm[0];
        if (wcnt == 0) break;       // no more windows
        const int64_t wn0 = wm[1], wc0 = wm[2];
        const uint32_t wfl = (uint32_t)wm[3];
        const int32_t wh0 = (int32_t)wm[4], wimg0 = (int32_t)wm[5];
        const uint8_t *recs = s.win + buf * kWinBytes;
        // flags of the window's chunks: the unit's first and last chunk, and
        // whether the unit is the CTA's final one
        const uint32_t ufin = (wfl & kWinFinal) ? kStageFinal : 0u;
        const int64_t jfirst = (wfl & kWinFirst) ? 0 : -1, jlast = (wfl & kWinLast) ? wcnt - 1 : -1;
        for (int64_t j = 0; j < wcnt; ++j) {
            const int64_t seq = count;
            BP_TR(seq, 4);
            if (!mbar_wait(&s.empty[stage], phase ^ 1u, p.watchdog_ns, abort_flag)) {
                ok = false;
                break;
            }
            BP_TR(seq, 0);
            const uint32_t uflag =
                (j == jfirst ? kStageFirst : 0u) | (j == jlast ? kStageLast | ufin : 0u);
            // the plan: words 0..11 in three 16-byte loads
            const uint4 *pv = reinterpret_cast<const uint4 *>(recs + j * kMetaBytes + kListBytes);
            const uint4 q0 = pv[0], q1 = pv[1], q2 = pv[2];
            const int nb = (int)q0.x;
            const bool tma = nb > 0 && !p.direct;
            ++count;
            // the weight tile of the first chunks was requested before the
            // dependency wait
            const bool wpre = seq < npre;
            if (p.impl && !(blockIdx.x == 0 && seq == p.drop_stage)) {
                // implicit convolution: the weight tile and one box of 64
                // channels at kernel position (i, j) for the tile's pixels (the
                // padding and channels past C read as zeros)
                const int32_t d = *reinterpret_cast<const int32_t *>(recs + j * kMetaBytes);
                // window offset (di, dj) of kernel position (i, j); stride 2: the
                // phase it falls in and the offset within that phase
                int di = ((d >> 8) & 0xff) - p.i_ph, dj = (d & 0xff) - p.i_pw, img = 0;
                if (p.i_s == 2) {
                    img = (di & 1) * 2 + (dj & 1);
                    di >>= 1;       // floor((d - phase) / 2) = floor(d / 2)
                    dj >>= 1;
                }
                s.sflag[stage] = kStageTma | uflag;
                mbar_arrive_expect_tx(&s.wfull[stage], (wpre ? 0u : kWTileBytes) + p.i_box_bytes);
                if (!wpre)
                    bulk_g2s(smem_u32(s.w + stage * kWTileBytes),
                             p.tiles + (wc0 + j) * (int64_t)kWTileBytes, kWTileBytes,
                             &s.wfull[stage]);
                tma_load_4d(smem_u32(s.x + stage * kXTileBytes), &p.imap, (d >> 16) * 64, dj,
                            wh0 + di, img * (int32_t)p.i_Nb + wimg0,
                            &s.wfull[stage]);
            } else if (!(blockIdx.x == 0 && seq == p.drop_stage)) {
                s.sflag[stage] = (tma ? kStageTma : 0u) | uflag;  // read by the MMA thread after wfull
                mbar_arrive_expect_tx(&s.wfull[stage],
                                      (wpre ? 0u : kWTileBytes) +
                                          (tma ? (uint32_t)p.xboxes * (kBK * 128) : 0u));
                BP_TR(seq, 6);
                if (!wpre)
                    bulk_g2s(smem_u32(s.w + stage * kWTileBytes),
                             p.tiles + (wc0 + j) * (int64_t)kWTileBytes, kWTileBytes,
                             &s.wfull[stage]);
                BP_TR(seq, 7);
                if (tma) {
                    // load b: rows y[b] .. + (8 << lg) - 1 of X into list positions
                    // 8g ..; x = a multiple of 64 tokens (16-byte aligned), and
                    // columns past N, rows past K read as zero
                    const uint32_t ys[8] = {q0.y, q0.z, q0.w, q1.x, q1.y, q1.z, q1.w, q2.x};
                    const uint32_t xs = smem_u32(s.x + stage * kXTileBytes);
#pragma unroll
                    for (int b = 0; b < kMaxBoxes; ++b) {
                        if (b >= nb) break;
                        const uint32_t d = ((b < 4 ? q2.y : q2.z) >> (8 * (b & 3))) & 0xffu;
                        const uint32_t dst = xs + (d & 7u) * 1024;
                        const CUtensorMap *map = &p.xmap[(d >> 4) & 3u];
#pragma unroll
                        for (int cn = 0; cn < p.xboxes; ++cn)
                            tma_load_2d(dst + cn * 8192, map, (int32_t)(wn0 + cn * 64),
                                        (int32_t)ys[b], &s.wfull[stage]);
                    }
                }
            }
            if (++stage == p.stages) {
                stage = 0;
                phase ^= 1u;
            }
        }
        if (!ok) break;
        mbar_arrive(&s.pempty[buf]);
    }
    if (ok) {
        // no more chunks: the end marker for the tensor-core thread
        if (mbar_wait(&s.empty[stage], phase ^ 1u, p.watchdog_ns, abort_flag)) {
            s.sflag[stage] = kStageEnd;
            mbar_arrive_cnt(&s.wfull[stage], kStageArrivals);
        } else {
            ok = false;
        }
    }
    if (!ok) {
        raise_timeout(p, s);
        // unwinding: the copies of the last stages and the window copies may still
        // be in flight; let them land before the CTA exits.  A stage completes
        // once its TMA bytes have landed and its arrivals are in: the ones of
        // gather warps that left their loop before the chunk, and this thread's
        // own for a chunk whose weight tile was requested before the dependency
        // wait but not reached, are added here.  The gather warps leave once
        // they see the abort flag; their progress is read after they have.
        const volatile int64_t *gprog = s.gprog;
        {
            uint64_t deadline = 0;
            for (uint32_t it = 1; gprog[kGatherWarps] < kGatherWarps; ++it) {
                __nanosleep(64);
                if ((it & 15u) == 0u) {
                    const uint64_t now = globaltimer_ns();
                    if (deadline == 0) deadline = now + kDrainNs;
                    else if (now > deadline) break;
                }
            }
        }
        const int64_t reach = count > npre ? count : npre;
        for (int64_t q = reach > p.stages ? reach - p.stages : 0; q < reach; ++q) {
            if (blockIdx.x == 0 && q == p.drop_stage) continue;
            uint32_t missing = q >= count ? 1u : 0u;
            const int g0 = (int)(q % kGatherGroups) * kGroupWarps;
            for (int w = g0; w < g0 + kGroupWarps; ++w)
                if (gprog[w] <= q) missing += 32u;
            if (missing) mbar_arrive_cnt(&s.wfull[q % p.stages], missing);
            if (!mbar_wait(&s.wfull[q % p.stages], (uint32_t)((q / p.stages) & 1), kDrainNs,
                           nullptr))
                atomicOr(p.status, kDevTimeout);
        }
    }
}

// ------------------------------------------------------------------ MMA issuer
__device__ void mma_issuer(const Params &p, const Smem &s, uint32_t tmem) {
    // Everything the loop needs lives in registers: the per-chunk path is a
    // chain of dependent barrier probes and issues, so any reload from the
    // parameter bank or shared memory adds to every chunk.  The thread decodes
    // no work units: each stage's flags (set by the control thread) say where
    // its chunk sits in its unit, and a stage flagged kStageEnd ends the loop.
    volatile int *abort_flag = s.abort_flag;
    const uint64_t wdog = p.watchdog_ns;
    const int nst = (int)p.stages;
    const uint32_t acc_cols = p.acc_cols;
    uint64_t *const wfull = s.wfull, *const empty = s.empty;
    const volatile uint32_t *const sflag = s.sflag;
    // B: MN-major activation rows, or for the implicit convolution K-major
    // pixel rows (both with the 128-byte swizzle)
    const uint32_t idesc = make_idesc(p.dtype == BP_BF16, false, !p.impl, kSlab, p.nt);
    // descriptors of stage 0; a stage / K=16 step adds its byte offset / 16 to
    // the start-address field (shared addresses stay below 256 KB: no carry)
    const uint64_t wdesc0 = make_sdesc_sw128(smem_u32(s.w), 16, 1024);
    const uint64_t xdesc0 = p.impl ? make_sdesc_sw128(smem_u32(s.x), 16, 1024)
                                   : make_sdesc_sw128(smem_u32(s.x), 8192, 1024);
    // one K=16 step: 16 activation rows (MN-major) or 32 bytes of every pixel
    // row (implicit: K-major pixel rows of 64 channels)
    const uint32_t xkstep = p.impl ? 32u >> 4 : 2048u >> 4;
    int stage = 0;
    uint32_t phase = 0;
    int acc = 0;
    uint32_t acc_phase = 0;
    uint32_t d = tmem;
#ifdef BP_TRACE
    int64_t tseq = 0, titem = 0;
#else
    constexpr int64_t tseq = 0;
#endif
    bool ready = mbar_test_wait(&wfull[0], 0);
    for (;;) {
        if (!ready && !mbar_wait(&wfull[stage], phase, wdog, abort_flag)) {
            raise_timeout(p, s);
            break;
        }
        BP_TR(tseq, 3);
        const uint32_t f = sflag[stage];
        if (f & kStageEnd) break;
        // gathered rows: order their generic-proxy (cp.async) writes, acquired
        // through the barrier, before the tensor core's async-proxy reads
        if (!(f & kStageTma)) fence_proxy_async_smem();
        if (f & kStageFirst) {
            // a unit's first chunk: the next accumulator, once drained
            if (!mbar_wait(&s.tempty[acc], acc_phase ^ 1u, wdog, abort_flag)) {
                raise_timeout(p, s);
                break;
            }
#ifdef BP_TRACE
            BP_TR(384 + titem, 4);
            ++titem;
#endif
            d = tmem + acc * acc_cols;
        }
        // order the MMAs below after the barrier waits above
        tc_fence_after();
        const uint64_t wd = wdesc0 + (uint32_t)(stage * (kWTileBytes >> 4));
        const uint64_t xd = xdesc0 + (uint32_t)(stage * (kXTileBytes >> 4));
        const int nstage = stage + 1 == nst ? 0 : stage + 1;
        const uint32_t nphase = stage + 1 == nst ? phase ^ 1u : phase;
        // probe the next stage now: the answer is needed only after the MMAs
        // below have been issued
        ready = mbar_test_wait(&wfull[nstage], nphase);
        const uint32_t acc0 = (f & kStageFirst) ? 0u : 1u;
#pragma unroll
        for (int kk = 0; kk < kBK / 16; ++kk)
            umma_f16_ss(d, wd + kk * (32 >> 4), xd + kk * xkstep, idesc, kk > 0 ? 1u : acc0);
        umma_commit(&empty[stage]);
        BP_TR(tseq, 5);
#ifdef BP_TRACE
        ++tseq;
#endif
        if (f & kStageLast) {
            umma_commit(&s.tfull[acc]);
            if (f & kStageFinal) umma_commit(s.ffull);
            if (++acc == 2) {
                acc = 0;
                acc_phase ^= 1u;
            }
        }
        stage = nstage;
        phase = nphase;
    }
    // all issued tensor-core work must finish before tensor memory is freed
    umma_commit(s.drain);
    if (!mbar_wait(s.drain, 0, kDrainNs, nullptr)) atomicOr(p.status, kDevTimeout);
}

// ------------------------------------------------------------------ epilogue
// slot 0: an epilogue warp, every item; slots 1, 2: gather warps 0-3 and 4-7
// after their last gather, the final item only.  The final item's 64-column
// pairs k go to slot k mod 3 of the warps of each quadrant.
template <bool kSplit, bool kConv>
__device__ void epilogue(const Params &p, const Smem &s, uint32_t tmem, int slot) {
    const int64_t *kcp = s.kc ? s.kc : p.kc_ptr;
    volatile int *abort_flag = s.abort_flag;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int q = warp & 3;                  // tensor-memory lane quadrant this warp may read
    // 4 KB of staging per warp: the epilogue's own area, or for a gather warp
    // the idle activation stage area
    uint8_t *const stgp = slot == 0 ? s.ystage + (warp - kEpiWarp0) * 4096 : s.x + warp * 4096;
    const uint32_t stg = smem_u32(stgp);
    uint32_t yseq = 0;                       // TMA box stores issued by this warp
    // a 64-column box whose left half (the previous group) is staged, and where
    // it goes; whether the last store issued was such a box
    bool pend = false, prev_big = false;
    int64_t pn = 0;
    uint32_t pbb = 0, phw = 0;
    int acc = 0;
    uint32_t acc_phase = 0;
#ifdef BP_TRACE
    int64_t titem = 0, tgrp = 0;
#define BP_TRE(ev)                                                 \
    do {                                                           \
        if (warp == kEpiWarp0 && lane == 0) BP_TR(512 + tgrp, ev); \
    } while (0)
#else
#define BP_TRE(ev) \
    do {           \
    } while (0)
#endif
    UnitIter ui;
    Item t;
    for (ui.init(p, s.skv); ui.valid(); ui.step(p, t)) {
        t = ui.get(p, kcp);
        const bool has = t.nkc > 0;
        const bool fin = !kSplit && final_unit(p, ui, t);
        if (slot > 0 && !fin) {
            if (has && ++acc == 2) {      // the accumulator this item used
                acc = 0;
                acc_phase ^= 1u;
            }
            continue;
        }
        // lane = output row of the slab; its bias is requested before the wait
        const int64_t row0 = 32 * q;
        const bool vrow = row0 + lane < t.rows;
        const int64_t m = t.slab * kSlab + row0 + lane;
        const float bv = (p.bias && vrow) ? p.bias[m] : 0.f;
        if (has) {
            // warp-uniform outcome: tcgen05.ld below is a warp-collective instruction
            const bool ok = slot > 0 ? mbar_wait(s.ffull, 0, p.watchdog_ns, abort_flag)
                                     : mbar_wait(&s.tfull[acc], acc_phase, p.watchdog_ns, abort_flag);
            if (!__all_sync(0xffffffffu, ok)) {
                raise_timeout(p, s);
                break;
            }
            tc_fence_after();
        }
#ifdef BP_TRACE
        if (warp == kEpiWarp0 && lane == 0) BP_TR(384 + titem, 5);
#endif
        // tensor-memory lanes = the warp's rows; columns = the tile's columns
        const uint32_t tacc = tmem + ((uint32_t)(32 * q) << 16) + acc * p.acc_cols;
        // this warp's groups: all, or for the final item the 64-column pairs
        // k = slot (mod 3): first group and the step between pairs
        const int g0 = fin ? 2 * slot : 0, pstep = fin ? 3 : 1;
        // convolution: (image, pixel) of the next 32-column group to store
        uint32_t cbb = 0, chw = 0;
        if (kConv) {
            const uint32_t n1 = (uint32_t)t.n0 + 32u * (uint32_t)g0;
            cbb = n1 / (uint32_t)p.HoWo;
            chw = n1 - cbb * (uint32_t)p.HoWo;
        }
        // Column groups of 32: once group g's accumulators are converted (pk),
        // the tensor-memory load of group g + 1 is issued into the same
        // registers and runs while group g is stored.
        // A warp whose 32 rows are all past the slab's real rows has nothing to write.
        // bias + ReLU + cast of a 32-column group, one branch per group
        auto pack = [&](const uint32_t (&r)[32], uint32_t (&pk)[16]) { cvt_any(p, r, bv, pk); };
        // 64-column output boxes: an even group whose pair lies in the tile (and,
        // for NCHW, in one image) is staged as the left half of a 64 x 32 box
        // (128-byte swizzle: chunk c of row r at c ^ (r & 7)); the next group
        // adds the right half and issues one TMA store for both.  Returns true
        // when the group was handled here.
        auto stage_pair = [&](const uint32_t (&pk)[16], int c0, int64_t n, uint32_t bb,
                              uint32_t hw) -> bool {
            if (pend) {
                BP_TRE(0);
                BP_TRE(1);
                pend = false;
#pragma unroll
                for (int ch = 0; ch < 4; ++ch)
                    st_shared_v4(stg + lane * 128 + (((ch + 4) ^ (lane & 7)) << 4),
                                 make_uint4(pk[4 * ch], pk[4 * ch + 1], pk[4 * ch + 2], pk[4 * ch + 3]));
                fence_proxy_async_smem();
                __syncwarp();
                BP_TRE(2);
                if (lane == 0) {
                    if (kConv)
                        tma_store_3d(&p.ymap64, stg, (int32_t)phw, (int32_t)(t.slab * kSlab + row0),
                                     (int32_t)pbb);
                    else
                        tma_store_2d(&p.ymap64, stg, (int32_t)pn, (int32_t)(t.slab * kSlab + row0));
                    bulk_commit();
                }
                prev_big = true;
                BP_TRE(3);
                return true;
            }
            const bool pair = p.ytma && (c0 & 63) == 0 && c0 + 64 <= t.ncols &&
                              (!kConv || (hw + 64 <= (uint32_t)p.HoWo && (hw & 7u) == 0));
            if (!pair) return false;
            BP_TRE(0);
            if (lane == 0) bulk_wait_read<0>();     // every earlier store read its box
            __syncwarp();
            BP_TRE(1);
#pragma unroll
            for (int ch = 0; ch < 4; ++ch)
                st_shared_v4(stg + lane * 128 + ((ch ^ (lane & 7)) << 4),
                             make_uint4(pk[4 * ch], pk[4 * ch + 1], pk[4 * ch + 2], pk[4 * ch + 3]));
            pend = true;
            pn = n;
            pbb = bb;
            phw = hw;
            BP_TRE(2);
            BP_TRE(3);
            return true;
        };
        auto store = [&](const uint32_t (&pk)[16], int c0) {
            const int64_t n = t.n0 + c0;
#ifdef BP_EPI_DIRECT
            // (Measurement build.)  The 32 x 32 box goes through shared memory
            // (row = lane, 64 bytes; 16-byte chunk c of row r at c ^ ((r >> 1) &
            // 3), conflict-free both ways) and back out row by row with plain
            // stores: per instruction 8 rows x 64 contiguous bytes, lanes 4r ..
            // 4r + 3 on row r; the box's buffer alternates over the warp's
            // groups.  Measured slower than the TMA box stores below on every
            // workload (the 4096^3 layer 43.6 against 41.9 us, BERT 3072 x 768
            // 32.1 against 25.5 us): the stores share the load/store unit with
            // the activation gathers.
            if (!kConv || p.yvec) {
                const uint32_t sb = stg + (yseq & 1u) * 2048;
                ++yseq;
#pragma unroll
                for (int ch = 0; ch < 4; ++ch)
                    st_shared_v4(sb + lane * 64 + ((ch ^ ((lane >> 1) & 3)) << 4),
                                 make_uint4(pk[4 * ch], pk[4 * ch + 1], pk[4 * ch + 2],
                                            pk[4 * ch + 3]));
                __syncwarp();
                const int c = lane & 3;
                const int64_t nc = n + 8 * c;          // this lane's 8 columns
                const int64_t nend = kConv ? t.n0 + t.ncols : p.N;
                uint16_t *dst0;
                if (kConv) {
                    // NCHW, Ho*Wo a multiple of 8 and nc too: the 8 pixels lie in one
                    // image, 16-byte aligned
                    const uint32_t bb = (uint32_t)nc / (uint32_t)p.HoWo;
                    const uint32_t hw = (uint32_t)nc - bb * (uint32_t)p.HoWo;
                    dst0 = p.Y + ((int64_t)bb * p.M + t.slab * kSlab + row0) * p.HoWo + hw;
                } else {
                    dst0 = p.Y + (t.slab * kSlab + row0) * p.ldy + nc;
                }
                const int64_t ystride = kConv ? p.HoWo : p.ldy;
#pragma unroll
                for (int it = 0; it < 4; ++it) {
                    const int rr = it * 8 + (lane >> 2);
                    const uint4 v = ld_shared_v4(sb + rr * 64 + ((c ^ ((rr >> 1) & 3)) << 4));
                    if (row0 + rr < t.rows && nc < nend) {
                        uint16_t *dst = dst0 + rr * ystride;
                        if (nc + 8 <= nend) {
                            *reinterpret_cast<uint4 *>(dst) = v;
                        } else {
                            const uint32_t w[4] = {v.x, v.y, v.z, v.w};
                            for (int u = 0; u < 8 && nc + u < nend; ++u)
                                dst[u] = (uint16_t)(w[u >> 1] >> (16 * (u & 1)));
                        }
                    }
                }
                return;
            }
#endif
            if (kConv) {
                // NCHW output, pixel n = b*HoWo + hw is element (b, m, hw); the
                // groups are stored in order, so (b, hw) advances by 32 pixels
                // per call from the item's first pixel
                const uint32_t bb = cbb, hw = chw;
                {
                    // one division instead of a loop per image passed (images of
                    // a few pixels pass eight per group; the loop's dependent
                    // steps on the captured counters cost ~850 cycles on 2 x 2)
                    const uint32_t nh = chw + 32u, HWu = (uint32_t)p.HoWo;
                    const uint32_t adv = nh >= HWu ? nh / HWu : 0u;
                    cbb += adv;
                    chw = nh - adv * HWu;
                }
                if (stage_pair(pk, c0, n, bb, hw)) return;
                if (p.ytma && hw + 32 <= (uint32_t)p.HoWo && c0 + 32 <= t.ncols && (hw & 7u) == 0) {
                    // the 32 pixels lie in one image and in the tile: stage the box
                    // like a GEMM box (below) and store it at (hw, m, b) of the
                    // 3-D output map (a TMA store needs hw 16-byte aligned)
                    BP_TRE(0);
                    const uint32_t sb = stg + (yseq & 1u) * 2048;
                    ++yseq;
                    if (lane == 0) {
                        if (prev_big) bulk_wait_read<0>();
                        else bulk_wait_read<1>();
                    }
                    prev_big = false;
                    __syncwarp();
                    BP_TRE(1);
#pragma unroll
                    for (int ch = 0; ch < 4; ++ch)
                        st_shared_v4(sb + lane * 64 + ((ch ^ ((lane >> 1) & 3)) << 4),
                                     make_uint4(pk[4 * ch], pk[4 * ch + 1], pk[4 * ch + 2],
                                                pk[4 * ch + 3]));
                    fence_proxy_async_smem();
                    __syncwarp();
                    BP_TRE(2);
                    if (lane == 0) {
                        tma_store_3d(&p.ymap, sb, (int32_t)hw, (int32_t)(t.slab * kSlab + row0),
                                     (int32_t)bb);
                        bulk_commit();
                    }
                    BP_TRE(3);
                    return;
                }
                // Ho*Wo not a multiple of 8, the 32 pixels cross an image
                // boundary or the tile's end: stage the 32 x 32 box (lane = channel row, 80-byte
                // rows), then write it with lanes along the pixels, one
                // coalesced 64-byte store per channel
                const int rmax = (int)min((int64_t)32, t.rows - row0);
                // Ho*Wo dividing 32 and the group starting at an image: the group
                // holds whole images, and each image's 32 channels x Ho*Wo pixels
                // are one run of 64 Ho*Wo contiguous bytes of the NCHW output,
                // written from registers (store_images).  (One 2-byte store per
                // lane and channel, pixels across lanes, took ~3,000 cycles per
                // group on 2 x 2 images.)
                {
                    const uint32_t HW = (uint32_t)p.HoWo;
                    const int64_t cols = min((int64_t)32, t.n0 + t.ncols - n);
                    if (hw == 0u && HW < 32u && (32u % HW) == 0u && rmax == 32 && cols > 0 &&
                        cols % HW == 0) {
                        store_images(p.Y + ((int64_t)bb * p.M + t.slab * kSlab + row0 + lane) * HW,
                                     (int64_t)p.M * HW, HW, (int)(cols / HW), pk);
                        return;
                    }
                }
                uint8_t *box = stgp;
                // the box overlaps both TMA staging boxes: their stores must
                // have read them
                if (p.ytma && lane == 0) bulk_wait_read<0>();
                __syncwarp();                      // the previous box has been read
#pragma unroll
                for (int ch = 0; ch < 4; ++ch)
                    st_shared_v4(smem_u32(box + lane * 80 + ch * 16),
                                 make_uint4(pk[4 * ch], pk[4 * ch + 1], pk[4 * ch + 2], pk[4 * ch + 3]));
                __syncwarp();
                const int64_t nn = n + lane;
                // only the tile's own pixels: an implicit convolution's tile
                // holds fewer pixels than the MMA's N
                if (nn < t.n0 + t.ncols && rmax > 0) {
                    const uint32_t bb = (uint32_t)nn / (uint32_t)p.HoWo;
                    const uint32_t hw = (uint32_t)nn - bb * (uint32_t)p.HoWo;
                    uint16_t *dst = p.Y + ((int64_t)bb * p.M + t.slab * kSlab + row0) * p.HoWo + hw;
                    const uint16_t *src = reinterpret_cast<const uint16_t *>(box) + lane;
                    for (int r = 0; r < rmax; ++r) dst[r * p.HoWo] = src[r * 40];
                }
                return;
            }
            // GEMM: 32 x 32 box staged in shared memory (64-byte swizzle: 16-byte
            // chunk c of row r sits at chunk c ^ ((r >> 1) & 3)), then TMA-stored;
            // rows past M and columns past N of the box are not written
            // the two boxes alternate over the warp's stores, across items (an
            // item may have an odd number of groups): the box about to be written
            // was used by the store before last
            if (stage_pair(pk, c0, n, 0u, 0u)) return;
            BP_TRE(0);
            const uint32_t sb = stg + (yseq & 1u) * 2048;
            ++yseq;
            if (lane == 0) {                        // the store that used this box is done
                if (prev_big) bulk_wait_read<0>();
                else bulk_wait_read<1>();
            }
            prev_big = false;
            __syncwarp();
            BP_TRE(1);
#pragma unroll
            for (int ch = 0; ch < 4; ++ch)
                st_shared_v4(sb + lane * 64 + ((ch ^ ((lane >> 1) & 3)) << 4),
                             make_uint4(pk[4 * ch], pk[4 * ch + 1], pk[4 * ch + 2], pk[4 * ch + 3]));
            fence_proxy_async_smem();
            __syncwarp();
            BP_TRE(2);
            if (lane == 0) {
                tma_store_2d(&p.ymap, sb, (int32_t)n, (int32_t)(t.slab * kSlab + row0));
                bulk_commit();
            }
            BP_TRE(3);
                };
        const int64_t cols = t.ncols;
        const int G = (int)((cols + 31) / 32);
        if (row0 < t.rows && g0 < G) {
            uint32_t r[32], pk[16];
            if (has) {
                tmem_ld_32x32b_x32(tacc + 32 * g0, r);
                tmem_ld_wait();
            } else {
#pragma unroll
                for (int e = 0; e < 32; ++e) r[e] = 0u;
            }
            constexpr int64_t kQuad = 8 * 8 * 32;            // float4 per (tile, quadrant)
            if (kSplit && t.role == 2) {
                // Balanced launch, a later range of the item's chunks: this CTA's
                // fp32 partial rows go to its own tile of the workspace, then the
                // quadrant's flag is raised for the CTA that finishes the item.
                float4 *slot = reinterpret_cast<float4 *>(p.part) +
                               ((int64_t)blockIdx.x * 4 + q) * kQuad + lane;
                for (int g = 0; g < G; ++g) {
#pragma unroll
                    for (int e = 0; e < 8; ++e)
                        __stcg(slot + (g * 8 + e) * 32,
                               make_float4(__uint_as_float(r[4 * e]), __uint_as_float(r[4 * e + 1]),
                                           __uint_as_float(r[4 * e + 2]), __uint_as_float(r[4 * e + 3])));
                    if (g + 1 < G) {
                        tmem_ld_32x32b_x32(tacc + 32 * (g + 1), r);
                        tmem_ld_wait();
                    }
                }
                __threadfence();
                __syncwarp();
                if (lane == 0) st_release_gpu(p.cnt + (int64_t)blockIdx.x * 4 + q, 1);
            } else if (kSplit && t.role == 1) {
                // Balanced launch, the item's first chunks: add the partial rows of
                // the CTAs that own the rest of its chunks (each raised its flag
                // first thing in its range), then the usual epilogue.  This is the
                // CTA's last unit, so its pipeline stages are idle: the first
                // partial's quadrant (32 KB) comes in with one TMA bulk copy into
                // the stage area (a latency-bound load loop over eight column
                // groups measured several microseconds); further partials (items
                // spread over three or more ranges) are read directly.
                const int64_t c0 = sk_owner(s.skv, t.gpos + t.nkc);
                const int64_t c1 = sk_owner(s.skv, t.gpos + t.nitem - 1);
                const float4 *part4 = reinterpret_cast<const float4 *>(p.part);
                uint8_t *fbuf = s.w + q * (kQuad * 16);
                bool okw = true;
                if (lane == 0) {
                    for (int64_t c = c0; c <= c1 && okw; ++c)
                        okw = wait_flag_gpu(p.cnt + c * 4 + q, p.watchdog_ns, abort_flag);
                    if (okw) {
                        mbar_arrive_expect_tx(&s.fixbar[q], (uint32_t)(kQuad * 16));
                        bulk_g2s(smem_u32(fbuf), part4 + (c0 * 4 + q) * kQuad,
                                 (uint32_t)(kQuad * 16), &s.fixbar[q]);
                        okw = mbar_wait(&s.fixbar[q], 0, p.watchdog_ns, abort_flag);
                    }
                }
                okw = __shfl_sync(0xffffffffu, okw ? 1 : 0, 0) != 0;
                if (!okw) raise_timeout(p, s);
                const float4 *sm4 = reinterpret_cast<const float4 *>(fbuf) + lane;
                for (int g = 0; g < G && okw; ++g) {
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        const float4 v = sm4[(g * 8 + e) * 32];
                        r[4 * e] = __float_as_uint(__uint_as_float(r[4 * e]) + v.x);
                        r[4 * e + 1] = __float_as_uint(__uint_as_float(r[4 * e + 1]) + v.y);
                        r[4 * e + 2] = __float_as_uint(__uint_as_float(r[4 * e + 2]) + v.z);
                        r[4 * e + 3] = __float_as_uint(__uint_as_float(r[4 * e + 3]) + v.w);
                    }
                    for (int64_t c = c0 + 1; c <= c1; ++c) {
                        const float4 *src = part4 + (c * 4 + q) * kQuad + lane + g * 8 * 32;
                        float4 v[8];
#pragma unroll
                        for (int e = 0; e < 8; ++e) v[e] = __ldcg(src + e * 32);
#pragma unroll
                        for (int e = 0; e < 8; ++e) {
                            r[4 * e] = __float_as_uint(__uint_as_float(r[4 * e]) + v[e].x);
                            r[4 * e + 1] = __float_as_uint(__uint_as_float(r[4 * e + 1]) + v[e].y);
                            r[4 * e + 2] = __float_as_uint(__uint_as_float(r[4 * e + 2]) + v[e].z);
                            r[4 * e + 3] = __float_as_uint(__uint_as_float(r[4 * e + 3]) + v[e].w);
                        }
                    }
                    pack(r, pk);
                    if (g + 1 < G) tmem_ld_32x32b_x32(tacc + 32 * (g + 1), r);
                    store(pk, 32 * g);
                    if (g + 1 < G) tmem_ld_wait();
                }
                // zero the flags again for the next launch (read, and only written
                // again, after this launch: launches on one stream are ordered)
                if (lane == 0 && okw)
                    for (int64_t c = c0; c <= c1; ++c) p.cnt[c * 4 + q] = 0;
            } else if (!kSplit || t.S == 1) {
                for (int g = g0; g < G;) {
                    // the next group of this warp: the pair's second, or the
                    // first of its next pair
                    const int gn = (g & 1) == 0 ? g + 1 : g + 1 + 2 * (pstep - 1);
                    BP_TRE(4);
                    pack(r, pk);
                    BP_TRE(6);
                    if (has && gn < G) tmem_ld_32x32b_x32(tacc + 32 * gn, r);
                    BP_TRE(7);
                    store(pk, 32 * g);
                    if (kConv && gn != g + 1) {
                        // skipped pairs (their pixels) before the next group
                        const uint32_t nh = chw + 32u * (uint32_t)(gn - g - 1), HWu = (uint32_t)p.HoWo;
                        const uint32_t adv = nh >= HWu ? nh / HWu : 0u;
                        cbb += adv;
                        chw = nh - adv * HWu;
                    }
                    if (has && gn < G) tmem_ld_wait();
                    BP_TRE(5);
#ifdef BP_TRACE
                    ++tgrp;
#endif
                    g = gn;
                }
            } else {
                // Split item: the units of an item add their fp32 partial rows
                // into the item's accumulator tile in the workspace with vector
                // reductions (no value returned, so no unit waits on them); the
                // unit whose arrival completes the (item, quadrant) count reads
                // the sum back, zeroes the tile again for the next launch and
                // writes the output.  No unit waits for another.  Tile layout
                // per quadrant: [group][8 float4][lane], so each warp access is
                // 512 contiguous bytes.  (Summing per-unit partial tiles in the
                // last unit instead left that unit reading S x 128 KB alone,
                // latency-bound: 20-30 us on the 512-filter VGG-16 layers.)
                float4 *acc4 = reinterpret_cast<float4 *>(p.part) + (t.j * 4 + q) * kQuad;
#ifdef BP_TRACE
#define BP_TRS(ev)                                                                     \
    do {                                                                               \
        if (lane == 0 && ((ev) < 4 ? blockIdx.x == 0 : t.j == 0))                       \
            bp::g_trace[(1000 + q) * bp::kTraceEvents + (ev)] = clock64();             \
    } while (0)
#else
#define BP_TRS(ev) \
    do {           \
    } while (0)
#endif
                BP_TRS(0);
                if (has) {
                    for (int g = 0; g < G; ++g) {
#pragma unroll
                        for (int e = 0; e < 8; ++e)
                            red_add_f32x4(acc4 + (g * 8 + e) * 32 + lane, __uint_as_float(r[4 * e]),
                                          __uint_as_float(r[4 * e + 1]), __uint_as_float(r[4 * e + 2]),
                                          __uint_as_float(r[4 * e + 3]));
                        if (g + 1 < G) {
                            tmem_ld_32x32b_x32(tacc + 32 * (g + 1), r);
                            tmem_ld_wait();
                        }
                    }
                }
                BP_TRS(1);
                __threadfence();
                __syncwarp();
                BP_TRS(2);
                int last = 0;
                if (lane == 0) last = atomicAdd(p.cnt + t.j * 4 + q, 1) == t.S - 1;
                BP_TRS(3);
                if (__shfl_sync(0xffffffffu, last, 0)) {
                    __threadfence();
                    if (lane == 0) p.cnt[t.j * 4 + q] = 0;     // zero again for the next launch
                    // Every CTA of a split launch runs one unit, so its activation
                    // stages are idle now: the quadrant's 32 KB of sums come in
                    // with one TMA bulk copy (plain loads, 8 per lane in flight,
                    // would take a round trip per column group).
                    uint8_t *qbuf = s.w + q * (kQuad * 16);    // inside the stage area (checked at launch)
                    bool okw = true;
                    if (lane == 0) {
                        fence_proxy_async_global();
                        mbar_arrive_expect_tx(&s.fixbar[q], (uint32_t)(kQuad * 16));
                        bulk_g2s(smem_u32(qbuf), acc4, (uint32_t)(kQuad * 16), &s.fixbar[q]);
                    }
                    okw = mbar_wait(&s.fixbar[q], 0, p.watchdog_ns, abort_flag);
                    BP_TRS(4);
                    if (!__all_sync(0xffffffffu, okw)) {
                        raise_timeout(p, s);
                    } else {
                        BP_TRS(5);
                        const float4 *sm4 = reinterpret_cast<const float4 *>(qbuf) + lane;
                        // an NCHW output whose groups hold whole images: the runs
                        // are written here directly (the generic store path
                        // reloads its spilled per-item state every group, ~800
                        // cycles of round trips per group)
                        const uint32_t HWw = kConv ? (uint32_t)p.HoWo : 1u;
                        const bool whole = kConv && HWw < 32u && (32u % HWw) == 0u &&
                                           (uint32_t)t.n0 % HWw == 0u && row0 + 32 <= t.rows;
                        uint16_t *yw = nullptr;
                        int64_t iw = 0;
                        if (whole) {
                            iw = (int64_t)p.M * HWw;
                            yw = p.Y + (((int64_t)t.n0 / HWw) * p.M + t.slab * kSlab + row0 + lane) * HWw;
                        }
                        for (int g = 0; g < G; ++g) {
#pragma unroll
                            for (int e = 0; e < 8; ++e) {
                                const float4 v = sm4[(g * 8 + e) * 32];
                                r[4 * e] = __float_as_uint(v.x);
                                r[4 * e + 1] = __float_as_uint(v.y);
                                r[4 * e + 2] = __float_as_uint(v.z);
                                r[4 * e + 3] = __float_as_uint(v.w);
                            }
                            pack(r, pk);
                            if (whole) {
                                const int cols = (int)min((int64_t)32, t.ncols - 32 * g);
                                store_images(yw + (int64_t)(32 / HWw) * g * iw, iw, HWw, cols / (int)HWw, pk);
                            } else {
                                store(pk, 32 * g);
                            }
#ifdef BP_TRACE
                            if (lane == 0 && g < 8 && t.j == 0)
                                bp::g_trace[(1004 + q) * bp::kTraceEvents + g] = clock64();
#endif
                        }
                        // the copy has read the tile: zero it for the next launch
                        // (after the output, which the next layer waits for)
                        for (int i = 0; i < 8 * 8; ++i)
                            __stcg(acc4 + i * 32 + lane, make_float4(0.f, 0.f, 0.f, 0.f));
                        BP_TRS(6);
                    }
                }
#undef BP_TRS
            }
        }
        if (has && slot == 0) {
            tc_fence_before();
            mbar_arrive(&s.tempty[acc]);
            if (++acc == 2) {
                acc = 0;
                acc_phase ^= 1u;
            }
        }
#ifdef BP_TRACE
        if (warp == kEpiWarp0 && lane == 0) BP_TR(384 + titem, 6);
        ++titem;
#endif
    }
    if (p.ytma && lane == 0) bulk_wait_all();    // staged output fully written before exit
#undef BP_TRE
}

// kSplit: the launch has split items (a separate instantiation keeps the
// common kernel free of the partial-tile code); kConv: the output is the NCHW
// tensor of a convolution (GEMM launches compile no convolution store code).
template <bool kSplit, bool kConv>
__global__ void __launch_bounds__(kThreads, 1) bp_mma_kernel(const __grid_constant__ Params p) {
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    const Smem s = carve(smem_raw, p);
    const int warp = threadIdx.x >> 5;
    if (threadIdx.x == 0) {
        for (int i = 0; i < p.stages; ++i) {
            mbar_init(&s.wfull[i], kStageArrivals);
            mbar_init(&s.empty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&s.tfull[i], 1);
            mbar_init(&s.tempty[i], 128);
        }
        mbar_init(s.drain, 1);
        for (int i = 0; i < 4; ++i) mbar_init(&s.fixbar[i], 1);
        mbar_init(s.ffull, 1);
        for (int i = 0; i < kWinBufs; ++i) {
            mbar_init(&s.pfull[i], 1);
            mbar_init(&s.pempty[i], kGatherWarps + 1);
        }
        *s.abort_flag = 0;
        for (int i = 0; i <= kGatherWarps; ++i) s.gprog[i] = 0;
        fence_mbar_init();
    }
    if (warp == kMmaWarp) {
        tmem_alloc(s.tmem_base, p.tmem_cols);
        tmem_relinquish();
    }
    if (warp == kCtrlWarp && (threadIdx.x & 31) == 0)
        for (int i = 0; i < 4; ++i) prefetch_tmap(&p.xmap[i]);
    // Launched as a programmatic dependent: the set-up overlaps the end of the
    // previous kernel in the stream.  The packed image (written by bp_pack,
    // which synchronises) is read before the dependency wait: the chunk
    // pointers, the first window of chunk records and the first weight tiles.
    // The activations, the output and the workspace are touched only after
    // it (the previous kernel may have written the inputs, or still read the
    // output); then the next kernel may start its own set-up as SMs come free.
    if (s.kc)
        for (int64_t i = threadIdx.x; i < p.kc_cached; i += kThreads) s.kc[i] = p.kc_ptr[i];
    __syncthreads();
    int pre = -1;
    if (warp == kCtrlWarp && (threadIdx.x & 31) == 0) {
        pre = control_prefetch(p, s);
        *s.pre = pre;           // read by the scheduler warp after the barrier below
    }
    grid_dependency_wait();
    grid_launch_dependents();
#ifdef BP_TRACE
    if (threadIdx.x == 0 && blockIdx.x < 248) g_trace[448 * kTraceEvents + 2 * blockIdx.x] = globaltimer_ns();
    if (threadIdx.x == 0) BP_TR(511, 0);
#endif
    if (p.sk && threadIdx.x == 0) {
        // the balanced launch's constants, once per CTA (64-bit divisions)
        const int64_t tile = p.sk_i0 / p.num_slabs;
        const int64_t p0 = tile * p.kc_total + p.kc_ptr[p.sk_i0 - tile * p.num_slabs];
        const int64_t T = p.sk_total - p0;
        s.skv[0] = p0;
        s.skv[1] = T;
        s.skv[2] = p0 + (int64_t)blockIdx.x * T / gridDim.x;
        s.skv[3] = p0 + ((int64_t)blockIdx.x + 1) * T / gridDim.x;
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *s.tmem_base;

    if (warp < kGatherWarps) {
        gather_warps(p, s);
        // then a share of the final item's output (pipeline stages idle by then)
        if (!kSplit) epilogue<kSplit, kConv>(p, s, tmem, 1 + (warp >> 2));
    } else if (warp == kCtrlWarp) {
        if ((threadIdx.x & 31) == 0) control_thread(p, s, pre);
        __syncwarp();
    } else if (warp == kMmaWarp) {
        if ((threadIdx.x & 31) == 0) mma_issuer(p, s, tmem);
        __syncwarp();
    } else if (warp < kSchedWarp) {
        epilogue<kSplit, kConv>(p, s, tmem, 0);
    } else {
        if ((threadIdx.x & 31) == 0) scheduler_thread(p, s);
        __syncwarp();
    }

    tc_fence_before();
    __syncthreads();
    tc_fence_after();
#ifdef BP_TRACE
    if (threadIdx.x == 0 && blockIdx.x < 248) g_trace[448 * kTraceEvents + 2 * blockIdx.x + 1] = globaltimer_ns();
    if (threadIdx.x == 0) BP_TR(511, 1);
#endif
    if (warp == kMmaWarp) tmem_dealloc(tmem, p.tmem_cols);
}

// Activation columns per tile (the MMA's N; a multiple of 32, the epilogue's
// column group, from 64 to 256).  A chunk costs about the same whatever the
// width: its 64 activation rows take one gather instruction per row and warp,
// however many columns the lanes cover.  Persistent CTAs take work units in
// waves, each unit the same number of chunks, so the kernel lasts about
// (waves x chunks per unit): pick the widest tile with the fewest waves, no
// wider than N needs (the MMA's time does grow with the width).
int pick_tile_width(int64_t N, int64_t slabs, int sms) {
    const int widest = (int)std::max<int64_t>(64, std::min<int64_t>(kNT, (N + 31) / 32 * 32));
    int best = widest;
    int64_t best_waves = INT64_MAX;
    for (int nt = widest; nt >= 64; nt -= 32) {
        const int64_t items = (N + nt - 1) / nt * slabs;
        const int64_t waves = (items + sms - 1) / sms;
        if (waves < best_waves) {
            best_waves = waves;
            best = nt;
        }
    }
    return best;
}

}  // namespace

PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *f = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
    });
    return fn;
}

SplitPlan plan_split(const DevLayout &dl, int64_t N, bool allow_split, const ImplicitTiles *it) {
    SplitPlan sp{};
    const int sms = num_sms();
    sp.nt = it ? it->nt : pick_tile_width(N, dl.num_slabs, sms);
    sp.items = (it ? it->tiles : (N + sp.nt - 1) / sp.nt) * dl.num_slabs;
    sp.full = sp.items;
    sp.split = 1;
    // chunks of all slabs (the implicit convolution's section: its capacity)
    const int64_t kct = it ? dl.c3max : dl.kc_total;
    if (allow_split && sp.items < sms && kct > 0) {
        // Fewer items than SMs: split every item along its chunks so that the
        // units fill the SMs, each unit keeping at least four chunks on
        // average.  (Splitting only a partial last wave of a larger problem
        // measured slower: the partial tiles' write, read and second epilogue
        // cost more than the chunks they move.)
        int64_t S = sms / sp.items;
        const int64_t avg = kct / dl.num_slabs;
        if (S > avg / 4) S = avg / 4;
        if (S > 32) S = 32;
        if (S >= 2) {
            sp.split = (int)S;
            sp.full = 0;
        }
    }
#ifdef BP_BALANCE
    if (!it)
    // Balanced launches are built only with BP_BALANCE: on this kernel they
    // measured slower than whole items in waves on the 4096^3 layer at 1/4
    // (46.5 against 41.7 us) and the BERT 3072 x 768 layer (32.6 against 25.4
    // us), faster only on long dense-union items (4096^3, 8 x 64 blocks at
    // 1/2: 136.5 against 147.9 us).
    if (allow_split && sp.items >= sms && dl.kc_total > 0) {
        // Whole items run in waves of `sms`; when the last wave is partial
        // the busiest SMs run ceil(items / sms) items against items / sms on
        // average.  Cut the chunks into equal ranges instead (widest tile:
        // waves no longer matter) when that wins at least 10 % and every CTA
        // keeps at least 8 chunks.
        const int nt = (int)std::max<int64_t>(64, std::min<int64_t>(kNT, (N + 31) / 32 * 32));
        const int64_t items = (N + nt - 1) / nt * dl.num_slabs;
        const int64_t total = (N + nt - 1) / nt * dl.kc_total;
        const double waves = (double)((items + sms - 1) / sms), avg = (double)items / sms;
        if (waves > 1.1 * avg && total / sms >= 8 && total < INT32_MAX) {
            sp.nt = nt;
            sp.items = items;
            // whole items for all but the last full wave; the ranges then cover
            // between one and two waves of items
            sp.full = (items / sms - 1) * sms;
            sp.balanced = true;
            sp.total = total;
            sp.units = sms;
            sp.bytes = (size_t)((int64_t)sms * kSlab * kNT * 4 + (int64_t)sms * 16);
            sp.bytes = (sp.bytes + 255) / 256 * 256;
            return sp;
        }
    }
#endif
    sp.units = sp.full + (sp.items - sp.full) * sp.split;
    if (sp.split > 1) {
        // one fp32 accumulator tile per split item, then its arrival counters
        const int64_t tiles = sp.items - sp.full;
        sp.bytes = (size_t)((tiles * kSlab * kNT * 4 + 255) / 256 * 256 +
                            (tiles * 16 + 255) / 256 * 256);
    }
    return sp;
}

cudaError_t launch_mma(const bp_packed &P, const DevLayout &dl, const void *X, int64_t N,
                       int64_t ldx, const float *bias, int relu, void *Y, int64_t ldy,
                       const ConvShape *conv, void *ws, cudaStream_t st, bool implicit,
                       bool direct) {
    Params p{};
    const uint8_t *dev = static_cast<const uint8_t *>(P.dev);
    p.dtype = P.lay.dtype;
    p.relu = relu;
    p.conv = conv ? 1 : 0;
    p.M = P.lay.M;
    p.num_slabs = dl.num_slabs;
    p.N = N;
    if (implicit && (!conv || dl.c3max == 0)) return cudaErrorInvalidValue;
    const ImplicitTiles itl = implicit ? implicit_tiles(*conv) : ImplicitTiles{};
    if (implicit && !itl.ok) return cudaErrorInvalidValue;
    const SplitPlan sp = plan_split(dl, N, ws != nullptr, implicit ? &itl : nullptr);
    p.nt = sp.nt;
    p.xboxes = (p.nt + 63) / 64;
    p.num_items = sp.items;
    p.full_items = sp.full;
    p.split = sp.split;
    p.num_units = sp.units;
    if (p.num_items == 0) return cudaSuccess;
    if (p.num_units >= INT32_MAX) return cudaErrorInvalidValue;   // 32-bit unit decoding
    if (sp.balanced) {
        // one partial tile per CTA, then the per-(CTA, quadrant) flags (zero
        // on entry: the caller zero-fills a new workspace, and the CTA that
        // reads a flag zeroes it again)
        p.sk = 1;
        p.sk_i0 = sp.full;
        p.sk_total = sp.total;
        p.kc_total = dl.kc_total;
        p.part = static_cast<float *>(ws);
        p.cnt = reinterpret_cast<int32_t *>(static_cast<uint8_t *>(ws) +
                                            (int64_t)sp.units * kSlab * kNT * 4);
    }
    if (sp.split > 1) {
        // accumulator tiles, then the arrival counters (zero on entry: the
        // caller zero-fills a new workspace, and each item's last unit zeroes
        // its tile and counters again)
        const int64_t tiles = sp.items - sp.full;
        p.part = static_cast<float *>(ws);
        p.cnt = reinterpret_cast<int32_t *>(static_cast<uint8_t *>(ws) +
                                            (tiles * kSlab * kNT * 4 + 255) / 256 * 256);
    }
    p.ystage_bytes = 4 * 4096;     // per epilogue warp: two 2 KB boxes (GEMM) or one (conv)
    // shared memory: stages, output staging, barriers, index ring, and a copy of
    // kc_ptr when that costs no pipeline stage
    auto stages_for = [&](int64_t kc) {
        int64_t n = kMaxStages;
        while (n > 0 && (int64_t)smem_bytes(n, p.ystage_bytes, kc) > kMaxSmem) --n;
        return n;
    };
    p.stages = stages_for(0);
    if (p.stages < 2) return cudaErrorInvalidValue;
    // a split or balanced launch's last unit stages four 32 KB quadrants of
    // fp32 sums in the stage area
    if ((sp.split > 1 || sp.balanced) &&
        p.stages * (int64_t)(kWTileBytes + kXTileBytes) < 4 * (int64_t)kSlab / 4 * kNT * 4)
        return cudaErrorInvalidValue;
    const int64_t kc_entries = p.num_slabs + 1;
    p.kc_cached = (kc_entries <= kMaxCachedKc && stages_for(kc_entries) == p.stages) ? kc_entries : 0;
    p.acc_cols = kNT;
    p.tmem_cols = 2 * kNT;
    p.kc_ptr = reinterpret_cast<const int64_t *>(dev);
    p.tiles = dev + dl.off_tiles;
    // a convolution's X holds only the listed rows: use the compacted records
    // a convolution's im2col matrix holds the listed rows only (compacted
    // records); a 1 x 1 layer read in place uses the column indices themselves
    p.meta = dev + (conv && !direct ? dl.off_meta2 : dl.off_meta);
    p.direct = direct ? 1 : 0;
    if (direct) {
        if (!conv || conv->kh != 1 || conv->kw != 1 || ldx != conv->H * conv->W || ldx % 8)
            return cudaErrorInvalidValue;
        p.d_CHW = conv->C * conv->H * conv->W;
    }
    if (implicit) {
        // section 3 of the image: K-group chunks
        p.impl = 1;
        p.kc_ptr = reinterpret_cast<const int64_t *>(dev + dl.off_sec3);
        p.tiles = dev + dl.off_tiles3;
        p.meta = dev + dl.off_meta3;
        p.i_ipt = itl.ipt;
        p.i_rpt = itl.rpt;
        p.i_tpi = itl.tpi;
        p.i_HoWo = conv->Ho * conv->Wo;
        p.i_Wo = conv->Wo;
        p.i_Ho = conv->Ho;
        p.i_Nb = conv->Nb;
        p.i_ph = conv->ph;
        p.i_pw = conv->pw;
        p.i_s = conv->sh;
    }
    p.X = static_cast<const uint16_t *>(X);
    p.ldx = ldx;
    p.Y = static_cast<uint16_t *>(Y);
    p.ldy = ldy;
    p.HoWo = conv ? conv->Ho * conv->Wo : 0;
    p.bias = bias;
    p.watchdog_ns = watchdog_ns();
    p.drop_stage = debug_drop_stage();
    p.status = device_status_ptr();

    PFN_cuTensorMapEncodeTiled_v12000 enc = tensor_map_encoder();
    if (!enc) return cudaErrorNotSupported;
    const CUtensorMapDataType tdt =
        P.lay.dtype == BP_BF16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT16;
    if (implicit) {
        // NHWC input, channels padded to C8: boxes of 64 channels x Wo x hbox x
        // nbox (channels past C8 read as zero), written as K-major 128-byte rows
        // with the 128-byte swizzle
        // (stride 2: the four phases, each ceil(H/2) x ceil(W/2), as 4 Nb images)
        const int64_t C8 = (conv->C + 7) / 8 * 8;
        const int64_t s2 = conv->sh == 2;
        const int64_t Wi = s2 ? (conv->W + 1) / 2 : conv->W, Hi = s2 ? (conv->H + 1) / 2 : conv->H;
        const cuuint64_t gdim[4] = {(cuuint64_t)C8, (cuuint64_t)Wi, (cuuint64_t)Hi,
                                    (cuuint64_t)(s2 ? 4 * conv->Nb : conv->Nb)};
        const cuuint64_t gstride[3] = {(cuuint64_t)(C8 * 2), (cuuint64_t)(Wi * C8 * 2),
                                       (cuuint64_t)(Hi * Wi * C8 * 2)};
        const cuuint32_t hbox = (cuuint32_t)(itl.ipt > 0 ? conv->Ho : itl.rpt);
        const cuuint32_t nbox = (cuuint32_t)(itl.ipt > 0 ? itl.ipt : 1);
        const cuuint32_t box[4] = {64, (cuuint32_t)conv->Wo, hbox, nbox};
        const cuuint32_t estride[4] = {1, 1, 1, 1};
        p.i_box_bytes = 128u * box[1] * hbox * nbox;
        if (p.i_box_bytes > 128u * (uint32_t)p.nt) return cudaErrorInvalidValue;
        if (enc(&p.imap, tdt, 4, const_cast<void *>(X), gdim, gstride, box, estride,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return cudaErrorInvalidValue;
    }
    for (int i = 0; i < 4 && !implicit && !direct; ++i) {
        // X (N inner, K rows): 64-token x (8 << i)-row boxes for runs of consecutive columns
        const cuuint64_t gdim[2] = {(cuuint64_t)N, (cuuint64_t)P.lay.K};
        const cuuint64_t gstride[1] = {(cuuint64_t)ldx * 2};
        const cuuint32_t box[2] = {64, (cuuint32_t)(8 << i)};
        const cuuint32_t estride[2] = {1, 1};
        if (enc(&p.xmap[i], tdt, 2, const_cast<void *>(X), gdim, gstride, box, estride,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return cudaErrorInvalidValue;
    }
    p.yvec = conv && p.HoWo % 8 == 0;
#ifndef BP_EPI_DIRECT
    if (!conv) {
        // Y (N inner, M rows) for the epilogue's 32 x 32 box stores
        const cuuint64_t gdim[2] = {(cuuint64_t)N, (cuuint64_t)P.lay.M};
        const cuuint64_t gstride[1] = {(cuuint64_t)ldy * 2};
        const cuuint32_t box[2] = {32, 32};
        const cuuint32_t estride[2] = {1, 1};
        if (enc(&p.ymap, tdt, 2, Y, gdim, gstride, box, estride, CU_TENSOR_MAP_INTERLEAVE_NONE,
                CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return cudaErrorInvalidValue;
        const cuuint32_t box64[2] = {64, 32};
        if (enc(&p.ymap64, tdt, 2, Y, gdim, gstride, box64, estride, CU_TENSOR_MAP_INTERLEAVE_NONE,
                CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return cudaErrorInvalidValue;
        p.ytma = 1;
    } else if (p.HoWo % 8 == 0) {
        // NCHW output as (Ho*Wo, M, Nb): 32-pixel x 32-channel boxes of one
        // image (the image stride, Ho*Wo*2 bytes, must be a multiple of 16)
        const cuuint64_t gdim[3] = {(cuuint64_t)p.HoWo, (cuuint64_t)P.lay.M,
                                    (cuuint64_t)conv->Nb};
        const cuuint64_t gstride[2] = {(cuuint64_t)p.HoWo * 2, (cuuint64_t)(P.lay.M * p.HoWo * 2)};
        const cuuint32_t box[3] = {32, 32, 1};
        const cuuint32_t estride[3] = {1, 1, 1};
        if (enc(&p.ymap, tdt, 3, Y, gdim, gstride, box, estride, CU_TENSOR_MAP_INTERLEAVE_NONE,
                CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return cudaErrorInvalidValue;
        const cuuint32_t box64[3] = {64, 32, 1};
        if (enc(&p.ymap64, tdt, 3, Y, gdim, gstride, box64, estride, CU_TENSOR_MAP_INTERLEAVE_NONE,
                CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return cudaErrorInvalidValue;
        p.ytma = 1;
    }
#endif
    static std::once_flag once;
    static cudaError_t attr_err = cudaSuccess;
    std::call_once(once, [] {
        const void *fns[4] = {(const void *)bp_mma_kernel<false, false>,
                              (const void *)bp_mma_kernel<true, false>,
                              (const void *)bp_mma_kernel<false, true>,
                              (const void *)bp_mma_kernel<true, true>};
        for (const void *f : fns)
            if (attr_err == cudaSuccess)
                attr_err = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                (int)kMaxSmem);
    });
    if (attr_err != cudaSuccess) return attr_err;
    const int64_t grid = p.num_units < num_sms() ? p.num_units : num_sms();
    // programmatic dependent launch: the kernel's set-up may overlap the tail of
    // the previous kernel in the stream (the kernel waits for it before any
    // global memory access)
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)grid);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem_bytes(p.stages, p.ystage_bytes, p.kc_cached);
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
#ifdef BP_NO_PDL
    cfg.numAttrs = 0;       // (measurement build) an ordinary stream-ordered launch
#else
    cfg.numAttrs = 1;
#endif
    const bool parts = p.split > 1 || p.sk;
    if (conv)
        return parts ? cudaLaunchKernelEx(&cfg, bp_mma_kernel<true, true>, p)
                     : cudaLaunchKernelEx(&cfg, bp_mma_kernel<false, true>, p);
    return parts ? cudaLaunchKernelEx(&cfg, bp_mma_kernel<true, false>, p)
                 : cudaLaunchKernelEx(&cfg, bp_mma_kernel<false, false>, p);
}

}  // namespace bp

#ifdef BP_TRACE
// Copies the trace (kTraceChunks x kTraceEvents clock64 values) to host memory.
extern "C" int bp_debug_trace_read(unsigned long long *host, int n) {
    if (n > bp::kTraceChunks * bp::kTraceEvents) n = bp::kTraceChunks * bp::kTraceEvents;
    return cudaMemcpyFromSymbol(host, bp::g_trace, n * sizeof(unsigned long long)) == cudaSuccess ? n : -1;
}
extern "C" int bp_debug_trace_clear(void) {
    static unsigned long long zero[bp::kTraceChunks * bp::kTraceEvents];
    return cudaMemcpyToSymbol(bp::g_trace, zero, sizeof(zero)) == cudaSuccess ? 0 : -1;
}
#endif
