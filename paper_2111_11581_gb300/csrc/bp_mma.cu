// Block-sparse GEMM / implicit-GEMM convolution on the sm_103a tensor cores.
//
// Each work item is one row-block (or one 128-row slab of it) times one tile
// of activation columns.  The row-block's compact weights Wc (bm x K'_rb,
// Sec. 4.3) multiply the activation rows selected by its kept-column list, so
// pruned weights never enter the product.  Per k-chunk of 64 kept columns a
// pipeline stage holds the chunk's pre-swizzled weight tile and the 64
// activation rows it names, laid out as a 128-byte-swizzled MN-major tile:
//
//   warps 0-3   producers.  Thread 0 copies the weight tile with one TMA
//               bulk copy (completion counted in bytes on the stage's
//               weight barrier).  GEMM: the 128 threads gather the rows of X
//               with 16-byte cp.async (one 512- or 256-byte row segment per
//               warp instruction) and arrive on the stage's data barrier
//               when their copies land, without blocking.  CONV: im2col rows
//               are built in registers (zero outside the image) and stored.
//               (TMA tile::gather4 moves 4 x 128 B per instruction and
//               measured about 6x slower per byte than this path.)
//   warp 4      MMA issuer: tcgen05.mma (K = 16 per instruction) into an
//               fp32 accumulator in tensor memory, double-buffered;
//   warps 5-8   epilogue: tcgen05.ld, + bias, ReLU, round to fp16/bf16, store
//               (weight-as-A tiles: through a swizzled shared-memory staging
//               buffer and TMA tensor stores of 32 x 32 boxes, which keeps the
//               output off the load/store unit the gather needs).
//
// Two operand orientations:
//   kWeightA (bm a multiple of 128): D[128 weight rows x 256 tokens]
//            = Wc tile (A, K-major) * gathered X (B, MN-major);
//   kWeightB (bm <= 256): D[128 tokens x rows_pad] = gathered X^T (A,
//            MN-major) * Wc^T (B, K-major), rows_pad = bm rounded up to 16.
//
// Every wait is bounded (see mbar_wait); on expiry the kernel records
// kDevTimeout in the device status word, drains its own copies and tensor
// core work, frees tensor memory and returns.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cudaTypedefs.h>

#include <mutex>

#include "bp_common.cuh"

namespace bp {
namespace {

constexpr uint64_t kDrainNs = 1000000000ull;
constexpr int kMaxStages = 8;
constexpr int kIdxSlots = 8;           // index lists copied to shared memory this many chunks ahead
constexpr int kMaxCachedRb = 2047;     // kc_ptr kept in shared memory up to this many row-blocks
constexpr int64_t kMaxSmem = 232448;   // dynamic shared memory per CTA (227 KB)

struct alignas(64) Params {
    CUtensorMap ymap;       // weight-as-A GEMM: Y as a 2-D tensor, box 32 x 32, 64-byte swizzle
    int dtype;
    int relu;
    int64_t M, bm, rows_pad, num_rb, nslab;
    int64_t N;              // tokens (GEMM) or Nb*Ho*Wo pixels (conv)
    int64_t num_items;
    int64_t stages;
    uint32_t w_tile_bytes, x_tile_bytes, tmem_cols, acc_cols, ystage_bytes;
    const int64_t *kc_ptr;
    int64_t kc_cached;      // entries of kc_ptr copied to shared memory (0 = none)
    const uint8_t *chunks;  // k-chunks: weight tile, then 64 int32 column indices
    int64_t tile_bytes, chunk_bytes;
    const uint16_t *X;
    int64_t ldx;
    uint16_t *Y;
    int64_t ldy;
    const float *bias;
    // convolution
    int64_t C, H, W, Ho, Wo, HoWo, KK;
    int kw, ph, pw, sh, sw;
    uint64_t watchdog_ns;
    int64_t drop_stage;     // fault injection: CTA 0 never fills this stage (-1 = off)
    unsigned *status;
};

// Warp roles.  GEMM: 8 gather warps, 1 control warp (index lists + weight
// tiles through TMA), 1 MMA warp, 4 epilogue warps.  CONV: 4 im2col warps
// (thread 0 also copies weight tiles), 1 MMA warp, 4 epilogue warps.
template <bool CONV>
struct Roles {
    static constexpr int kGatherWarps = CONV ? 4 : 8;
    static constexpr int kCtrlWarp = CONV ? -1 : 8;
    static constexpr int kMmaWarp = CONV ? 4 : 9;
    static constexpr int kEpiWarp0 = kMmaWarp + 1;
    static constexpr int kThreads = (kEpiWarp0 + 4) * 32;
    static constexpr uint32_t kGatherThreads = kGatherWarps * 32;
};

__device__ __forceinline__ uint32_t pack2(float a, float b, int dtype) {
    if (dtype == BP_BF16) {
        const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
        return *reinterpret_cast<const uint32_t *>(&h);
    }
    const __half2 h = __floats2half2_rn(a, b);
    return *reinterpret_cast<const uint32_t *>(&h);
}

__device__ __forceinline__ uint16_t cvt1(float a, int dtype) {
    if (dtype == BP_BF16) return __bfloat16_as_ushort(__float2bfloat16_rn(a));
    return __half_as_ushort(__float2half_rn(a));
}

struct Smem {
    uint8_t *w;          // stages x w_tile_bytes
    uint8_t *x;          // stages x x_tile_bytes
    uint8_t *ystage;     // weight-as-A: 4 epilogue warps x 2 buffers x 2 KB
    uint64_t *full;      // [stages] activation tile landed (128 producer arrivals)
    uint64_t *wfull;     // [stages] weight tile landed (TMA byte count)
    uint64_t *empty;     // [stages] tensor cores done with the stage
    uint64_t *tfull;     // [2]
    uint64_t *tempty;    // [2]
    uint64_t *drain;     // [1]
    uint64_t *ifull;     // [kIdxSlots] index list of a chunk landed (TMA byte count)
    uint64_t *iempty;    // [kIdxSlots] all producer threads have read the slot
    int32_t *idx;        // [kIdxSlots][64] index lists of upcoming chunks
    uint32_t *tmem_base;
    int *abort_flag;
    int64_t *kc;         // [kc_cached] copy of kc_ptr, or nullptr
};

__device__ __forceinline__ Smem carve(uint8_t *raw, const Params &p) {
    Smem s;
    uint8_t *base = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(raw) + 1023) & ~static_cast<uintptr_t>(1023));
    s.w = base;
    s.x = base + p.stages * p.w_tile_bytes;
    s.ystage = s.x + p.stages * p.x_tile_bytes;
    uint8_t *b = s.ystage + p.ystage_bytes;
    s.full = reinterpret_cast<uint64_t *>(b);
    s.wfull = s.full + p.stages;
    s.empty = s.wfull + p.stages;
    s.tfull = s.empty + p.stages;
    s.tempty = s.tfull + 2;
    s.drain = s.tempty + 2;
    s.ifull = s.drain + 1;
    s.iempty = s.ifull + kIdxSlots;
    s.tmem_base = reinterpret_cast<uint32_t *>(s.iempty + kIdxSlots);
    s.abort_flag = reinterpret_cast<int *>(s.tmem_base + 1);
    // TMA bulk copies need a 16-byte-aligned destination: round up to 128 bytes
    const uintptr_t after = reinterpret_cast<uintptr_t>(s.iempty + kIdxSlots + 2);
    s.idx = reinterpret_cast<int32_t *>((after + 127) & ~static_cast<uintptr_t>(127));
    s.kc = p.kc_cached ? reinterpret_cast<int64_t *>(s.idx + kIdxSlots * kBK) : nullptr;
    return s;
}

__device__ __forceinline__ void raise_timeout(const Params &p, const Smem &s) {
    *reinterpret_cast<volatile int *>(s.abort_flag) = 1;
    atomicOr(p.status, kDevTimeout);
}

struct Item {
    int64_t rb, slab, n0, kc0, nkc, rows;   // rows = real rows of the row-block
};

__device__ __forceinline__ Item decode(const Params &p, const int64_t *kc, int64_t it, bool wa) {
    Item t;
    const int64_t R = p.num_rb * p.nslab;
    const int64_t rs = it % R;
    t.n0 = (it / R) * (wa ? 256 : 128);
    t.rb = rs / p.nslab;
    t.slab = rs % p.nslab;
    t.kc0 = kc[t.rb];
    t.nkc = kc[t.rb + 1] - t.kc0;
    t.rows = min(p.bm, p.M - t.rb * p.bm);
    return t;
}

// Walks this CTA's (work item, k-chunk) sequence, skipping empty row-blocks.
struct Cursor {
    int64_t it;
    int64_t kc;
    Item t;
    __device__ __forceinline__ void first(const Params &p, const int64_t *kcp, bool wa) {
        kc = 0;
        for (it = blockIdx.x; it < p.num_items; it += gridDim.x) {
            t = decode(p, kcp, it, wa);
            if (t.nkc > 0) return;
        }
    }
    __device__ __forceinline__ void next(const Params &p, const int64_t *kcp, bool wa) {
        if (++kc < t.nkc) return;
        kc = 0;
        for (it += gridDim.x; it < p.num_items; it += gridDim.x) {
            t = decode(p, kcp, it, wa);
            if (t.nkc > 0) return;
        }
    }
    __device__ __forceinline__ bool valid(const Params &p) const { return it < p.num_items; }
};

// ------------------------------------------------------------------ producers
// Weight tile of a stage: thread 0 of the producers, TMA bulk copy.
struct WeightCopier {
    uint32_t last_phase[kMaxStages];
    bool issued[kMaxStages];
    __device__ __forceinline__ void init() {
        for (int i = 0; i < kMaxStages; ++i) issued[i] = false;
    }
    __device__ __forceinline__ void copy(const Params &p, const Smem &s, int stage, uint32_t phase,
                                         const uint8_t *src) {
        mbar_arrive_expect_tx(&s.wfull[stage], p.w_tile_bytes);
        bulk_g2s(smem_u32(s.w + stage * p.w_tile_bytes), src, p.w_tile_bytes, &s.wfull[stage]);
        issued[stage] = true;
        last_phase[stage] = phase;
    }
    // the CTA is unwinding: let every weight copy already issued land first
    __device__ __forceinline__ void drain(const Params &p, const Smem &s) {
        for (int i = 0; i < p.stages; ++i)
            if (issued[i] && !mbar_wait(&s.wfull[i], last_phase[i], kDrainNs, nullptr))
                atomicOr(p.status, kDevTimeout);
    }
};

// Index lists of upcoming chunks, copied by TMA (256 B each) into a ring of
// kIdxSlots shared-memory slots up to kIdxSlots chunks ahead of their use, so
// the producers never wait on a global load for them.  Every producer thread
// arrives on the slot's iempty barrier once it has read the list; thread 0
// refills a slot only after that (bounded wait), one chunk later.
struct IndexRing {
    Cursor look;         // next chunk whose list is to be fetched (thread 0)
    int64_t fetched;     // lists fetched so far
    uint32_t last_phase[kIdxSlots];
    bool pending[kIdxSlots];
    __device__ __forceinline__ void fetch_one(const Params &p, const Smem &s, const int64_t *kcp,
                                              bool wa) {
        const int slot = (int)(fetched % kIdxSlots);
        const uint32_t ph = (uint32_t)((fetched / kIdxSlots) & 1);
        mbar_arrive_expect_tx(&s.ifull[slot], kBK * 4);
        bulk_g2s(smem_u32(s.idx + slot * kBK),
                 p.chunks + (look.t.kc0 + look.kc) * p.chunk_bytes + p.tile_bytes, kBK * 4,
                 &s.ifull[slot]);
        pending[slot] = true;
        last_phase[slot] = ph;
        ++fetched;
        look.next(p, kcp, wa);
    }
    // thread 0: start the first kIdxSlots fetches
    __device__ __forceinline__ void start(const Params &p, const Smem &s, const int64_t *kcp,
                                          bool wa, const Cursor &first) {
        look = first;
        fetched = 0;
        for (int i = 0; i < kIdxSlots; ++i) pending[i] = false;
        for (int i = 0; i < kIdxSlots && look.valid(p); ++i) fetch_one(p, s, kcp, wa);
    }
    // thread 0, after the list of chunk `used` was read by everyone: refill its slot
    __device__ __forceinline__ bool refill(const Params &p, const Smem &s, const int64_t *kcp,
                                           bool wa, int64_t used, volatile int *abort_flag) {
        const int slot = (int)(used % kIdxSlots);
        pending[slot] = false;
        if (!look.valid(p)) return true;
        if (!mbar_wait(&s.iempty[slot], (uint32_t)((used / kIdxSlots) & 1), p.watchdog_ns,
                       abort_flag))
            return false;
        // the readers' loads completed before their (release) arrivals, which the
        // wait above acquired, so the TMA overwrite cannot overtake them
        fetch_one(p, s, kcp, wa);
        return true;
    }
    // the CTA is unwinding: let every list copy in flight land first
    __device__ __forceinline__ void drain(const Params &p, const Smem &s) {
        for (int i = 0; i < kIdxSlots; ++i)
            if (pending[i] && !mbar_wait(&s.ifull[i], last_phase[i], kDrainNs, nullptr))
                atomicOr(p.status, kDevTimeout);
    }
};

// Gather warps (GEMM): per chunk, read the chunk's index list from the shared
// ring, then copy the 64 activation rows it names into the stage with 16-byte
// cp.async straight into the swizzled layout; arrive on the stage's data
// barrier when the copies land (no blocking).
template <bool WA>
__device__ void gather_warps(const Params &p, const Smem &s) {
    constexpr int GW = Roles<false>::kGatherWarps;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t *kcp = s.kc ? s.kc : p.kc_ptr;
    volatile int *abort_flag = s.abort_flag;
    Cursor cur;
    cur.first(p, kcp, WA);
    int stage = 0;
    uint32_t phase = 0;
    int64_t count = 0;
    while (cur.valid(p)) {
        const Item t = cur.t;
        cur.next(p, kcp, WA);
        const int slot = (int)(count % kIdxSlots);
        if (!mbar_wait(&s.ifull[slot], (uint32_t)((count / kIdxSlots) & 1), p.watchdog_ns,
                       abort_flag)) {
            raise_timeout(p, s);
            break;
        }
        // two entries of the list per lane, broadcast below by shuffles
        const int2 iv = make_int2(s.idx[slot * kBK + lane], s.idx[slot * kBK + 32 + lane]);
        mbar_arrive(&s.iempty[slot]);
        const int64_t seq = count++;
        const bool drop = blockIdx.x == 0 && seq == p.drop_stage;
        if (!mbar_wait(&s.empty[stage], phase ^ 1u, p.watchdog_ns, abort_flag)) {
            raise_timeout(p, s);
            break;
        }
        if (!drop) {
            const uint32_t xs = smem_u32(s.x + stage * p.x_tile_bytes);
            if (WA) {
                // 64 rows x 256 tokens: one warp instruction per 512-byte row segment
                const int cn = lane >> 3, j = lane & 7;
                const int64_t n = t.n0 + lane * 8;
                const uint32_t nb = n < p.N ? (uint32_t)min((int64_t)16, (p.N - n) * 2) : 0u;
                const uint16_t *xcol = p.X + (nb ? n : 0);
#pragma unroll
                for (int i = 0; i < 64 / GW; ++i) {
                    const int r = warp + GW * i;
                    const int idx = __shfl_sync(0xffffffffu, r < 32 ? iv.x : iv.y, r & 31);
                    cp_async_16(xs + cn * 8192 + r * 128 + ((j ^ (r & 7)) << 4),
                                xcol + (int64_t)idx * p.ldx, nb);
                }
            } else {
                // 64 rows x 128 tokens: one warp instruction covers two rows
                const int u16 = lane & 15, cn = u16 >> 3, j = u16 & 7;
                const int64_t n = t.n0 + u16 * 8;
                const uint32_t nb = n < p.N ? (uint32_t)min((int64_t)16, (p.N - n) * 2) : 0u;
                const uint16_t *xcol = p.X + (nb ? n : 0);
#pragma unroll
                for (int i = 0; i < 32 / GW; ++i) {
                    const int r = 2 * (warp + GW * i) + (lane >> 4);
                    const int idx = __shfl_sync(0xffffffffu, r < 32 ? iv.x : iv.y, r & 31);
                    cp_async_16(xs + cn * 8192 + r * 128 + ((j ^ (r & 7)) << 4),
                                xcol + (int64_t)idx * p.ldx, nb);
                }
            }
            // Signal the stage once this thread's copies have landed, without
            // blocking.  The tile was written through the generic proxy; the
            // tensor-core thread orders it before its async-proxy reads with a
            // proxy fence after acquiring the barrier.
            cp_async_arrive_noinc(&s.full[stage]);
        }
        if (++stage == p.stages) {
            stage = 0;
            phase ^= 1u;
        }
    }
    cp_async_wait_all();
}

// Control thread (GEMM, lane 0 of the control warp): keeps the index-list ring
// kIdxSlots chunks ahead and copies each stage's weight tile (TMA bulk) as
// soon as the stage is free.
template <bool WA>
__device__ void control_thread(const Params &p, const Smem &s) {
    const int64_t *kcp = s.kc ? s.kc : p.kc_ptr;
    volatile int *abort_flag = s.abort_flag;
    WeightCopier wc;
    wc.init();
    Cursor cur;
    cur.first(p, kcp, WA);
    IndexRing ring;
    ring.start(p, s, kcp, WA, cur);
    int stage = 0;
    uint32_t phase = 0;
    bool ok = true;
    int64_t count = 0;
    while (cur.valid(p)) {
        const Item t = cur.t;
        const int64_t kc = cur.kc;
        cur.next(p, kcp, WA);
        const int64_t seq = count++;
        if (!mbar_wait(&s.empty[stage], phase ^ 1u, p.watchdog_ns, abort_flag)) {
            raise_timeout(p, s);
            ok = false;
            break;
        }
        if (!(blockIdx.x == 0 && seq == p.drop_stage))
            wc.copy(p, s, stage, phase,
                    p.chunks + (t.kc0 + kc) * p.chunk_bytes + t.slab * (kSlab * kBK * 2));
        if (seq > 0 && !ring.refill(p, s, kcp, WA, seq - 1, abort_flag)) {
            raise_timeout(p, s);
            ok = false;
            break;
        }
        if (++stage == p.stages) {
            stage = 0;
            phase ^= 1u;
        }
    }
    if (!ok) {
        wc.drain(p, s);
        ring.drain(p, s);
    }
}

// ------------------------------------------------------------------ CONV producer (im2col)
__device__ void producer_im2col(const Params &p, const Smem &s) {
    const int64_t *kcp = s.kc ? s.kc : p.kc_ptr;
    const int tid = threadIdx.x;            // 0..127
    const int warp = tid >> 5, lane = tid & 31;
    volatile int *abort_flag = s.abort_flag;
    int stage = 0;
    uint32_t phase = 0;
    bool ok = true;
    const int u16 = lane & 15;           // 16-byte unit (8 pixels) within a 128-pixel row
    const int cn = u16 >> 3, j = u16 & 7;
    int64_t count = 0;
    WeightCopier wc;
    wc.init();

    for (int64_t it = blockIdx.x; it < p.num_items && ok; it += gridDim.x) {
        const Item t = decode(p, kcp, it, false);
        if (t.nkc == 0) continue;
        // this thread's 8 pixels are fixed for the whole tile
        int64_t pbase[8];
        int ih0[8], iw0[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const int64_t pix = t.n0 + u16 * 8 + e;
            if (pix < p.N) {
                const int64_t b = pix / p.HoWo, hw = pix % p.HoWo;
                const int oh = (int)(hw / p.Wo), ow = (int)(hw % p.Wo);
                pbase[e] = b * p.C * p.H * p.W;
                ih0[e] = oh * p.sh - p.ph;
                iw0[e] = ow * p.sw - p.pw;
            } else {
                pbase[e] = 0;
                ih0[e] = -(1 << 29);     // never inside the image
                iw0[e] = 0;
            }
        }
        for (int64_t kc = 0; kc < t.nkc; ++kc) {
            if (!mbar_wait(&s.empty[stage], phase ^ 1u, p.watchdog_ns, abort_flag)) {
                raise_timeout(p, s);
                ok = false;
                break;
            }
            const int64_t seq = count++;
            if (blockIdx.x == 0 && seq == p.drop_stage) {       // injected lost stage
                if (++stage == p.stages) {
                    stage = 0;
                    phase ^= 1u;
                }
                continue;
            }
            const uint32_t xs = smem_u32(s.x + stage * p.x_tile_bytes);
            const uint8_t *chunk = p.chunks + (t.kc0 + kc) * p.chunk_bytes;
            if (tid == 0) wc.copy(p, s, stage, phase, chunk);
            const int32_t *cl = reinterpret_cast<const int32_t *>(chunk + p.tile_bytes);
#pragma unroll 2
            for (int i = 0; i < 8; ++i) {
                const int r = 2 * (warp + 4 * i) + (lane >> 4);
                const int32_t idx = cl[r];
                uint32_t v[4] = {0u, 0u, 0u, 0u};
                const int64_t c = idx / p.KK;
                const int rs = (int)(idx - c * p.KK);
                const int di = rs / p.kw, dj = rs - (rs / p.kw) * p.kw;
                const uint16_t *plane = p.X + c * p.H * p.W;
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    const int ih = ih0[e] + di, iw = iw0[e] + dj;
                    uint32_t h = 0u;
                    if ((unsigned)ih < (unsigned)p.H && (unsigned)iw < (unsigned)p.W)
                        h = __ldg(plane + pbase[e] + (int64_t)ih * p.W + iw);
                    v[e >> 1] |= h << ((e & 1) * 16);
                }
                st_shared_v4(xs + cn * 8192 + r * 128 + ((j ^ (r & 7)) << 4),
                             make_uint4(v[0], v[1], v[2], v[3]));
            }
            fence_proxy_async_smem();
            mbar_arrive(&s.full[stage]);
            if (++stage == p.stages) {
                stage = 0;
                phase ^= 1u;
            }
        }
    }
    if (!ok && tid == 0) wc.drain(p, s);
}

// ------------------------------------------------------------------ MMA issuer
template <bool WA>
__device__ void mma_issuer(const Params &p, const Smem &s, uint32_t tmem) {
    const int64_t *kcp = s.kc ? s.kc : p.kc_ptr;
    volatile int *abort_flag = s.abort_flag;
    const bool bf16 = p.dtype == BP_BF16;
    const uint32_t idesc = WA ? make_idesc(bf16, false, true, 128, 256)
                              : make_idesc(bf16, true, false, 128, (int)p.rows_pad);
    int stage = 0;
    uint32_t phase = 0;
    int acc = 0;
    uint32_t acc_phase = 0;
    bool ok = true;
    for (int64_t it = blockIdx.x; it < p.num_items && ok; it += gridDim.x) {
        const Item t = decode(p, kcp, it, WA);
        if (t.nkc == 0) continue;
        if (!mbar_wait(&s.tempty[acc], acc_phase ^ 1u, p.watchdog_ns, abort_flag)) {
            raise_timeout(p, s);
            break;
        }
        tc_fence_after();
        const uint32_t d = tmem + acc * p.acc_cols;
        for (int64_t kc = 0; kc < t.nkc; ++kc) {
            if (!mbar_wait(&s.full[stage], phase, p.watchdog_ns, abort_flag) ||
                !mbar_wait(&s.wfull[stage], phase, p.watchdog_ns, abort_flag)) {
                raise_timeout(p, s);
                ok = false;
                break;
            }
            // the activation tile was written through the generic proxy (cp.async /
            // st.shared): order those writes, acquired through the barrier, before
            // the tensor core's async-proxy reads
            fence_proxy_async_smem();
            tc_fence_after();
            const uint32_t ws = smem_u32(s.w + stage * p.w_tile_bytes);
            const uint32_t xs = smem_u32(s.x + stage * p.x_tile_bytes);
#pragma unroll
            for (int kk = 0; kk < kBK / 16; ++kk) {
                const uint64_t wdesc = make_sdesc_sw128(ws + kk * 32, 16, 1024);
                const uint64_t xdesc = make_sdesc_sw128(xs + kk * 2048, 8192, 1024);
                const uint32_t accum = (kc > 0 || kk > 0) ? 1u : 0u;
                if (WA) umma_f16_ss(d, wdesc, xdesc, idesc, accum);
                else umma_f16_ss(d, xdesc, wdesc, idesc, accum);
            }
            umma_commit(&s.empty[stage]);
            if (++stage == p.stages) {
                stage = 0;
                phase ^= 1u;
            }
        }
        if (!ok) break;
        umma_commit(&s.tfull[acc]);
        if (++acc == 2) {
            acc = 0;
            acc_phase ^= 1u;
        }
    }
    // all issued tensor-core work must finish before tensor memory is freed
    umma_commit(s.drain);
    if (!mbar_wait(s.drain, 0, kDrainNs, nullptr)) atomicOr(p.status, kDevTimeout);
}

// ------------------------------------------------------------------ epilogue
template <bool WA, bool CONV>
__device__ void epilogue(const Params &p, const Smem &s, uint32_t tmem) {
    const int64_t *kcp = s.kc ? s.kc : p.kc_ptr;
    volatile int *abort_flag = s.abort_flag;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int q = warp & 3;                  // tensor-memory lane quadrant of this warp
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int64_t it = blockIdx.x; it < p.num_items; it += gridDim.x) {
        const Item t = decode(p, kcp, it, WA);
        const bool has = t.nkc > 0;
        if (has) {
            if (!mbar_wait(&s.tfull[acc], acc_phase, p.watchdog_ns, abort_flag)) {
                raise_timeout(p, s);
                break;
            }
            tc_fence_after();
        }
        const uint32_t tacc = tmem + ((uint32_t)(32 * q) << 16) + acc * p.acc_cols;
        if (WA) {
            // lane = output row; 32 x 32 boxes staged in shared memory (64-byte swizzle:
            // 16-byte chunk c of row r sits at chunk c ^ ((r >> 1) & 3)), then TMA-stored
            const int64_t row0 = t.slab * kSlab + 32 * q;
            const bool vrow = row0 + lane < t.rows;
            const float bv = (p.bias && vrow) ? p.bias[t.rb * p.bm + row0 + lane] : 0.f;
            const uint32_t stg = smem_u32(s.ystage + (warp - Roles<CONV>::kEpiWarp0) * 4096);
            for (int c0 = 0; c0 < 256 && t.n0 + c0 < p.N; c0 += 32) {
                uint32_t r[32];
                if (has) {
                    tmem_ld_32x32b_x32(tacc + c0, r);
                    tmem_ld_wait();
                } else {
#pragma unroll
                    for (int e = 0; e < 32; ++e) r[e] = 0u;
                }
                uint32_t pk[16];
#pragma unroll
                for (int e = 0; e < 16; ++e) {
                    float a = __uint_as_float(r[2 * e]) + bv, b = __uint_as_float(r[2 * e + 1]) + bv;
                    if (p.relu) {
                        a = fmaxf(a, 0.f);
                        b = fmaxf(b, 0.f);
                    }
                    pk[e] = pack2(a, b, p.dtype);
                }
                const uint32_t sb = stg + ((c0 >> 5) & 1) * 2048;
                if (lane == 0) bulk_wait_read<1>();     // the store that used this buffer is done
                __syncwarp();
#pragma unroll
                for (int ch = 0; ch < 4; ++ch)
                    st_shared_v4(sb + lane * 64 + ((ch ^ ((lane >> 1) & 3)) << 4),
                                 make_uint4(pk[4 * ch], pk[4 * ch + 1], pk[4 * ch + 2], pk[4 * ch + 3]));
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) {
                    tma_store_2d(&p.ymap, sb, (int32_t)(t.n0 + c0), (int32_t)(t.rb * p.bm + row0));
                    bulk_commit();
                }
            }
        } else {
            const int64_t n = t.n0 + 32 * q + lane;
            const bool vcol = n < p.N;
            int64_t obase = 0;                 // output offset of this token / pixel
            int64_t ostride = p.ldy;           // between consecutive output rows
            if (CONV) {
                const int64_t b = vcol ? n / p.HoWo : 0, hw = vcol ? n % p.HoWo : 0;
                obase = b * p.M * p.HoWo + hw;
                ostride = p.HoWo;
            } else {
                obase = n;
            }
            for (int c0 = 0; c0 < p.rows_pad; c0 += 16) {
                uint32_t r[16];
                if (has) {
                    tmem_ld_32x32b_x16(tacc + c0, r);
                    tmem_ld_wait();
                } else {
#pragma unroll
                    for (int e = 0; e < 16; ++e) r[e] = 0u;
                }
                if (!vcol) continue;
#pragma unroll
                for (int e = 0; e < 16; ++e) {
                    const int64_t row = c0 + e;
                    if (row < t.rows) {
                        const int64_t m = t.rb * p.bm + row;
                        float v = __uint_as_float(r[e]) + (p.bias ? p.bias[m] : 0.f);
                        if (p.relu && v < 0.f) v = 0.f;
                        p.Y[obase + m * ostride] = cvt1(v, p.dtype);
                    }
                }
            }
        }
        if (has) {
            tc_fence_before();
            mbar_arrive(&s.tempty[acc]);
            if (++acc == 2) {
                acc = 0;
                acc_phase ^= 1u;
            }
        }
    }
    if (WA && lane == 0) bulk_wait_all();       // staged output fully written before exit
}

template <bool WA, bool CONV>
__global__ void __launch_bounds__(Roles<CONV>::kThreads, 1)
    bp_mma_kernel(const __grid_constant__ Params p) {
    using R = Roles<CONV>;
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    const Smem s = carve(smem_raw, p);
    const int warp = threadIdx.x >> 5;
    if (threadIdx.x == 0) {
        for (int i = 0; i < p.stages; ++i) {
            mbar_init(&s.full[i], R::kGatherThreads);
            mbar_init(&s.wfull[i], 1);
            mbar_init(&s.empty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&s.tfull[i], 1);
            mbar_init(&s.tempty[i], 128);
        }
        mbar_init(s.drain, 1);
        for (int i = 0; i < kIdxSlots; ++i) {
            mbar_init(&s.ifull[i], 1);
            mbar_init(&s.iempty[i], R::kGatherThreads);
        }
        *s.abort_flag = 0;
        fence_mbar_init();
    }
    if (s.kc)
        for (int64_t i = threadIdx.x; i < p.kc_cached; i += R::kThreads) s.kc[i] = p.kc_ptr[i];
    if (warp == R::kMmaWarp) {
        tmem_alloc(s.tmem_base, p.tmem_cols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *s.tmem_base;

    if (warp < R::kGatherWarps) {
        if (CONV) producer_im2col(p, s);
        else gather_warps<WA>(p, s);
    } else if (warp == R::kCtrlWarp) {
        if ((threadIdx.x & 31) == 0) control_thread<WA>(p, s);
        __syncwarp();
    } else if (warp == R::kMmaWarp) {
        if ((threadIdx.x & 31) == 0) mma_issuer<WA>(p, s, tmem);
        __syncwarp();
    } else {
        epilogue<WA, CONV>(p, s, tmem);
    }

    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == R::kMmaWarp) tmem_dealloc(tmem, p.tmem_cols);
}

uint32_t pow2_at_least(uint32_t v) {
    uint32_t r = 32;
    while (r < v) r <<= 1;
    return r;
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
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

template <bool WA, bool CONV>
cudaError_t launch_variant(Params &p, cudaStream_t st) {
    static std::once_flag once;
    static cudaError_t attr_err = cudaSuccess;
    std::call_once(once, [] {
        attr_err = cudaFuncSetAttribute(bp_mma_kernel<WA, CONV>,
                                        cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kMaxSmem);
    });
    if (attr_err != cudaSuccess) return attr_err;
    const size_t smem = 1024 + (size_t)p.stages * (p.w_tile_bytes + p.x_tile_bytes) +
                        p.ystage_bytes + (3 * (size_t)p.stages + 7 + 2 * kIdxSlots) * 8 +
                        128 + (size_t)kIdxSlots * kBK * 4 + 8 * (size_t)p.kc_cached;
    const int64_t grid = p.num_items < num_sms() ? p.num_items : num_sms();
    bp_mma_kernel<WA, CONV><<<(unsigned)grid, Roles<CONV>::kThreads, smem, st>>>(p);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_mma(const bp_packed &P, const DevLayout &dl, const void *X, int64_t N,
                       int64_t ldx, const float *bias, int relu, void *Y, int64_t ldy,
                       const ConvShape *conv, cudaStream_t st) {
    Params p{};
    // GEMMs put 128-row weight slabs on the MMA M side when bm allows it;
    // convolutions (and bm not a multiple of 128) put 128 pixels / tokens there.
    // Both read the same device image when rows_pad <= 256.
    const bool wa = conv == nullptr && dl.orient == kWeightA;
    if (!wa && dl.rows_pad > 256) return cudaErrorInvalidValue;
    const uint8_t *dev = static_cast<const uint8_t *>(P.dev);
    p.dtype = P.lay.dtype;
    p.relu = relu;
    p.M = P.lay.M;
    p.bm = P.lay.bm;
    p.rows_pad = dl.rows_pad;
    p.num_rb = P.num_rb;
    p.nslab = wa ? dl.rows_pad / kSlab : 1;
    p.N = N;
    const int64_t nt = wa ? 256 : 128;
    p.num_items = (N + nt - 1) / nt * p.num_rb * p.nslab;
    p.w_tile_bytes = (uint32_t)((wa ? kSlab : dl.rows_pad) * kBK * 2);
    p.x_tile_bytes = (uint32_t)(nt * kBK * 2);
    p.ystage_bytes = wa ? 4 * 2 * 2048 : 0;
    p.kc_cached = p.num_rb + 1 <= kMaxCachedRb + 1 ? p.num_rb + 1 : 0;
    // shared memory: stages + output staging + barriers + kc_ptr copy, within 227 KB
    auto stages_for = [&](int64_t kc) {
        const int64_t avail =
            kMaxSmem - 1024 - p.ystage_bytes - 8 * 48 - 128 - kIdxSlots * kBK * 4 - 8 * kc;
        const int64_t st = avail / (p.w_tile_bytes + p.x_tile_bytes);
        return st > kMaxStages ? (int64_t)kMaxStages : st;
    };
    if (stages_for(p.kc_cached) < 3) p.kc_cached = 0;
    p.stages = stages_for(p.kc_cached);
    if (p.stages < 2) return cudaErrorInvalidValue;
    p.acc_cols = pow2_at_least(wa ? 256u : (uint32_t)dl.rows_pad);
    p.tmem_cols = 2 * p.acc_cols;
    p.kc_ptr = reinterpret_cast<const int64_t *>(dev);
    p.chunks = dev + dl.off_chunks;
    p.tile_bytes = dl.tile_bytes;
    p.chunk_bytes = dl.chunk_bytes;
    p.X = static_cast<const uint16_t *>(X);
    p.ldx = ldx;
    p.Y = static_cast<uint16_t *>(Y);
    p.ldy = ldy;
    p.bias = bias;
    p.watchdog_ns = watchdog_ns();
    p.drop_stage = debug_drop_stage();
    p.status = device_status_ptr();
    if (p.num_items == 0) return cudaSuccess;
    if (conv) {
        p.C = conv->C;
        p.H = conv->H;
        p.W = conv->W;
        p.Ho = conv->Ho;
        p.Wo = conv->Wo;
        p.HoWo = conv->Ho * conv->Wo;
        p.KK = (int64_t)conv->kh * conv->kw;
        p.kw = conv->kw;
        p.ph = conv->ph;
        p.pw = conv->pw;
        p.sh = conv->sh;
        p.sw = conv->sw;
        return launch_variant<false, true>(p, st);
    }
    if (!wa) return launch_variant<false, false>(p, st);
    // Y as a 2-D tensor (N inner, M rows) for the epilogue's 32 x 32 box stores
    PFN_cuTensorMapEncodeTiled_v12000 enc = encode_fn();
    if (!enc) return cudaErrorNotSupported;
    const cuuint64_t gdim[2] = {(cuuint64_t)N, (cuuint64_t)P.lay.M};
    const cuuint64_t gstride[1] = {(cuuint64_t)ldy * 2};
    const cuuint32_t box[2] = {32, 32};
    const cuuint32_t estride[2] = {1, 1};
    if (enc(&p.ymap,
            P.lay.dtype == BP_BF16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT16,
            2, Y, gdim, gstride, box, estride, CU_TENSOR_MAP_INTERLEAVE_NONE,
            CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
        return cudaErrorInvalidValue;
    return launch_variant<true, false>(p, st);
}

}  // namespace bp
