// Reweighted group-Lasso regulariser of one layer and its gradient (Sec. 4.2,
// the block problem with the column groups of block-based pruning and the
// kernel-position groups of block-punched pruning; the factors follow the
// reweighted l1 rule of Candes et al.):
//   s_u = ||W_u||_F^2,  alpha_u = 1 / (s_u + eps),
//   R = lambda * sum_u alpha_u^2 s_u,  grad = 2 lambda alpha_u^2 W.
//
// One launch reads W once from HBM and writes alpha and grad once.  The unit
// norms are summed in fp32 (squares of 16-bit values are exact in fp32) and
// the per-unit factors are formed in fp32 -- the precision of the paper's
// training -- since GB300's fp64 pipe is too narrow to keep up with HBM; only
// R is accumulated in fp64.  R is a fixed-order sum: every block reduces its
// units' terms in a fixed tree and stores the partial in the workspace; the
// last block to finish adds the partials in block order.
//
// Units are numbered as in bp_prune: u = rb*K + column for block-based layers,
// u = (rb*CB + cb)*KK + position for block-punched ones.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <map>
#include <mutex>

#include "bp_common.cuh"

namespace bp {
namespace {

constexpr int kThreads = 256;
constexpr int kMaxBlocks = 2048;
constexpr int kTileFloats = 2048;   // row slices x tile columns

struct Geo {
    int M, K, KK, C, bm, bk, RB, CB, U;
    int S;      // row slices of a tile (power of two)
    int G;      // column groups of 8 per tile (kThreads / S)
    int TC;     // tiles across K
    int tiles;  // RB * TC
};

template <bool kBF16>
__device__ __forceinline__ float to_f32(uint32_t b) {
    if constexpr (kBF16) return __uint_as_float(b << 16);
    else return __half2float(__ushort_as_half((unsigned short)b));
}

// The per-unit factors in fp32: alpha (stored as fp64), the unit's term
// alpha^2 s of R (added to the thread's fp64 sum) and the gradient factor
// 2 lambda alpha^2.
__device__ __forceinline__ float finish_unit(float s, float eps, float lambda2,
                                             double *alpha_out, double &rsum) {
    const float a = 1.0f / (s + eps);
    *alpha_out = (double)a;
    rsum += (double)((a * a) * s);
    return (lambda2 * a) * a;
}

// Fixed-tree block reduction of each thread's R terms; the last block to
// arrive adds the per-block partials in block order and resets the counter.
__device__ void finish_R(double rsum, double lambda, double *part, unsigned *count, double *R) {
    __shared__ double red[kThreads];
    __shared__ bool last;
    red[threadIdx.x] = rsum;
    __syncthreads();
    for (int w = kThreads / 2; w > 0; w >>= 1) {
        if ((int)threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
        __syncthreads();
    }
    if (threadIdx.x == 0) {
        part[blockIdx.x] = red[0];
        __threadfence();
        last = atomicAdd(count, 1u) == gridDim.x - 1;
    }
    __syncthreads();
    if (!last) return;
    __threadfence();
    double acc = 0.0;
    for (unsigned b = threadIdx.x; b < gridDim.x; b += kThreads) acc += __ldcg(part + b);
    red[threadIdx.x] = acc;
    __syncthreads();
    for (int w = kThreads / 2; w > 0; w >>= 1) {
        if ((int)threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
        __syncthreads();
    }
    if (threadIdx.x == 0) {
        *R = lambda * red[0];
        *count = 0;
    }
}

// Block-based layers with K % 8 == 0 and bm <= 256: a tile is one row-block x
// BW columns (BW = 8 G), brought into shared memory by one TMA box load.
// The grid is persistent; each block keeps NS tiles in flight in a ring of
// stages (one mbarrier each), so HBM reads overlap the reduction and the
// gradient stores of earlier tiles.  Thread (slice, group) takes columns
// 4 group .. 4 group + 3 of each half of the tile, in rows slice, slice + S,
// ... of the stage, so that the lanes' 16-B gradient stores of a row are
// contiguous; out-of-range rows and columns of a box read as zeros.  The slices' fp32 sums meet in shared
// memory and are added in slice order, one thread per column (= unit); the
// unit factors go back through shared memory and every thread writes the
// gradient of its elements, read again from the stage.
struct TmaArgs {
    CUtensorMap wmap;        // W: K inner, M rows; box BW x brows, no swizzle
    Geo g;
    int ns;                  // stages
    int brows;               // box rows = min(bm, M)
    uint32_t stage_bytes;    // brows * BW * 2
    float eps, lambda2;
    double lambda;
    double *alpha;
    float *grad;
    double *part;
    unsigned *count;
    double *R;
    unsigned *status;
    uint64_t watchdog_ns;
};

constexpr uint64_t kDrainNs = 1000000000ull;

template <bool kBF16>
__global__ void __launch_bounds__(kThreads) penalty_tma_kernel(const __grid_constant__ TmaArgs p) {
    extern __shared__ __align__(128) uint8_t smem_raw[];
    // TMA destinations 128-B aligned
    uint8_t *smem = smem_raw + ((128u - (smem_u32(smem_raw) & 127u)) & 127u);
    const Geo &g = p.g;
    const int tw = 8 * g.G;
    float *colsum = reinterpret_cast<float *>(smem + (size_t)p.ns * p.stage_bytes);
    float *coef = colsum + kThreads * 8;
    uint64_t *full = reinterpret_cast<uint64_t *>(coef + 256);
    __shared__ int timed_out;
    const int slice = threadIdx.x / g.G, grp = threadIdx.x % g.G;
    const int grid = gridDim.x;

    int issued = 0;              // thread 0: iterations whose loads are issued
    auto issue = [&](int it) {   // tile of the block's it-th iteration into stage it % ns
        const int t = blockIdx.x + it * grid;
        if (t >= g.tiles) return;
        issued = it + 1;
        const int rb = t / g.TC, tc = t - rb * g.TC;
        uint64_t *bar = &full[it % p.ns];
        mbar_arrive_expect_tx(bar, p.stage_bytes);
        tma_load_2d(smem_u32(smem + (size_t)(it % p.ns) * p.stage_bytes), &p.wmap, tc * tw,
                    rb * g.bm, bar);
    };

    if (threadIdx.x == 0) {
        timed_out = 0;
        for (int i = 0; i < p.ns; ++i) mbar_init(&full[i], 1);
        fence_mbar_init();
        prefetch_tmap(&p.wmap);
    }
    __syncthreads();
    if (threadIdx.x == 0)
        for (int i = 0; i < p.ns; ++i) issue(i);

    double rsum = 0.0;
    int it = 0;
    const int hw = tw / 2;   // a thread's columns: 4 g .. 4 g + 3 of each half of the tile
    for (int t = blockIdx.x; t < g.tiles; t += grid, ++it) {
        const int rb = t / g.TC, tc = t - rb * g.TC;
        const int nr = min(g.bm, g.M - rb * g.bm);   // rows of this row-block
        const int c0 = tc * tw + grp * 4;
        const bool v0 = c0 < g.K, v1 = c0 + hw < g.K;
        const int nrow = v0 && nr > slice ? (nr - slice + g.S - 1) / g.S : 0;
        const uint8_t *mine = smem + (size_t)(it % p.ns) * p.stage_bytes +
                              (size_t)slice * tw * 2 + grp * 8;
        const size_t rstride = (size_t)tw * 2 * g.S;   // bytes between a thread's rows

        const bool ok = mbar_wait(&full[it % p.ns], (uint32_t)((it / p.ns) & 1), p.watchdog_ns,
                                  nullptr);
        if (__syncthreads_or(!ok)) {
            if (threadIdx.x == 0) {
                atomicOr(p.status, kDevTimeout);
                timed_out = 1;
            }
            break;
        }
        float acc[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[j] = 0.f;
#pragma unroll 4
        for (int i = 0; i < nrow; ++i) {
            const uint2 a = *reinterpret_cast<const uint2 *>(mine + i * rstride);
            const uint2 b = *reinterpret_cast<const uint2 *>(mine + i * rstride + hw * 2);
            const uint32_t w4[4] = {a.x, a.y, b.x, b.y};
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const float lo = to_f32<kBF16>(w4[j] & 0xffffu);
                const float hi = to_f32<kBF16>(w4[j] >> 16);
                acc[2 * j] = fmaf(lo, lo, acc[2 * j]);
                acc[2 * j + 1] = fmaf(hi, hi, acc[2 * j + 1]);
            }
        }
        *reinterpret_cast<float4 *>(colsum + slice * tw + grp * 4) =
            make_float4(acc[0], acc[1], acc[2], acc[3]);
        *reinterpret_cast<float4 *>(colsum + slice * tw + hw + grp * 4) =
            make_float4(acc[4], acc[5], acc[6], acc[7]);
        __syncthreads();
        // every thread is past the previous iteration's stage: refill it
        if (threadIdx.x == 0 && it > 0) issue(it - 1 + p.ns);
        if ((int)threadIdx.x < tw) {
            // column j's S slice sums in slice order (S is a multiple of 8:
            // eight loads in flight per step)
            const int j = threadIdx.x, col = tc * tw + j;
            float sum = 0.f;
            for (int q = 0; q < g.S; q += 8) {
                float v[8];
#pragma unroll
                for (int u = 0; u < 8; ++u) v[u] = colsum[(q + u) * tw + j];
#pragma unroll
                for (int u = 0; u < 8; ++u) sum += v[u];
            }
            if (col < g.K)
                coef[j] = finish_unit(sum, p.eps, p.lambda2, p.alpha + (size_t)rb * g.K + col, rsum);
        }
        __syncthreads();
        if (nrow > 0) {
            // each warp store covers whole 32-B sectors: 8 lanes x 16 B per row
            const float4 k0 = *reinterpret_cast<const float4 *>(coef + grp * 4);
            const float4 k1 = *reinterpret_cast<const float4 *>(coef + hw + grp * 4);
            float *dst = p.grad + (size_t)(rb * g.bm + slice) * g.K + c0;
            const size_t gstep = (size_t)g.S * g.K;
#pragma unroll 4
            for (int i = 0; i < nrow; ++i) {
                const uint2 a = *reinterpret_cast<const uint2 *>(mine + i * rstride);
                const uint2 b = *reinterpret_cast<const uint2 *>(mine + i * rstride + hw * 2);
                float *d = dst + (size_t)i * gstep;
                *reinterpret_cast<float4 *>(d) =
                    make_float4(k0.x * to_f32<kBF16>(a.x & 0xffffu), k0.y * to_f32<kBF16>(a.x >> 16),
                                k0.z * to_f32<kBF16>(a.y & 0xffffu), k0.w * to_f32<kBF16>(a.y >> 16));
                if (v1)
                    *reinterpret_cast<float4 *>(d + hw) = make_float4(
                        k1.x * to_f32<kBF16>(b.x & 0xffffu), k1.y * to_f32<kBF16>(b.x >> 16),
                        k1.z * to_f32<kBF16>(b.y & 0xffffu), k1.w * to_f32<kBF16>(b.y >> 16));
            }
        }
    }
    if (timed_out && threadIdx.x == 0) {
        // let the loads already issued land before the block's shared memory
        // is released (R is then meaningless, but the workspace counter stays
        // consistent)
        for (int k = it; k < issued; ++k)
            mbar_wait(&full[k % p.ns], (uint32_t)((k / p.ns) & 1), kDrainNs, nullptr);
    }
    finish_R(rsum, p.lambda, p.part, p.count, p.R);
}

// Block-based layers with K % 8 == 0 and taller row-blocks: as above with
// S = 256 slices, but each thread walks its rows r0 + slice + 256 i in a loop
// and reads them a second time (from L1/L2) to write the gradient.  The slices' sums
// meet in shared memory and are added in slice order, one thread per column
// (= unit); the unit factors go back through shared memory and every thread
// writes the gradient of the elements it loaded.
template <bool kBF16>
__global__ void __launch_bounds__(kThreads) penalty_based_loop_kernel(
    Geo g, float eps, float lambda2, double lambda, const uint16_t *__restrict__ W,
    double *__restrict__ alpha, float *__restrict__ grad, double *__restrict__ part,
    unsigned *__restrict__ count, double *__restrict__ R) {
    __shared__ __align__(16) float colsum[kTileFloats];
    __shared__ __align__(16) float coef[kTileFloats];
    const int slice = threadIdx.x / g.G, grp = threadIdx.x % g.G;
    const int tw = 8 * g.G;   // tile width in columns
    double rsum = 0.0;
    for (int t = blockIdx.x; t < g.tiles; t += gridDim.x) {
        const int rb = t / g.TC, tc = t - rb * g.TC;
        const int r0 = rb * g.bm, r1 = min(r0 + g.bm, g.M);
        const int c0 = tc * tw + grp * 8;
        const bool active = c0 < g.K;
        const int nrow = r1 - r0 > slice ? (r1 - r0 - slice + g.S - 1) / g.S : 0;
        const uint16_t *src = W + (size_t)(r0 + slice) * g.K + c0;
        const size_t step = (size_t)g.S * g.K;
        float acc[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[j] = 0.f;
        if (active) {
            int i = 0;
            for (; i + 4 <= nrow; i += 4) {
                uint4 v[4];
#pragma unroll
                for (int q = 0; q < 4; ++q)
                    v[q] = __ldg(reinterpret_cast<const uint4 *>(src + (size_t)(i + q) * step));
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const uint32_t w4[4] = {v[q].x, v[q].y, v[q].z, v[q].w};
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        const float lo = to_f32<kBF16>(w4[j] & 0xffffu);
                        const float hi = to_f32<kBF16>(w4[j] >> 16);
                        acc[2 * j] = fmaf(lo, lo, acc[2 * j]);
                        acc[2 * j + 1] = fmaf(hi, hi, acc[2 * j + 1]);
                    }
                }
            }
            for (; i < nrow; ++i) {
                const uint4 v = __ldg(reinterpret_cast<const uint4 *>(src + (size_t)i * step));
                const uint32_t w4[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const float lo = to_f32<kBF16>(w4[j] & 0xffffu);
                    const float hi = to_f32<kBF16>(w4[j] >> 16);
                    acc[2 * j] = fmaf(lo, lo, acc[2 * j]);
                    acc[2 * j + 1] = fmaf(hi, hi, acc[2 * j + 1]);
                }
            }
        }
        float4 *cs = reinterpret_cast<float4 *>(colsum + slice * tw + grp * 8);
        cs[0] = make_float4(acc[0], acc[1], acc[2], acc[3]);
        cs[1] = make_float4(acc[4], acc[5], acc[6], acc[7]);
        __syncthreads();
        for (int j = threadIdx.x; j < tw; j += kThreads) {
            const int col = tc * tw + j;
            if (col >= g.K) break;
            float s = 0.f;
            for (int q = 0; q < g.S; ++q) s += colsum[q * tw + j];
            coef[j] = finish_unit(s, eps, lambda2, alpha + (size_t)rb * g.K + col, rsum);
        }
        __syncthreads();
        if (active) {
            const float4 k0 = *reinterpret_cast<const float4 *>(coef + grp * 8);
            const float4 k1 = *reinterpret_cast<const float4 *>(coef + grp * 8 + 4);
            const float k[8] = {k0.x, k0.y, k0.z, k0.w, k1.x, k1.y, k1.z, k1.w};
            float *dst = grad + (size_t)(r0 + slice) * g.K + c0;
            int i = 0;
            for (; i + 4 <= nrow; i += 4) {
                uint4 v[4];
#pragma unroll
                for (int q = 0; q < 4; ++q)
                    v[q] = __ldg(reinterpret_cast<const uint4 *>(src + (size_t)(i + q) * step));
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const uint32_t w4[4] = {v[q].x, v[q].y, v[q].z, v[q].w};
                    float o[8];
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        o[2 * j] = k[2 * j] * to_f32<kBF16>(w4[j] & 0xffffu);
                        o[2 * j + 1] = k[2 * j + 1] * to_f32<kBF16>(w4[j] >> 16);
                    }
                    float4 *d = reinterpret_cast<float4 *>(dst + (size_t)(i + q) * step);
                    d[0] = make_float4(o[0], o[1], o[2], o[3]);
                    d[1] = make_float4(o[4], o[5], o[6], o[7]);
                }
            }
            for (; i < nrow; ++i) {
                const uint4 v = __ldg(reinterpret_cast<const uint4 *>(src + (size_t)i * step));
                const uint32_t w4[4] = {v.x, v.y, v.z, v.w};
                float o[8];
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    o[2 * j] = k[2 * j] * to_f32<kBF16>(w4[j] & 0xffffu);
                    o[2 * j + 1] = k[2 * j + 1] * to_f32<kBF16>(w4[j] >> 16);
                }
                float4 *d = reinterpret_cast<float4 *>(dst + (size_t)i * step);
                d[0] = make_float4(o[0], o[1], o[2], o[3]);
                d[1] = make_float4(o[4], o[5], o[6], o[7]);
            }
        }
    }
    finish_R(rsum, lambda, part, count, R);
}

// Any layout: one thread per unit (neighbouring threads take neighbouring
// columns / kernel positions), fp32 sum over the unit's rows ascending, then
// channels ascending; the gradient from a second read of the unit.
template <bool kBF16>
__global__ void __launch_bounds__(kThreads) penalty_unit_kernel(
    Geo g, int scheme, float eps, float lambda2, double lambda, const uint16_t *__restrict__ W,
    double *__restrict__ alpha, float *__restrict__ grad, double *__restrict__ part,
    unsigned *__restrict__ count, double *__restrict__ R) {
    double rsum = 0.0;
    for (int64_t uu = blockIdx.x * kThreads + threadIdx.x; uu < g.U;
         uu += (int64_t)gridDim.x * kThreads) {
        const int u = (int)uu;
        int r0, col, c0 = 0, nc = 1, cs = 0;
        if (scheme == BP_BLOCK_BASED) {
            const int rb = u / g.K;
            col = u - rb * g.K;
            r0 = rb * g.bm;
        } else {
            const int b = u / g.KK, pos = u - b * g.KK;
            const int rb = b / g.CB, cb = b - rb * g.CB;
            r0 = rb * g.bm;
            c0 = cb * g.bk;
            nc = min(g.bk, g.C - c0);
            col = c0 * g.KK + pos;
            cs = g.KK;
        }
        const int r1 = min(r0 + g.bm, g.M);
        float s = 0.f;
        for (int r = r0; r < r1; ++r) {
            const uint16_t *row = W + (size_t)r * g.K + col;
            for (int c = 0; c < nc; ++c) {
                const float w = to_f32<kBF16>(__ldg(row + c * cs));
                s = fmaf(w, w, s);
            }
        }
        const float k = finish_unit(s, eps, lambda2, alpha + u, rsum);
        for (int r = r0; r < r1; ++r) {
            const size_t e = (size_t)r * g.K + col;
            for (int c = 0; c < nc; ++c)
                grad[e + (size_t)c * cs] = k * to_f32<kBF16>(__ldg(W + e + (size_t)c * cs));
        }
    }
    finish_R(rsum, lambda, part, count, R);
}

// Row groups of block-based layers (Eq. row): unit u = r * CB + cb is the
// contiguous segment W[r, cb*bk .. min(cb*bk + bk, K) - 1]; one thread per
// unit, so a warp reads 32 neighbouring segments of a row.  kVec: bk and K
// multiples of 8, segments read and written 16 B at a time.
template <bool kBF16, bool kVec>
__global__ void __launch_bounds__(kThreads) penalty_rows_kernel(
    Geo g, float eps, float lambda2, double lambda, const uint16_t *__restrict__ W,
    double *__restrict__ alpha, float *__restrict__ grad, double *__restrict__ part,
    unsigned *__restrict__ count, double *__restrict__ R) {
    double rsum = 0.0;
    for (int64_t uu = blockIdx.x * kThreads + threadIdx.x; uu < g.U;
         uu += (int64_t)gridDim.x * kThreads) {
        const int u = (int)uu;
        const int r = u / g.CB, cb = u - r * g.CB;
        const int k0 = cb * g.bk, n = min(g.bk, g.K - k0);
        const size_t e0 = (size_t)r * g.K + k0;
        float s = 0.f;
        if constexpr (kVec) {
            const uint4 *src = reinterpret_cast<const uint4 *>(W + e0);
            for (int i = 0; i < n / 8; ++i) {
                const uint4 v = __ldg(src + i);
                const uint32_t w4[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const float lo = to_f32<kBF16>(w4[j] & 0xffffu);
                    const float hi = to_f32<kBF16>(w4[j] >> 16);
                    s = fmaf(lo, lo, s);
                    s = fmaf(hi, hi, s);
                }
            }
        } else {
            for (int i = 0; i < n; ++i) {
                const float w = to_f32<kBF16>(__ldg(W + e0 + i));
                s = fmaf(w, w, s);
            }
        }
        const float k = finish_unit(s, eps, lambda2, alpha + u, rsum);
        if constexpr (kVec) {
            const uint4 *src = reinterpret_cast<const uint4 *>(W + e0);
            float4 *dst = reinterpret_cast<float4 *>(grad + e0);
            for (int i = 0; i < n / 8; ++i) {
                const uint4 v = __ldg(src + i);
                dst[2 * i] = make_float4(k * to_f32<kBF16>(v.x & 0xffffu), k * to_f32<kBF16>(v.x >> 16),
                                         k * to_f32<kBF16>(v.y & 0xffffu), k * to_f32<kBF16>(v.y >> 16));
                dst[2 * i + 1] =
                    make_float4(k * to_f32<kBF16>(v.z & 0xffffu), k * to_f32<kBF16>(v.z >> 16),
                                k * to_f32<kBF16>(v.w & 0xffffu), k * to_f32<kBF16>(v.w >> 16));
            }
        } else {
            for (int i = 0; i < n; ++i) grad[e0 + i] = k * to_f32<kBF16>(__ldg(W + e0 + i));
        }
    }
    finish_R(rsum, lambda, part, count, R);
}

// Row groups when bk is 8, 16, ..., 256 and divides K: the weight is one
// stream of M K / bk whole segments, taken 256 weights per warp.  Lane l loads
// weights 8l .. 8l + 7 (16 B; a warp load covers 512 contiguous bytes); the
// L = bk / 8 lanes of a segment add their fp32 sums with a fixed butterfly,
// the segment's first lane forms the factors, and the factor goes back to the
// segment by a shuffle.  (Lanes store their 32 gradient bytes as two 16-B
// halves; exchanging values between lanes so that each warp store covers
// whole sectors, or 8-byte loads with that layout, measured slower.)
template <bool kBF16>
__global__ void __launch_bounds__(kThreads) penalty_rows_warp_kernel(
    Geo g, float eps, float lambda2, double lambda, const uint16_t *__restrict__ W,
    double *__restrict__ alpha, float *__restrict__ grad, double *__restrict__ part,
    unsigned *__restrict__ count, double *__restrict__ R) {
    const int lane = threadIdx.x & 31;
    const int L = g.bk / 8;                        // lanes per segment (a power of two)
    const int64_t total = (int64_t)g.M * g.K;      // a multiple of bk
    const int64_t chunks = (total + 255) / 256;    // 256 weights per warp
    const int64_t warps = (int64_t)gridDim.x * (kThreads / 32);
    double rsum = 0.0;
    for (int64_t c = blockIdx.x * (int64_t)(kThreads / 32) + threadIdx.x / 32; c < chunks;
         c += warps) {
        const int64_t e = c * 256 + lane * 8;
        const bool in = e < total;
        uint4 v = make_uint4(0, 0, 0, 0);
        if (in) v = __ldg(reinterpret_cast<const uint4 *>(W + e));
        const uint32_t w4[4] = {v.x, v.y, v.z, v.w};
        float s = 0.f;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const float lo = to_f32<kBF16>(w4[j] & 0xffffu);
            const float hi = to_f32<kBF16>(w4[j] >> 16);
            s = fmaf(lo, lo, s);
            s = fmaf(hi, hi, s);
        }
        for (int m = 1; m < L; m *= 2) s += __shfl_xor_sync(0xffffffffu, s, m);
        float k = 0.f;
        if (in && (lane & (L - 1)) == 0)
            k = finish_unit(s, eps, lambda2, alpha + e / g.bk, rsum);
        k = __shfl_sync(0xffffffffu, k, lane & ~(L - 1));
        if (in) {
            float4 *d = reinterpret_cast<float4 *>(grad + e);
            d[0] = make_float4(k * to_f32<kBF16>(v.x & 0xffffu), k * to_f32<kBF16>(v.x >> 16),
                               k * to_f32<kBF16>(v.y & 0xffffu), k * to_f32<kBF16>(v.y >> 16));
            d[1] = make_float4(k * to_f32<kBF16>(v.z & 0xffffu), k * to_f32<kBF16>(v.z >> 16),
                               k * to_f32<kBF16>(v.w & 0xffffu), k * to_f32<kBF16>(v.w >> 16));
        }
    }
    finish_R(rsum, lambda, part, count, R);
}

enum class Path { kTma, kLoop, kUnit, kRows, kRowsWarp };

constexpr int kMaxBoxRows = 256;   // TMA box dimension limit

Path path_of(const bp_layout &l, int groups) {
    if (groups == BP_GROUPS_ROWS) {
        const bool pow2 = (l.bk & (l.bk - 1)) == 0;
        return l.bk % 8 == 0 && l.bk <= 256 && pow2 && l.K % l.bk == 0 ? Path::kRowsWarp
                                                                     : Path::kRows;
    }
    if (l.scheme != BP_BLOCK_BASED || l.K % 8 != 0) return Path::kUnit;
    return (l.bm < l.M ? l.bm : l.M) <= kMaxBoxRows ? Path::kTma : Path::kLoop;
}

// TMA tiles: about 16 KB per stage, BW in {64, 128, 256} columns.
int box_width(int brows) {
    int bw = 64;
    while (bw < 256 && brows * bw * 2 * 2 <= 16384) bw *= 2;
    return bw;
}

Geo make_geo(const bp_layout &l, int groups) {
    Geo g{};
    g.M = (int)l.M;
    g.K = (int)l.K;
    g.KK = l.kh * l.kw;
    g.C = g.K / g.KK;
    g.bm = l.bm;
    g.bk = l.bk;
    g.RB = (int)((l.M + l.bm - 1) / l.bm);
    if (l.scheme == BP_BLOCK_BASED) {
        g.CB = (g.K + l.bk - 1) / l.bk;
        g.U = groups == BP_GROUPS_ROWS ? g.M * g.CB : g.RB * g.K;
    } else {
        g.CB = (g.C + l.bk - 1) / l.bk;
        g.U = g.RB * g.CB * g.KK;
    }
    const int brows = min(l.bm, g.M);
    g.G = path_of(l, groups) == Path::kTma ? box_width(brows) / 8 : 16;
    g.S = kThreads / g.G;
    g.TC = (g.K + 8 * g.G - 1) / (8 * g.G);
    g.tiles = g.RB * g.TC;
    return g;
}

// Upper bound of the grid (what the workspace is sized for).
int max_grid(const bp_layout &l, int groups, const Geo &g) {
    const Path path = path_of(l, groups);
    int n = g.tiles;
    if (path == Path::kUnit || path == Path::kRows) n = (g.U + kThreads - 1) / kThreads;
    if (path == Path::kRowsWarp)   // eight warps of 256 weights per block
        n = (int)(((int64_t)g.M * g.K + 2047) / 2048);
    return max(1, min(n, kMaxBlocks));
}

cudaError_t launch_tma(const bp_layout &lay, const Geo &g, const void *W, float eps,
                       float lambda2, double lambda, double *alpha, float *grad, double *part,
                       unsigned *count, double *R, cudaStream_t s) {
    TmaArgs a{};
    a.g = g;
    a.brows = min(lay.bm, g.M);
    a.stage_bytes = (uint32_t)a.brows * (uint32_t)(8 * g.G) * 2u;
    a.ns = max(2, min(8, 65536 / (int)a.stage_bytes));
    a.eps = eps;
    a.lambda2 = lambda2;
    a.lambda = lambda;
    a.alpha = alpha;
    a.grad = grad;
    a.part = part;
    a.count = count;
    a.R = R;
    a.status = device_status_ptr();
    a.watchdog_ns = watchdog_ns();
    PFN_cuTensorMapEncodeTiled_v12000 enc = tensor_map_encoder();
    if (!enc || !a.status) return cudaErrorNotSupported;
    const cuuint64_t gdim[2] = {(cuuint64_t)g.K, (cuuint64_t)g.M};
    const cuuint64_t gstride[1] = {(cuuint64_t)g.K * 2};
    const cuuint32_t box[2] = {(cuuint32_t)(8 * g.G), (cuuint32_t)a.brows};
    const cuuint32_t estride[2] = {1, 1};
    const CUtensorMapDataType tdt =
        lay.dtype == BP_BF16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT16;
    if (enc(&a.wmap, tdt, 2, const_cast<void *>(W), gdim, gstride, box, estride,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
        return cudaErrorInvalidValue;
    const size_t smem = 128 + (size_t)a.ns * a.stage_bytes +
                        sizeof(float) * (kThreads * 8 + 256) + sizeof(uint64_t) * 8;
    const bool bf = lay.dtype == BP_BF16;
    auto k = bf ? penalty_tma_kernel<true> : penalty_tma_kernel<false>;
    // the shared-memory ceiling once (ns * stage_bytes <= 64 KB for every
    // layout), then the resident blocks per SM for each (dtype, size)
    static std::once_flag once;
    static cudaError_t attr_err = cudaSuccess;
    std::call_once(once, [] {
        const int most = (int)(128 + 65536 + sizeof(float) * (kThreads * 8 + 256) +
                               sizeof(uint64_t) * 8);
        attr_err = cudaFuncSetAttribute(penalty_tma_kernel<true>,
                                        cudaFuncAttributeMaxDynamicSharedMemorySize, most);
        if (attr_err == cudaSuccess)
            attr_err = cudaFuncSetAttribute(penalty_tma_kernel<false>,
                                            cudaFuncAttributeMaxDynamicSharedMemorySize, most);
    });
    if (attr_err != cudaSuccess) return attr_err;
    static std::mutex mu;
    static std::map<std::pair<bool, size_t>, int> resident;
    int per_sm = 0;
    {
        std::lock_guard<std::mutex> lock(mu);
        auto f = resident.find({bf, smem});
        if (f == resident.end()) {
            const cudaError_t e =
                cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k, kThreads, smem);
            if (e != cudaSuccess) return e;
            f = resident.emplace(std::make_pair(bf, smem), max(1, per_sm)).first;
        }
        per_sm = f->second;
    }
    const int grid = max(1, min(max_grid(lay, BP_GROUPS_LAYOUT, g), per_sm * num_sms()));
    k<<<grid, kThreads, smem, s>>>(a);
    return cudaGetLastError();
}

}  // namespace

size_t penalty_workspace_bytes(const bp_layout &lay, int groups) {
    return 256 + sizeof(double) * (size_t)max_grid(lay, groups, make_geo(lay, groups));
}

cudaError_t launch_penalty(const bp_layout &lay, int groups, const void *W, double eps,
                           double lambda, double *alpha, double *R, float *grad, void *ws,
                           cudaStream_t s) {
    const Geo g = make_geo(lay, groups);
    int grid = max_grid(lay, groups, g);
    unsigned *count = static_cast<unsigned *>(ws);
    double *part = reinterpret_cast<double *>(static_cast<char *>(ws) + 256);
    const uint16_t *w = static_cast<const uint16_t *>(W);
    const float eps_f = (float)eps, lambda2_f = (float)(2.0 * lambda);
    const bool bf = lay.dtype == BP_BF16;
    switch (path_of(lay, groups)) {
    case Path::kRowsWarp: {
        auto k = bf ? penalty_rows_warp_kernel<true> : penalty_rows_warp_kernel<false>;
        k<<<grid, kThreads, 0, s>>>(g, eps_f, lambda2_f, lambda, w, alpha, grad, part, count, R);
        break;
    }
    case Path::kRows: {
        const bool vec = lay.bk % 8 == 0 && lay.K % 8 == 0;
        auto k = bf ? (vec ? penalty_rows_kernel<true, true> : penalty_rows_kernel<true, false>)
                    : (vec ? penalty_rows_kernel<false, true> : penalty_rows_kernel<false, false>);
        k<<<grid, kThreads, 0, s>>>(g, eps_f, lambda2_f, lambda, w, alpha, grad, part, count, R);
        break;
    }
    case Path::kTma:
        return launch_tma(lay, g, W, eps_f, lambda2_f, lambda, alpha, grad, part, count, R, s);
    case Path::kLoop: {
        auto k = bf ? penalty_based_loop_kernel<true> : penalty_based_loop_kernel<false>;
        k<<<grid, kThreads, 0, s>>>(g, eps_f, lambda2_f, lambda, w, alpha, grad, part, count, R);
        break;
    }
    case Path::kUnit: {
        auto k = bf ? penalty_unit_kernel<true> : penalty_unit_kernel<false>;
        k<<<grid, kThreads, 0, s>>>(g, lay.scheme, eps_f, lambda2_f, lambda, w, alpha, grad, part,
                                    count, R);
        break;
    }
    }
    return cudaGetLastError();
}

}  // namespace bp
