// Packing kernels: mask -> per-row-block kept-column counts (with the check
// that all rows of a row-block agree, the BCS occurrence property of
// Sec. 4.3), then col_idx / values (the canonical compact arrays), the device
// image the tensor-core kernel streams (128-row slabs, see DevLayout), and the
// im2col expansion used by convolutions.
#include "bp_common.cuh"

namespace bp {
namespace {

constexpr int kScanThreads = 1024;

// One block per row-block: K'_rb from the first row; `bad` if another row of
// the row-block keeps a different set of columns.
__global__ void rb_counts_kernel(int64_t M, int64_t K, int64_t bm,
                                 const uint8_t *__restrict__ mask, int64_t *__restrict__ cnt,
                                 int *__restrict__ bad) {
    const int64_t rb = blockIdx.x;
    const int64_t r0 = rb * bm, r1 = min(r0 + bm, M);
    int local = 0;
    bool mismatch = false;
    for (int64_t k = threadIdx.x; k < K; k += blockDim.x) {
        const uint8_t m0 = mask[r0 * K + k] != 0;
        local += m0;
        for (int64_t r = r0 + 1; r < r1; ++r) mismatch |= ((mask[r * K + k] != 0) != m0);
    }
    __shared__ int total;
    if (threadIdx.x == 0) total = 0;
    __syncthreads();
    atomicAdd(&total, local);
    if (mismatch) atomicExch(bad, 1);
    __syncthreads();
    if (threadIdx.x == 0) cnt[rb] = total;
}

// In-place exclusive scan of n int64 values (one block).
__global__ void exclusive_scan_kernel(int64_t n, int64_t *__restrict__ v) {
    __shared__ int64_t part[kScanThreads];
    __shared__ int64_t carry;
    if (threadIdx.x == 0) carry = 0;
    __syncthreads();
    for (int64_t base = 0; base < n; base += kScanThreads) {
        const int64_t i = base + threadIdx.x;
        const int64_t x = i < n ? v[i] : 0;
        part[threadIdx.x] = x;
        __syncthreads();
        for (int off = 1; off < kScanThreads; off <<= 1) {
            const int64_t t = threadIdx.x >= off ? part[threadIdx.x - off] : 0;
            __syncthreads();
            part[threadIdx.x] += t;
            __syncthreads();
        }
        if (i < n) v[i] = carry + part[threadIdx.x] - x;
        __syncthreads();
        if (threadIdx.x == kScanThreads - 1) carry += part[threadIdx.x];
        __syncthreads();
    }
}

// Ordered compaction of the first row of each row-block: col_idx ascending.
__global__ void col_idx_kernel(int64_t K, int64_t bm, const uint8_t *__restrict__ mask,
                               const int64_t *__restrict__ rb_ptr, int32_t *__restrict__ col_idx) {
    __shared__ int part[kScanThreads];
    __shared__ int64_t carry;
    const int64_t rb = blockIdx.x;
    const uint8_t *row = mask + rb * bm * K;
    if (threadIdx.x == 0) carry = rb_ptr[rb];
    __syncthreads();
    for (int64_t base = 0; base < K; base += kScanThreads) {
        const int64_t k = base + threadIdx.x;
        const int f = (k < K && row[k]) ? 1 : 0;
        part[threadIdx.x] = f;
        __syncthreads();
        for (int off = 1; off < kScanThreads; off <<= 1) {
            const int t = threadIdx.x >= off ? part[threadIdx.x - off] : 0;
            __syncthreads();
            part[threadIdx.x] += t;
            __syncthreads();
        }
        if (f) col_idx[carry + part[threadIdx.x] - 1] = (int32_t)k;
        __syncthreads();
        if (threadIdx.x == kScanThreads - 1) carry += part[threadIdx.x];
        __syncthreads();
    }
}

// values[bm*rb_ptr[rb] + (r - r0)*K'_rb + i] = W[r, col_idx[rb_ptr[rb] + i]]
__global__ void values_kernel(int64_t M, int64_t K, int64_t bm,
                              const uint16_t *__restrict__ W, const int64_t *__restrict__ rb_ptr,
                              const int32_t *__restrict__ col_idx, uint16_t *__restrict__ values) {
    const int64_t rb = blockIdx.x;
    const int64_t r0 = rb * bm, rows = min(bm, M - r0);
    const int64_t p0 = rb_ptr[rb], kp = rb_ptr[rb + 1] - p0;
    const int64_t n = rows * kp;
    for (int64_t t = threadIdx.x; t < n; t += blockDim.x) {
        const int64_t r = t / kp, i = t % kp;
        values[bm * p0 + t] = W[(r0 + r) * K + col_idx[p0 + i]];
    }
}

// Is column k kept by any row of slab s?  (rows of a row-block are identical,
// so the first row of each row-block the slab touches decides)
__device__ __forceinline__ bool slab_keeps(const uint8_t *__restrict__ mask, int64_t M, int64_t K,
                                           int64_t bm, int64_t s, int64_t k) {
    const int64_t r0 = s * kSlab, r1 = min(r0 + kSlab, M);
    for (int64_t rb = r0 / bm; rb * bm < r1; ++rb)
        if (mask[rb * bm * K + k]) return true;
    return false;
}

// One block per slab, one warp per aligned 64-column block at a time.
__global__ void slab_counts_kernel(int64_t M, int64_t K, int64_t bm,
                                   const uint8_t *__restrict__ mask, int64_t *__restrict__ info) {
    const int64_t s = blockIdx.x;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nwarps = blockDim.x >> 5;
    int64_t dense = 0, sparse = 0;
    for (int64_t blk = warp; blk * kBK < K; blk += nwarps) {
        const int64_t k0 = blk * kBK;
        const bool a = k0 + lane < K && slab_keeps(mask, M, K, bm, s, k0 + lane);
        const bool b = k0 + 32 + lane < K && slab_keeps(mask, M, K, bm, s, k0 + 32 + lane);
        const int u = __popc(__ballot_sync(0xffffffffu, a)) + __popc(__ballot_sync(0xffffffffu, b));
        const bool whole = u >= kDenseMin && k0 + kBK <= K;
        if (whole) ++dense;
        else sparse += u;
    }
    __shared__ unsigned long long sd, ss;
    if (threadIdx.x == 0) sd = ss = 0;
    __syncthreads();
    if (lane == 0) {
        atomicAdd(&sd, (unsigned long long)dense);
        atomicAdd(&ss, (unsigned long long)sparse);
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        info[2 * s] = (int64_t)sd;
        info[2 * s + 1] = (int64_t)ss;
    }
}

// One warp per slab: the slab's chunk column lists, dense blocks first (in
// block order), then the remaining union columns ascending, 64 per chunk; the
// last chunk's unused entries repeat its last index.
__global__ void slab_lists_kernel(int64_t M, int64_t K, int64_t bm, const uint8_t *__restrict__ mask,
                                  const int64_t *__restrict__ kc_ptr, uint8_t *__restrict__ meta) {
    const int64_t s = blockIdx.x;
    const int lane = threadIdx.x;
    const int64_t c0 = kc_ptr[s], nkc = kc_ptr[s + 1] - c0;
    if (nkc == 0) return;
    auto list = [&](int64_t c) {
        return reinterpret_cast<int32_t *>(meta + (c0 + c) * kMetaBytes);
    };
    int64_t ndense = 0;
    for (int64_t k0 = 0; k0 < K; k0 += kBK) {
        const bool a = k0 + lane < K && slab_keeps(mask, M, K, bm, s, k0 + lane);
        const bool b = k0 + 32 + lane < K && slab_keeps(mask, M, K, bm, s, k0 + 32 + lane);
        const int u = __popc(__ballot_sync(0xffffffffu, a)) + __popc(__ballot_sync(0xffffffffu, b));
        if (u >= kDenseMin && k0 + kBK <= K) {
            int32_t *l = list(ndense++);
            l[lane] = (int32_t)(k0 + lane);
            l[lane + 32] = (int32_t)(k0 + 32 + lane);
        }
    }
    int64_t pos = ndense * kBK;        // next free slot (chunk-major)
    int32_t last = 0;
    for (int64_t k0 = 0; k0 < K; k0 += kBK) {
        const bool a = k0 + lane < K && slab_keeps(mask, M, K, bm, s, k0 + lane);
        const bool b = k0 + 32 + lane < K && slab_keeps(mask, M, K, bm, s, k0 + 32 + lane);
        const unsigned ba = __ballot_sync(0xffffffffu, a), bb = __ballot_sync(0xffffffffu, b);
        const int u = __popc(ba) + __popc(bb);
        if (u == 0 || (u >= kDenseMin && k0 + kBK <= K)) continue;
        const unsigned below = (1u << lane) - 1u;
        if (a) {
            const int64_t q = pos + __popc(ba & below);
            list(q / kBK)[q % kBK] = (int32_t)(k0 + lane);
        }
        if (b) {
            const int64_t q = pos + __popc(ba) + __popc(bb & below);
            list(q / kBK)[q % kBK] = (int32_t)(k0 + 32 + lane);
        }
        const int hi = bb ? 32 + (31 - __clz(bb)) : 31 - __clz(ba);
        last = (int32_t)(k0 + hi);
        pos += u;
    }
    __syncwarp();
    // pad the last sparse chunk
    const int64_t end = nkc * kBK;
    for (int64_t q = pos + lane; q < end; q += 32) list(q / kBK)[q % kBK] = last;
}

// Tiles: one thread per 16-byte unit (8 consecutive list entries of one row).
// Entry e of a chunk is live when e == 0 or its index differs from entry e-1
// (lists ascend; padding repeats); dead entries and pruned weights are 0.
__global__ void tiles_kernel(int64_t M, int64_t K, const uint16_t *__restrict__ W,
                             const uint8_t *__restrict__ mask, const int64_t *__restrict__ kc_ptr,
                             uint8_t *__restrict__ tiles, const uint8_t *__restrict__ meta,
                             int64_t tile_bytes) {
    const int64_t s = blockIdx.y;
    const int64_t c0 = kc_ptr[s], nkc = kc_ptr[s + 1] - c0;
    const int64_t units = nkc * kSlab * (kBK / 8);
    for (int64_t u = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; u < units;
         u += (int64_t)gridDim.x * blockDim.x) {
        const int64_t kc = u / (kSlab * (kBK / 8));
        const int64_t rem = u % (kSlab * (kBK / 8));
        const uint32_t row = (uint32_t)(rem / (kBK / 8));
        const uint32_t ch = (uint32_t)(rem % (kBK / 8));
        uint8_t *chunk = tiles + (c0 + kc) * tile_bytes;
        const int32_t *l = reinterpret_cast<const int32_t *>(meta + (c0 + kc) * kMetaBytes);
        const int64_t r = s * kSlab + row;
        uint16_t v[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const int q = (int)ch * 8 + e;
            const int32_t k = l[q];
            const bool live = q == 0 || k != l[q - 1];
            v[e] = (live && r < M && mask[r * K + k]) ? W[r * K + k] : (uint16_t)0;
        }
        uint4 pk;
        pk.x = v[0] | ((uint32_t)v[1] << 16);
        pk.y = v[2] | ((uint32_t)v[3] << 16);
        pk.z = v[4] | ((uint32_t)v[5] << 16);
        pk.w = v[6] | ((uint32_t)v[7] << 16);
        *reinterpret_cast<uint4 *>(chunk + sw128_kmajor_offset(row, ch * 8)) = pk;
    }
}

// Load plans: one thread per chunk.  The 64 list positions form 8 groups of 8;
// a group can be one tile load when each live entry (first occurrence of its
// index) is the group's first column plus its offset.  When every group can,
// maximal runs of groups that continue one another (first column 8 past the
// previous group's, or no live entry at all: padding, whose rows meet zero
// weights) become loads of 64, 32, 16 or 8 rows; otherwise the plan is empty
// and the kernel gathers the chunk's rows one by one.
// bound (device, or nullptr for none): no load may reach row *bound.
__global__ void plans_kernel(int64_t kc_total, uint8_t *__restrict__ meta_all,
                             const int64_t *__restrict__ bound) {
    const int64_t lim = bound ? *bound : INT64_MAX;
    for (int64_t c = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; c < kc_total;
         c += (int64_t)gridDim.x * blockDim.x) {
        uint8_t *meta = meta_all + c * kMetaBytes;
        const int32_t *l = reinterpret_cast<const int32_t *>(meta);
        int32_t first[8];
        bool ok = true;
        for (int g = 0; g < 8; ++g) {
            first[g] = l[8 * g];
            for (int i = 1; i < 8; ++i) {
                const int q = 8 * g + i;
                if (l[q] != l[q - 1] && l[q] != first[g] + i) ok = false;
            }
        }
        int32_t w[kPlanBytes / 4];
        for (int i = 0; i < kPlanBytes / 4; ++i) w[i] = 0;
        if (ok) {
            int nb = 0;
            uint32_t desc[2] = {0u, 0u};
            for (int g = 0; g < 8;) {
                int run = 1;
                while (g + run < 8 && (first[g + run] == first[g] + 8 * run ||
                                       l[8 * (g + run)] == l[8 * (g + run) - 1]))
                    ++run;
                const int lg = run >= 8 ? 3 : run >= 4 ? 2 : run >= 2 ? 1 : 0;
                if ((int64_t)first[g] + (8 << lg) > lim) {
                    nb = 0;
                    break;
                }
                w[1 + nb] = first[g];
                desc[nb >> 2] |= (uint32_t)(g | (lg << 4)) << (8 * (nb & 3));
                ++nb;
                g += 1 << lg;
            }
            if (nb == 0) desc[0] = desc[1] = 0u, w[1] = w[2] = w[3] = w[4] = w[5] = w[6] = w[7] = w[8] = 0;
            w[0] = nb;
            w[9] = (int32_t)desc[0];
            w[10] = (int32_t)desc[1];
        }
        int32_t *plan = reinterpret_cast<int32_t *>(meta + kListBytes);
        for (int i = 0; i < kPlanBytes / 4; ++i) plan[i] = w[i];
    }
}

// Columns listed by any slab: qmap[k] = 1 for every list entry (qmap zeroed
// first; equal values, so the racing writes agree).
__global__ void mark_listed_kernel(int64_t entries, const uint8_t *__restrict__ meta,
                                   int32_t *__restrict__ qmap) {
    for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < entries;
         e += (int64_t)gridDim.x * blockDim.x) {
        const int32_t k = reinterpret_cast<const int32_t *>(meta + (e / kBK) * kMetaBytes)[e % kBK];
        qmap[k] = 1;
    }
}

// One block: marks -> ranks (exclusive scan in column order), -1 where
// unmarked; *kc_out = number of listed columns.
__global__ void __launch_bounds__(1024) qmap_scan_kernel(int64_t K, int32_t *__restrict__ qmap,
                                                         int64_t *__restrict__ kc_out) {
    __shared__ int32_t warp_sum[32];
    __shared__ int32_t carry;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (threadIdx.x == 0) carry = 0;
    __syncthreads();
    for (int64_t k0 = 0; k0 < K; k0 += blockDim.x) {
        const int64_t k = k0 + threadIdx.x;
        const int32_t f = k < K ? qmap[k] : 0;
        const unsigned bal = __ballot_sync(0xffffffffu, f != 0);
        const int within = __popc(bal & ((1u << lane) - 1u));
        if (lane == 0) warp_sum[warp] = __popc(bal);
        __syncthreads();
        int before = 0, total = 0;
        for (int w = 0; w < (int)(blockDim.x >> 5); ++w) {
            if (w < warp) before += warp_sum[w];
            total += warp_sum[w];
        }
        if (k < K) qmap[k] = f ? carry + before + within : -1;
        __syncthreads();
        if (threadIdx.x == 0) carry += total;
        __syncthreads();
    }
    if (threadIdx.x == 0) *kc_out = carry;
}

// Records in compacted coordinates: each list entry replaced by its rank.
__global__ void compact_lists_kernel(int64_t entries, const uint8_t *__restrict__ meta,
                                     uint8_t *__restrict__ meta2, const int32_t *__restrict__ qmap) {
    for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < entries;
         e += (int64_t)gridDim.x * blockDim.x) {
        const int64_t c = e / kBK, i = e % kBK;
        const int32_t k = reinterpret_cast<const int32_t *>(meta + c * kMetaBytes)[i];
        reinterpret_cast<int32_t *>(meta2 + c * kMetaBytes)[i] = qmap[k];
    }
}

// im2col of a 1x1, stride-1, unpadded convolution: row c of the im2col
// matrix is the concatenation over images b of in[b, c, :, :].  One block per
// (channel, image): a contiguous copy of H*W values, 16 bytes per thread when
// source and destination are 16-byte aligned.
__global__ void __launch_bounds__(256) im2col_copy_kernel(int64_t C, int64_t HW, int64_t ldx,
                                                          const int32_t *__restrict__ qmap,
                                                          const uint16_t *__restrict__ in,
                                                          uint16_t *__restrict__ xcol) {
    const int64_t c = blockIdx.x, b = blockIdx.y;
    const int64_t q = qmap ? qmap[c] : c;      // the row this channel becomes, or none
    if (q < 0) return;
    const uint16_t *src = in + (b * C + c) * HW;
    uint16_t *dst = xcol + q * ldx + b * HW;
    if (((reinterpret_cast<uintptr_t>(src) | reinterpret_cast<uintptr_t>(dst)) & 15u) == 0) {
        const int64_t nv = HW / 8;
        for (int64_t q = threadIdx.x; q < nv; q += blockDim.x)
            reinterpret_cast<uint4 *>(dst)[q] = __ldg(reinterpret_cast<const uint4 *>(src) + q);
        for (int64_t e = nv * 8 + threadIdx.x; e < HW; e += blockDim.x) dst[e] = src[e];
    } else {
        for (int64_t e = threadIdx.x; e < HW; e += blockDim.x) dst[e] = __ldg(src + e);
    }
}

// im2col of a 1x1 convolution with stride or padding: row c of the im2col
// matrix holds in[b, c, oh*sh - ph, ow*sw - pw] (zero outside) for every output
// pixel.  One block per (channel, image); warps over output rows, lanes along
// them (coalesced stores, strided loads).
__global__ void __launch_bounds__(256) im2col_1x1_kernel(ConvShape cs, int64_t ldx,
                                                         const int32_t *__restrict__ qmap,
                                                         const uint16_t *__restrict__ in,
                                                         uint16_t *__restrict__ xcol) {
    const int H = (int)cs.H, W = (int)cs.W, Ho = (int)cs.Ho, Wo = (int)cs.Wo;
    const int64_t c = blockIdx.x, b = blockIdx.y;
    const int64_t q = qmap ? qmap[c] : c;
    if (q < 0) return;
    const uint16_t *src = in + (b * cs.C + c) * H * W;
    uint16_t *dst = xcol + q * ldx + b * Ho * Wo;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
    for (int oh = warp; oh < Ho; oh += nwarps) {
        const int ih = oh * cs.sh - cs.ph;
        const bool row_in = (unsigned)ih < (unsigned)H;
        for (int ow = lane; ow < Wo; ow += 32) {
            const int iw = ow * cs.sw - cs.pw;
            dst[oh * Wo + ow] =
                (row_in && (unsigned)iw < (unsigned)W) ? __ldg(src + ih * W + iw) : (uint16_t)0;
        }
    }
}

// im2col with threads along the rows (any kernel size, stride and
// padding; small or unaligned planes): row q = qmap[k] of the im2col matrix,
// k = c*kh*kw + i*kw + j, column e = b*Ho*Wo + oh*Wo + ow, holds
// in[b, c, oh*sh - ph + i, ow*sw - pw + j] (zero outside).  Grid (column
// groups, K): each thread writes 8 consecutive columns with one 16-byte store
// (ldx is a multiple of 8, so the group stays inside the row's ldx columns;
// columns past N get zeros), walking (b, oh, ow) incrementally from its first
// column.  A warp covers 256 consecutive columns of one row whatever the plane
// size; the rows of one channel read the same input pixels, from L2.
// k1: a 1x1 kernel (row k is channel k).
template <bool k1>
__global__ void __launch_bounds__(256) im2col_rows_kernel(ConvShape cs, int64_t ldx,
                                                          const int32_t *__restrict__ qmap,
                                                          const uint16_t *__restrict__ in,
                                                          uint16_t *__restrict__ xcol) {
    const int64_t k = blockIdx.y;
    const int64_t q = qmap ? qmap[k] : k;
    if (q < 0) return;
    uint32_t c = (uint32_t)k;                                   // k < 65536 (grid y)
    int di = -cs.ph, dj = -cs.pw;
    if (!k1) {
        const uint32_t kk = (uint32_t)(cs.kh * cs.kw);
        c = (uint32_t)k / kk;
        const int pos = (int)((uint32_t)k - c * kk);
        di += pos / cs.kw;
        dj += pos % cs.kw;
    }
    const uint32_t Wo = (uint32_t)cs.Wo, HoWo = (uint32_t)(cs.Ho * cs.Wo);
    const uint32_t N = (uint32_t)cs.Nb * HoWo;                  // < 2^31 (checked on the host)
    const uint32_t e0 = (blockIdx.x * 256u + threadIdx.x) * 8u;
    if (e0 >= N) return;
    uint32_t b = e0 / HoWo, r = e0 - b * HoWo;
    uint32_t oh = r / Wo, ow = r - oh * Wo;
    uint32_t w[4];
#pragma unroll
    for (int t = 0; t < 8; ++t) {
        uint16_t v = 0;
        if (e0 + t < N) {
            const int ih = (int)(oh * cs.sh) + di, iw = (int)(ow * cs.sw) + dj;
            if ((unsigned)ih < (unsigned)cs.H && (unsigned)iw < (unsigned)cs.W)
                v = __ldg(in + (((int64_t)b * cs.C + c) * cs.H + ih) * cs.W + iw);
            if (++ow == Wo) {
                ow = 0;
                if (++oh == (uint32_t)cs.Ho) {
                    oh = 0;
                    ++b;
                }
            }
        }
        if (t & 1)
            w[t >> 1] |= (uint32_t)v << 16;
        else
            w[t >> 1] = v;
    }
    *reinterpret_cast<uint4 *>(xcol + q * ldx + e0) = make_uint4(w[0], w[1], w[2], w[3]);
}

// im2col of a 3x3, stride-1, padding-1 convolution whose image has H*W a
// multiple of 8: one block per (group of ppb channels, image).  The block
// stages the channels' padded planes ((H+2) x (W+2) each) once, collects each
// channel's listed window positions, then writes each listed row 8 pixels
// (16 bytes) per thread, consecutive threads on consecutive pixels (512
// contiguous bytes per warp store).  A pixel group's 8 window offsets are
// computed once and reused for every listed position.  Small images take
// several channels per block so that every thread has a pixel group.
constexpr int kPlaneMaxChannels = 128;
constexpr int64_t kPlaneSmem = 40 * 1024;   // dynamic shared memory (the tables take ~7 KB)
__global__ void __launch_bounds__(256) im2col_3x3_plane_kernel(ConvShape cs, int64_t ldx, int ppb,
                                                               const int32_t *__restrict__ qmap,
                                                               const uint16_t *__restrict__ in,
                                                               uint16_t *__restrict__ xcol) {
    extern __shared__ __align__(16) uint8_t plane_smem[];
    __shared__ int32_t qrow[kPlaneMaxChannels][9];
    __shared__ int16_t qoff[kPlaneMaxChannels][9];
    __shared__ int8_t nlisted[kPlaneMaxChannels];
    const int H = (int)cs.H, W = (int)cs.W, wp = W + 2, HW = H * W, psz = (H + 2) * wp;
    const int64_t c0 = (int64_t)blockIdx.x * ppb, b = blockIdx.y;
    const int np = (int)min((int64_t)ppb, cs.C - c0);
    uint16_t *planes = reinterpret_cast<uint16_t *>(plane_smem);
    for (int ci = threadIdx.x; ci < np; ci += blockDim.x) {
        int n = 0;
        for (int pos = 0; pos < 9; ++pos) {
            const int64_t k = (c0 + ci) * 9 + pos;
            const int32_t q = qmap ? qmap[k] : (int32_t)k;
            if (q >= 0) {
                qrow[ci][n] = q;
                qoff[ci][n] = (int16_t)((pos / 3) * wp + pos % 3);
                ++n;
            }
        }
        nlisted[ci] = (int8_t)n;
    }
    // zero borders, then the planes (16-byte loads: H*W is a multiple of 8 and
    // each plane starts 16-byte aligned when the input does)
    for (int e = threadIdx.x; e < np * psz; e += blockDim.x) planes[e] = 0;
    __syncthreads();
    const int G = HW / 8;
    const uint4 *src = reinterpret_cast<const uint4 *>(in + (b * cs.C + c0) * (int64_t)HW);
    for (int t = threadIdx.x; t < np * G; t += blockDim.x) {
        const int ci = t / G, v = t - ci * G;
        const uint4 q = __ldg(src + (int64_t)ci * G + v);
        const uint32_t w[4] = {q.x, q.y, q.z, q.w};
        uint16_t *pl = planes + ci * psz;
        int p = v * 8, ih = p / W, iw = p - ih * W;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            pl[(ih + 1) * wp + iw + 1] = (uint16_t)(w[e >> 1] >> (16 * (e & 1)));
            if (++iw == W) {
                iw = 0;
                ++ih;
            }
        }
    }
    __syncthreads();
    uint16_t *dst = xcol + b * (int64_t)HW;
    for (int t = threadIdx.x; t < np * G; t += blockDim.x) {
        const int ci = t / G, g = t - ci * G;
        int off[8];
        int p = g * 8, oh = p / W, ow = p - oh * W;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            off[e] = oh * wp + ow;
            if (++ow == W) {
                ow = 0;
                ++oh;
            }
        }
        const uint16_t *pl0 = planes + ci * psz;
        const int L = nlisted[ci];
        for (int l = 0; l < L; ++l) {
            const uint16_t *pl = pl0 + qoff[ci][l];
            uint32_t v[4];
#pragma unroll
            for (int e = 0; e < 4; ++e)
                v[e] = (uint32_t)pl[off[2 * e]] | ((uint32_t)pl[off[2 * e + 1]] << 16);
            *reinterpret_cast<uint4 *>(dst + (int64_t)qrow[ci][l] * ldx + 8 * g) =
                make_uint4(v[0], v[1], v[2], v[3]);
        }
    }
}

// im2col of a 3x3, stride-1, padding-1 convolution whose H*W is not a
// multiple of 8: one block per (group of ppb channels, group of ig images),
// ig * H*W a multiple of 8 so that every block's columns start 16-byte
// aligned.  The block stages the zero-bordered planes [channel][image] in
// shared memory (one warp per plane, 2-byte loads: planes are not 16-byte
// aligned), then each thread writes 8 consecutive columns of a channel's
// listed rows with one 16-byte store; the 8 columns may span two images of
// the group.  Columns of the last group past N are written as zeros (inside
// the row's ldx).
__global__ void __launch_bounds__(256) im2col_3x3_images_kernel(ConvShape cs, int64_t ldx, int ppb,
                                                                int ig,
                                                                const int32_t *__restrict__ qmap,
                                                                const uint16_t *__restrict__ in,
                                                                uint16_t *__restrict__ xcol) {
    extern __shared__ __align__(16) uint8_t plane_smem[];
    __shared__ int32_t qrow[kPlaneMaxChannels][9];
    __shared__ int16_t qoff[kPlaneMaxChannels][9];
    __shared__ int8_t nlisted[kPlaneMaxChannels];
    const int H = (int)cs.H, W = (int)cs.W, wp = W + 2, HW = H * W, psz = (H + 2) * wp;
    const int64_t c0 = (int64_t)blockIdx.x * ppb, b0 = (int64_t)blockIdx.y * ig;
    const int np = (int)min((int64_t)ppb, cs.C - c0);
    const int ni = (int)min((int64_t)ig, cs.Nb - b0);       // images of this block
    uint16_t *planes = reinterpret_cast<uint16_t *>(plane_smem);   // [np][ig][psz]
    for (int ci = threadIdx.x; ci < np; ci += blockDim.x) {
        int n = 0;
        for (int pos = 0; pos < 9; ++pos) {
            const int64_t k = (c0 + ci) * 9 + pos;
            const int32_t q = qmap ? qmap[k] : (int32_t)k;
            if (q >= 0) {
                qrow[ci][n] = q;
                qoff[ci][n] = (int16_t)((pos / 3) * wp + pos % 3);
                ++n;
            }
        }
        nlisted[ci] = (int8_t)n;
    }
    for (int e = threadIdx.x; e < np * ig * psz; e += blockDim.x) planes[e] = 0;
    __syncthreads();
    // interiors: one warp per (channel, image) plane, lanes along its pixels;
    // (ih, iw) advance by 32 pixels per step (one conditional carry: the
    // column step 32 mod W is below W)
    const int per_ch = ni * HW;
    {
        const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
        const int dq = 32 / W, dr = 32 - dq * W, lq = lane / W, lr = lane - lq * W;
        for (int pl = warp; pl < np * ni; pl += nw) {
            const int ci = pl / ni, bi = pl - ci * ni;
            const uint16_t *src = in + ((b0 + bi) * cs.C + c0 + ci) * (int64_t)HW;
            uint16_t *pd = planes + (ci * ig + bi) * psz + wp + 1;
            int ih = lq, iw = lr;
            for (int p = lane; p < HW; p += 32) {
                pd[ih * wp + iw] = __ldg(src + p);
                ih += dq;
                iw += dr;
                if (iw >= W) {
                    iw -= W;
                    ++ih;
                }
            }
        }
    }
    __syncthreads();
    const int G = (per_ch + 7) / 8;                  // 8-column groups per channel row
    uint16_t *dst = xcol + b0 * (int64_t)HW;
    for (int t = threadIdx.x; t < np * G; t += blockDim.x) {
        const int ci = t / G, g = t - ci * G;
        int off[8];
        int lc = g * 8, bi = lc / HW, p = lc - bi * HW, oh = p / W, ow = p - oh * W;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            off[e] = lc + e < per_ch ? (ci * ig + bi) * psz + oh * wp + ow : -1;
            if (++ow == W) {
                ow = 0;
                if (++oh == H) {
                    oh = 0;
                    ++bi;
                }
            }
        }
        const int L = nlisted[ci];
        for (int l = 0; l < L; ++l) {
            const int qo = qoff[ci][l];
            uint32_t v[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const uint32_t lo = off[2 * e] >= 0 ? planes[off[2 * e] + qo] : 0u;
                const uint32_t hi = off[2 * e + 1] >= 0 ? planes[off[2 * e + 1] + qo] : 0u;
                v[e] = lo | (hi << 16);
            }
            *reinterpret_cast<uint4 *>(dst + (int64_t)qrow[ci][l] * ldx + 8 * g) =
                make_uint4(v[0], v[1], v[2], v[3]);
        }
    }
}

// Writes the block's im2col rows from the staged planes: segments of 32*V
// consecutive pixels of one channel per warp step, V pixels per lane (one
// 2V-byte store per window offset).  KH, KW > 0: the window's size at compile
// time (loops unrolled); 0: taken from kh, kw.  qtab: the im2col row of each
// (channel of the block, i, j), -1 for rows no slab lists.
template <int V, int KH, int KW>
__device__ __forceinline__ void im2col_emit(const uint16_t *plane, const int32_t *tab,
                                            const int32_t *qtab, uint16_t *out, int64_t ldx,
                                            int PB, int ncg, int chan_sz, int kh_rt, int kw_rt,
                                            int wp, int lane, int warp, int nwarps) {
    const int kh = KH > 0 ? KH : kh_rt, kw = KW > 0 ? KW : kw_rt;
    const int khw = kh * kw;
    const int segs = (PB + 32 * V - 1) / (32 * V);
    int cc = 0, sg = warp;
    while (sg >= segs) { sg -= segs; ++cc; }
    for (; cc < ncg;) {
        const int p = (sg * 32 + lane) * V;
        if (p < PB) {
            const uint16_t *pl = plane + cc * chan_sz;
            int o0[V];
#pragma unroll
            for (int e = 0; e < V; ++e) o0[e] = tab[p + e];
            const int32_t *qc = qtab + cc * khw;
            uint16_t *op = out + p;
#pragma unroll (KH > 0 ? KH : 1)
            for (int i = 0; i < kh; ++i) {
#pragma unroll (KW > 0 ? KW : 1)
                for (int j = 0; j < kw; ++j) {
                    const int q = qc[i * kw + j];
                    if (q < 0) continue;
                    const int o = i * wp + j;
                    uint32_t v[(V + 1) / 2];
#pragma unroll
                    for (int e = 0; e < V; e += 2) {
                        const uint32_t lo = pl[o0[e] + o];
                        const uint32_t hi = e + 1 < V ? (uint32_t)pl[o0[e + 1] + o] : 0u;
                        v[e / 2] = lo | (hi << 16);
                    }
                    uint16_t *dst = op + (int64_t)q * ldx;
                    if constexpr (V == 1) *dst = (uint16_t)v[0];
                    else if constexpr (V == 2) *reinterpret_cast<uint32_t *>(dst) = v[0];
                    else if constexpr (V == 4) *reinterpret_cast<uint2 *>(dst) = make_uint2(v[0], v[1]);
                    else *reinterpret_cast<uint4 *>(dst) = make_uint4(v[0], v[1], v[2], v[3]);
                }
            }
        }
        sg += nwarps;
        while (sg >= segs) { sg -= segs; ++cc; }
    }
}

// Picks the pixels per lane (alignment of the block's first im2col column and
// pixel count) and the window specialisation.
template <int KH, int KW>
__device__ __forceinline__ void im2col_emit_any(int64_t nbase, const uint16_t *plane,
                                                const int32_t *tab, const int32_t *qtab,
                                                uint16_t *out, int64_t ldx, int PB, int ncg,
                                                int chan_sz, int kh, int kw, int wp, int lane,
                                                int warp, int nwarps) {
    if (nbase % 8 == 0 && PB % 8 == 0)
        im2col_emit<8, KH, KW>(plane, tab, qtab, out, ldx, PB, ncg, chan_sz, kh, kw, wp, lane, warp, nwarps);
    else if (nbase % 4 == 0 && PB % 4 == 0)
        im2col_emit<4, KH, KW>(plane, tab, qtab, out, ldx, PB, ncg, chan_sz, kh, kw, wp, lane, warp, nwarps);
    else if (nbase % 2 == 0 && PB % 2 == 0)
        im2col_emit<2, KH, KW>(plane, tab, qtab, out, ldx, PB, ncg, chan_sz, kh, kw, wp, lane, warp, nwarps);
    else
        im2col_emit<1, KH, KW>(plane, tab, qtab, out, ldx, PB, ncg, chan_sz, kh, kw, wp, lane, warp, nwarps);
}

// im2col, one block per (group of cg channels, group of ig images, band of
// output rows; ig > 1 only when the band is the whole image).  The band's
// input rows of each (channel, image) are staged in shared memory with pw zero
// columns on either side (rows outside the image are zero too), so the window
// reads need no bounds checks; a table gives each of the block's output pixels
// (image-major: consecutive columns of the im2col matrix) its window's offset
// in the staged planes.  Then each warp takes 32 consecutive output pixels of
// one channel and writes them to the kh*kw rows that channel feeds:
// conflict-free shared-memory reads, 64-byte coalesced stores, no division
// per element.  Each input element is read from global memory once per band.
__global__ void __launch_bounds__(256) im2col_kernel(ConvShape cs, int64_t ldx, int band_rows,
                                                     int wp, int cg, int ig,
                                                     const int32_t *__restrict__ qmap,
                                                     const uint16_t *__restrict__ in,
                                                     uint16_t *__restrict__ xcol) {
    extern __shared__ __align__(16) uint8_t im2col_smem[];
    const int C = (int)cs.C, H = (int)cs.H, W = (int)cs.W, Ho = (int)cs.Ho, Wo = (int)cs.Wo;
    const int c0 = blockIdx.x * cg, b0 = blockIdx.y * ig;
    const int ncg = min(cg, C - c0), nig = min(ig, (int)cs.Nb - b0);
    const int oh0 = blockIdx.z * band_rows;
    const int R = min(Ho, oh0 + band_rows) - oh0;
    const int ih0 = oh0 * cs.sh - cs.ph;
    const int rows = (R - 1) * cs.sh + cs.kh;
    const int P = R * Wo;                      // the band's pixels per (channel, image)
    const int PB = nig * P;                    // the block's pixels per channel
    const int plane_sz = rows * wp;            // staged values per (channel, image)
    const int khw = cs.kh * cs.kw;
    int32_t *tab = reinterpret_cast<int32_t *>(im2col_smem);
    int32_t *qtab = tab + ig * P;
    uint16_t *plane =
        reinterpret_cast<uint16_t *>(im2col_smem + ((4 * (ig * P + cg * khw) + 15) & ~15));
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
    // stage: the staged rows (channel, image, row) are spread over the warps,
    // `lpr` lanes per row (a power of two, 32 for rows longer than 32 values),
    // so short rows still keep every lane busy; each lane walks its rows with
    // increments only and keeps 4 loads in flight
    {
        int lpr = 32;
        while (lpr > 1 && lpr / 2 >= wp) lpr >>= 1;
        const int rpw = 32 / lpr;                       // rows per warp step
        const int lr = lane / lpr, lx = lane - lr * lpr;
        const int step = nwarps * rpw;                  // rows per block step
        const int total = ncg * nig * rows;
        int first = warp * rpw + lr;
        // (cc, bb, r) of row index `first`, by division once
        int r = first % rows, ci = first / rows;
        int bb = ci % nig, cc = ci / nig;
        const int dr = step % rows, dci = step / rows;
        for (int row = first; row < total;) {
            int rr[4], rb[4], rc[4];
            bool ok[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                ok[q] = row < total;
                rr[q] = r; rb[q] = bb; rc[q] = cc;
                row += step;
                r += dr;
                int carry = dci;
                if (r >= rows) { r -= rows; ++carry; }
                bb += carry;
                while (bb >= nig) { bb -= nig; ++cc; }
            }
            for (int x0 = lx; x0 < wp; x0 += lpr) {
                uint16_t v[4];
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const int ih = ih0 + rr[q], iw = x0 - cs.pw;
                    v[q] = (ok[q] && (unsigned)ih < (unsigned)H && (unsigned)iw < (unsigned)W)
                               ? __ldg(in + (((int64_t)(b0 + rb[q]) * C + c0 + rc[q]) * H + ih) * W + iw)
                               : (uint16_t)0;
                }
#pragma unroll
                for (int q = 0; q < 4; ++q)
                    if (ok[q]) plane[(rc[q] * ig + rb[q]) * plane_sz + rr[q] * wp + x0] = v[q];
            }
        }
    }
    // pixel table: warps over (image, output row), lanes along the row
    for (int br = warp; br < nig * R; br += nwarps) {
        const int bb = br / R, orow = br - bb * R;
        const int base = bb * plane_sz + orow * cs.sh * wp;
        for (int ow = lane; ow < Wo; ow += 32) tab[bb * P + orow * Wo + ow] = base + ow * cs.sw;
    }
    // im2col row of each (channel, i, j) of the block: qmap[k], or k itself
    for (int e = threadIdx.x; e < ncg * khw; e += blockDim.x) {
        const int64_t k = (int64_t)c0 * khw + e;
        qtab[e] = qmap ? qmap[k] : (int32_t)k;
    }
    __syncthreads();
    const int64_t nbase = (int64_t)b0 * Ho * Wo + (int64_t)oh0 * Wo;
    uint16_t *out = xcol + nbase;
    const int chan_sz = ig * plane_sz;
    if (cs.kh == 3 && cs.kw == 3)
        im2col_emit_any<3, 3>(nbase, plane, tab, qtab, out, ldx, PB, ncg, chan_sz, 3, 3, wp, lane,
                              warp, nwarps);
    else
        im2col_emit_any<0, 0>(nbase, plane, tab, qtab, out, ldx, PB, ncg, chan_sz, cs.kh, cs.kw, wp,
                              lane, warp, nwarps);
}

}  // namespace

cudaError_t launch_rb_counts(const bp_layout &lay, const uint8_t *mask, int64_t *rb_ptr, int *bad,
                             cudaStream_t s) {
    const int64_t RB = (lay.M + lay.bm - 1) / lay.bm;
    cudaError_t e = cudaMemsetAsync(rb_ptr + RB, 0, sizeof(int64_t), s);
    if (e != cudaSuccess) return e;
    rb_counts_kernel<<<(unsigned)RB, 256, 0, s>>>(lay.M, lay.K, lay.bm, mask, rb_ptr, bad);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    exclusive_scan_kernel<<<1, kScanThreads, 0, s>>>(RB + 1, rb_ptr);
    return cudaGetLastError();
}

cudaError_t launch_slab_counts(const bp_layout &lay, const uint8_t *mask, int64_t *info,
                               cudaStream_t s) {
    const int64_t S = (lay.M + kSlab - 1) / kSlab;
    slab_counts_kernel<<<(unsigned)S, 256, 0, s>>>(lay.M, lay.K, lay.bm, mask, info);
    return cudaGetLastError();
}

// ---------------------------------------------------------------- section 3
// K-group q of a layer (list order: q = pos * C64 + c64, pos = i * kw + j):
// does any row of slab s keep any of its 64 columns?  (The first row of each
// row-block the slab touches decides: rows of a row-block are identical.)
__device__ __forceinline__ bool kg_listed(const uint8_t *__restrict__ mask, int64_t M, int64_t K,
                                          int64_t bm, int khw, int64_t C, int64_t C64, int64_t s,
                                          int64_t q) {
    const int64_t pos = q / C64, c64 = q - pos * C64;
    const int64_t r0 = s * kSlab, r1 = min(r0 + kSlab, M);
    const int64_t ce = min(C, 64 * c64 + 64);
    for (int64_t rb = r0 / bm; rb * bm < r1; ++rb) {
        const uint8_t *row = mask + rb * bm * K;
        for (int64_t c = 64 * c64; c < ce; ++c)
            if (row[c * khw + pos]) return true;
    }
    return false;
}

// One block per slab: its chunk count (listed K-groups).
__global__ void kg_counts_kernel(int64_t M, int64_t K, int64_t bm, int khw, int64_t C,
                                 int64_t C64, const uint8_t *__restrict__ mask,
                                 int64_t *__restrict__ counts) {
    const int64_t s = blockIdx.x, KG = C64 * khw;
    int n = 0;
    for (int64_t q = threadIdx.x; q < KG; q += blockDim.x)
        n += kg_listed(mask, M, K, bm, khw, C, C64, s, q) ? 1 : 0;
    __shared__ int tot;
    if (threadIdx.x == 0) tot = 0;
    __syncthreads();
    atomicAdd(&tot, n);
    __syncthreads();
    if (threadIdx.x == 0) counts[s] = tot;
}

// One block (256 threads) per slab: the records of its chunks, the listed
// K-groups in list order (block-wide ordered compaction).
__global__ void __launch_bounds__(256) kg_lists_kernel(int64_t M, int64_t K, int64_t bm, int khw,
                                                       int kw, int64_t C, int64_t C64,
                                                       const uint8_t *__restrict__ mask,
                                                       const int64_t *__restrict__ kc3,
                                                       uint8_t *__restrict__ meta3) {
    const int64_t s = blockIdx.x, KG = C64 * khw;
    const int64_t c0 = kc3[s];
    if (kc3[s + 1] == c0) return;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    __shared__ int wsum[8];
    int64_t running = 0;
    for (int64_t q0 = 0; q0 < KG; q0 += 256) {
        const int64_t q = q0 + threadIdx.x;
        const bool f = q < KG && kg_listed(mask, M, K, bm, khw, C, C64, s, q);
        const unsigned b = __ballot_sync(0xffffffffu, f);
        if (lane == 0) wsum[warp] = __popc(b);
        __syncthreads();
        int before = 0, total = 0;
        for (int w = 0; w < 8; ++w) {
            if (w < warp) before += wsum[w];
            total += wsum[w];
        }
        if (f) {
            const int64_t pos = q / C64, c64 = q - pos * C64;
            const int64_t e = running + before + __popc(b & ((1u << lane) - 1u));
            int32_t *r = reinterpret_cast<int32_t *>(meta3 + (c0 + e) * kMetaBytes);
            r[0] = (int32_t)((c64 << 16) | ((pos / kw) << 8) | (pos % kw));
            r[kListBytes / 4] = 1;
        }
        running += total;
        __syncthreads();
    }
}

// One thread per 16-byte unit (row, 8 channels) of a chunk's weight tile.
__global__ void kg_tiles_kernel(int64_t M, int64_t K, int khw, int kw, int64_t C,
                                const uint16_t *__restrict__ W, const uint8_t *__restrict__ mask,
                                const int64_t *__restrict__ kc3, uint8_t *__restrict__ tiles3,
                                const uint8_t *__restrict__ meta3) {
    const int64_t s = blockIdx.y;
    const int64_t c0 = kc3[s], nkc = kc3[s + 1] - c0;
    const int64_t units = nkc * kSlab * 8;
    for (int64_t u = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; u < units;
         u += (int64_t)gridDim.x * blockDim.x) {
        const int64_t kc = u / (kSlab * 8);
        const int64_t rem = u - kc * (kSlab * 8);
        const uint32_t row = (uint32_t)(rem >> 3), ch = (uint32_t)(rem & 7);
        const int32_t d = reinterpret_cast<const int32_t *>(meta3 + (c0 + kc) * kMetaBytes)[0];
        const int64_t c64 = d >> 16, pos = ((d >> 8) & 0xff) * kw + (d & 0xff);
        const int64_t r = s * kSlab + row;
        uint16_t v[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const int64_t c = 64 * c64 + 8 * ch + e;
            const int64_t k = c * khw + pos;
            v[e] = (r < M && c < C && mask[r * K + k]) ? W[r * K + k] : (uint16_t)0;
        }
        uint4 pk;
        pk.x = v[0] | ((uint32_t)v[1] << 16);
        pk.y = v[2] | ((uint32_t)v[3] << 16);
        pk.z = v[4] | ((uint32_t)v[5] << 16);
        pk.w = v[6] | ((uint32_t)v[7] << 16);
        *reinterpret_cast<uint4 *>(tiles3 + (c0 + kc) * (int64_t)(kSlab * kBK * 2) +
                                   sw128_kmajor_offset(row, ch * 8)) = pk;
    }
}

// NCHW -> NHWC with channels padded to a multiple of 8 (zeros): one block per
// (image, 64 consecutive pixels, 64 channels).  Each channel's 64 pixels are
// 128 contiguous bytes of the input, each pixel's 64 channels 128 contiguous
// bytes of the output; the transposition goes through shared memory.
__global__ void __launch_bounds__(256) nhwc8_kernel(ConvShape cs, const uint16_t *__restrict__ in,
                                                    uint16_t *__restrict__ out) {
    const int64_t HW = cs.H * cs.W, C8 = (cs.C + 7) / 8 * 8;
    const int64_t b = blockIdx.z, p0 = (int64_t)blockIdx.x * 64, c0 = (int64_t)blockIdx.y * 64;
    __shared__ uint16_t tile[64][66];           // [channel][pixel] (+2 against bank conflicts)
    const int np = (int)min((int64_t)64, HW - p0), nc = (int)min((int64_t)64, C8 - c0);
    const bool vec = HW % 8 == 0;               // channel planes start 16-byte aligned
    // 64 channels x 64 pixels, 8 pixels per thread and pass
    for (int e = threadIdx.x; e < 64 * 8; e += blockDim.x) {
        const int cc = e >> 3, q = (e & 7) * 8;
        const int64_t c = c0 + cc;
        uint16_t v[8];
        if (c < cs.C && q < np) {
            const uint16_t *src = in + (b * cs.C + c) * HW + p0 + q;
            if (vec && q + 8 <= np) {
                const uint4 w = *reinterpret_cast<const uint4 *>(src);
                v[0] = (uint16_t)w.x; v[1] = (uint16_t)(w.x >> 16);
                v[2] = (uint16_t)w.y; v[3] = (uint16_t)(w.y >> 16);
                v[4] = (uint16_t)w.z; v[5] = (uint16_t)(w.z >> 16);
                v[6] = (uint16_t)w.w; v[7] = (uint16_t)(w.w >> 16);
            } else {
#pragma unroll
                for (int u = 0; u < 8; ++u) v[u] = q + u < np ? src[u] : (uint16_t)0;
            }
        } else {
#pragma unroll
            for (int u = 0; u < 8; ++u) v[u] = 0;
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) tile[cc][q + u] = v[u];
    }
    __syncthreads();
    // each pixel's channels c0 .. c0 + nc - 1, 8 per 16-byte store
    const int ng = nc / 8;
    for (int e = threadIdx.x; e < np * ng; e += blockDim.x) {
        const int px = e / ng, g = e - px * ng;
        uint16_t v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) v[u] = tile[g * 8 + u][px];
        uint4 pk;
        pk.x = v[0] | ((uint32_t)v[1] << 16);
        pk.y = v[2] | ((uint32_t)v[3] << 16);
        pk.z = v[4] | ((uint32_t)v[5] << 16);
        pk.w = v[6] | ((uint32_t)v[7] << 16);
        *reinterpret_cast<uint4 *>(out + (b * HW + p0 + px) * C8 + c0 + g * 8) = pk;
    }
}

cudaError_t launch_pack_sec3(const bp_layout &lay, const void *W, const uint8_t *mask,
                             const bp_packed &P, const DevLayout &dl, int64_t *scratch,
                             cudaStream_t s) {
    if (dl.c3max == 0) return cudaSuccess;
    const int khw = lay.kh * lay.kw;
    const int64_t C = lay.K / khw, C64 = (C + 63) / 64;
    const int64_t S = dl.num_slabs;
    uint8_t *dev = static_cast<uint8_t *>(P.dev);
    int64_t *kc3 = reinterpret_cast<int64_t *>(dev + dl.off_sec3);
    cudaError_t e = cudaMemsetAsync(scratch, 0, 8 * (S + 1), s);
    if (e != cudaSuccess) return e;
    kg_counts_kernel<<<(unsigned)S, 256, 0, s>>>(lay.M, lay.K, lay.bm, khw, C, C64, mask, scratch);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    exclusive_scan_kernel<<<1, kScanThreads, 0, s>>>(S + 1, scratch);
    e = cudaGetLastError();
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(kc3, scratch, 8 * (S + 1), cudaMemcpyDeviceToDevice, s);
    if (e != cudaSuccess) return e;
    uint8_t *meta3 = dev + dl.off_meta3;
    kg_lists_kernel<<<(unsigned)S, 256, 0, s>>>(lay.M, lay.K, lay.bm, khw, lay.kw, C, C64, mask,
                                                 kc3, meta3);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    dim3 grid(16, (unsigned)S);
    kg_tiles_kernel<<<grid, 256, 0, s>>>(lay.M, lay.K, khw, lay.kw, C,
                                         static_cast<const uint16_t *>(W), mask, kc3,
                                         dev + dl.off_tiles3, meta3);
    return cudaGetLastError();
}

// Stride-2 layers: the input split into its four phases (even / odd rows x
// even / odd columns), each an NHWC image of ceil(H/2) x ceil(W/2) pixels and
// C8 channels.  Phase (a, c) of image b is image (2a + c) * Nb + b of the
// output and holds input pixel (2h + a, 2w + c) at (h, w), zero past the
// input's edge.  A stride-2 window then reads, for each kernel position, one
// phase at a unit-stride offset.  One block: 64 channels x one input row
// pair x 64 input columns through shared memory.
__global__ void __launch_bounds__(256) nhwc8_phase_kernel(ConvShape cs, int64_t xchunks,
                                                          const uint16_t *__restrict__ in,
                                                          uint16_t *__restrict__ out) {
    const int64_t H2 = (cs.H + 1) / 2, W2 = (cs.W + 1) / 2, C8 = (cs.C + 7) / 8 * 8;
    const int64_t b = blockIdx.z, c0 = (int64_t)blockIdx.y * 64;
    const int64_t r = blockIdx.x / xchunks, w0 = (blockIdx.x % xchunks) * 64;
    __shared__ uint16_t tile[64][2][66];        // [channel][row of the pair][column] (+2 pad)
    const bool vec = cs.W % 8 == 0;             // input rows start 16-byte aligned
    // 64 channels x 2 rows x 64 columns, 8 columns per thread and pass
    for (int v = threadIdx.x; v < 64 * 2 * 8; v += blockDim.x) {
        const int ch = v >> 4, row = (v >> 3) & 1, cq = (v & 7) * 8;
        const int64_t c = c0 + ch, h = 2 * r + row, w = w0 + cq;
        uint16_t e[8];
        if (c < cs.C && h < cs.H && w < cs.W) {
            const uint16_t *src = in + ((b * cs.C + c) * cs.H + h) * cs.W + w;
            if (vec && w + 8 <= cs.W) {
                const uint4 q = *reinterpret_cast<const uint4 *>(src);
                e[0] = (uint16_t)q.x; e[1] = (uint16_t)(q.x >> 16);
                e[2] = (uint16_t)q.y; e[3] = (uint16_t)(q.y >> 16);
                e[4] = (uint16_t)q.z; e[5] = (uint16_t)(q.z >> 16);
                e[6] = (uint16_t)q.w; e[7] = (uint16_t)(q.w >> 16);
            } else {
#pragma unroll
                for (int u = 0; u < 8; ++u) e[u] = w + u < cs.W ? src[u] : (uint16_t)0;
            }
        } else {
#pragma unroll
            for (int u = 0; u < 8; ++u) e[u] = 0;
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) tile[ch][row][cq + u] = e[u];
    }
    __syncthreads();
    // 4 phases x 32 phase columns x 8 groups of 8 channels, one 16-byte store each
    for (int v = threadIdx.x; v < 4 * 32 * 8; v += blockDim.x) {
        const int ph = v >> 8, j = (v >> 3) & 31, g = v & 7;
        const int a = ph >> 1, cp = ph & 1;
        const int64_t w2 = w0 / 2 + j;
        if (w2 >= W2 || c0 + g * 8 >= C8) continue;
        uint16_t e[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) e[u] = tile[g * 8 + u][a][2 * j + cp];
        uint4 pk;
        pk.x = e[0] | ((uint32_t)e[1] << 16);
        pk.y = e[2] | ((uint32_t)e[3] << 16);
        pk.z = e[4] | ((uint32_t)e[5] << 16);
        pk.w = e[6] | ((uint32_t)e[7] << 16);
        *reinterpret_cast<uint4 *>(out + ((((int64_t)ph * cs.Nb + b) * H2 + r) * W2 + w2) * C8 +
                                   c0 + g * 8) = pk;
    }
}

cudaError_t launch_nhwc8(const ConvShape &cs, const void *in, void *out, cudaStream_t s) {
    const int64_t HW = cs.H * cs.W, C8 = (cs.C + 7) / 8 * 8;
    if (cs.Nb * HW == 0) return cudaSuccess;
    if (cs.sh == 2) {
        const int64_t H2 = (cs.H + 1) / 2, xchunks = (cs.W + 63) / 64;
        const dim3 grid((unsigned)(H2 * xchunks), (unsigned)((C8 + 63) / 64), (unsigned)cs.Nb);
        nhwc8_phase_kernel<<<grid, 256, 0, s>>>(cs, xchunks, static_cast<const uint16_t *>(in),
                                                static_cast<uint16_t *>(out));
        return cudaGetLastError();
    }
    const dim3 grid((unsigned)((HW + 63) / 64), (unsigned)((C8 + 63) / 64), (unsigned)cs.Nb);
    nhwc8_kernel<<<grid, 256, 0, s>>>(cs, static_cast<const uint16_t *>(in),
                                      static_cast<uint16_t *>(out));
    return cudaGetLastError();
}

cudaError_t launch_pack(const bp_layout &lay, const void *W, const uint8_t *mask,
                        const bp_packed &P, const DevLayout &dl, cudaStream_t s) {
    const int64_t RB = P.num_rb;
    col_idx_kernel<<<(unsigned)RB, kScanThreads, 0, s>>>(lay.K, lay.bm, mask, P.rb_ptr,
                                                         P.col_idx);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    values_kernel<<<(unsigned)RB, 256, 0, s>>>(lay.M, lay.K, lay.bm,
                                               static_cast<const uint16_t *>(W), P.rb_ptr,
                                               P.col_idx, static_cast<uint16_t *>(P.values));
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    uint8_t *dev = static_cast<uint8_t *>(P.dev);
    if (dl.kc_total == 0)   // nothing listed: no im2col row is needed
        return cudaMemsetAsync(dev + dl.off_qmap, 0xff, 4 * lay.K, s);
    const int64_t *kc_ptr = reinterpret_cast<const int64_t *>(dev);
    uint8_t *tiles = dev + dl.off_tiles;
    uint8_t *meta = dev + dl.off_meta;
    uint8_t *meta2 = dev + dl.off_meta2;
    int32_t *qmap = reinterpret_cast<int32_t *>(dev + dl.off_qmap);
    int64_t *kc_hdr = reinterpret_cast<int64_t *>(dev) + dl.num_slabs + 1;
    slab_lists_kernel<<<(unsigned)dl.num_slabs, 32, 0, s>>>(lay.M, lay.K, lay.bm, mask, kc_ptr,
                                                           meta);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    const int64_t entries = dl.kc_total * kBK;
    int64_t eblocks = (entries + 255) / 256;
    if (eblocks > 4096) eblocks = 4096;
    e = cudaMemsetAsync(qmap, 0, 4 * lay.K, s);
    if (e != cudaSuccess) return e;
    mark_listed_kernel<<<(unsigned)eblocks, 256, 0, s>>>(entries, meta, qmap);
    qmap_scan_kernel<<<1, 1024, 0, s>>>(lay.K, qmap, kc_hdr);
    compact_lists_kernel<<<(unsigned)eblocks, 256, 0, s>>>(entries, meta, meta2, qmap);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    int64_t pblocks = (dl.kc_total + 127) / 128;
    if (pblocks > 1024) pblocks = 1024;
    plans_kernel<<<(unsigned)pblocks, 128, 0, s>>>(dl.kc_total, meta, nullptr);
    plans_kernel<<<(unsigned)pblocks, 128, 0, s>>>(dl.kc_total, meta2, kc_hdr);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    dim3 grid(16, (unsigned)dl.num_slabs);
    tiles_kernel<<<grid, 256, 0, s>>>(lay.M, lay.K, static_cast<const uint16_t *>(W), mask, kc_ptr,
                                      tiles, meta, dl.tile_bytes);
    return cudaGetLastError();
}

int64_t im2col_row_width(const ConvShape &cs) {
    // staged row: pw zeros, W values, pw zeros (window reads stay inside:
    // (Wo - 1) * sw + kw - 1 <= W + 2 pw - 1)
    return cs.W + 2 * cs.pw;
}

static bool rows_kernel_ok(const ConvShape &cs, int64_t ldx, const void *xcol) {
    return ldx % 8 == 0 && (reinterpret_cast<uintptr_t>(xcol) & 15u) == 0 &&
           cs.C * cs.kh * cs.kw <= 65535 && cs.Nb * cs.Ho * cs.Wo <= 0x7fffffffLL - 8;
}

static cudaError_t launch_im2col_rows(const ConvShape &cs, int64_t ldx, const void *in, void *xcol,
                                      const int32_t *qmap, cudaStream_t s) {
    const int64_t gx = (cs.Nb * cs.Ho * cs.Wo + 2047) / 2048;
    const dim3 grid((unsigned)gx, (unsigned)(cs.C * cs.kh * cs.kw));
    if (cs.kh == 1 && cs.kw == 1)
        im2col_rows_kernel<true><<<grid, 256, 0, s>>>(cs, ldx, qmap,
                                                      static_cast<const uint16_t *>(in),
                                                      static_cast<uint16_t *>(xcol));
    else
        im2col_rows_kernel<false><<<grid, 256, 0, s>>>(cs, ldx, qmap,
                                                       static_cast<const uint16_t *>(in),
                                                       static_cast<uint16_t *>(xcol));
    return cudaGetLastError();
}

cudaError_t launch_im2col(const ConvShape &cs, int64_t ldx, const void *in, void *xcol,
                          const int32_t *qmap, cudaStream_t s) {
    if (cs.kh == 1 && cs.kw == 1 && cs.sh == 1 && cs.sw == 1 && cs.ph == 0 && cs.pw == 0 &&
        (cs.H * cs.W) % 8 == 0 && cs.H * cs.W >= 256) {
        // large planes of 16-byte multiples: one block copies one plane
        if (cs.C > 0x7fffffffLL || cs.Nb > 65535) return cudaErrorInvalidValue;
        im2col_copy_kernel<<<dim3((unsigned)cs.C, (unsigned)cs.Nb), 256, 0, s>>>(
            cs.C, cs.H * cs.W, ldx, qmap, static_cast<const uint16_t *>(in),
            static_cast<uint16_t *>(xcol));
        return cudaGetLastError();
    }
    if (cs.kh == 1 && cs.kw == 1 && rows_kernel_ok(cs, ldx, xcol)) {
        // small or unaligned planes, strided or padded 1x1: threads along the rows
        return launch_im2col_rows(cs, ldx, in, xcol, qmap, s);
    }
    if (cs.kh == 1 && cs.kw == 1) {
        if (cs.C > 0x7fffffffLL || cs.Nb > 65535) return cudaErrorInvalidValue;
        im2col_1x1_kernel<<<dim3((unsigned)cs.C, (unsigned)cs.Nb), 256, 0, s>>>(
            cs, ldx, qmap, static_cast<const uint16_t *>(in), static_cast<uint16_t *>(xcol));
        return cudaGetLastError();
    }
    if (cs.kh == 3 && cs.kw == 3 && cs.sh == 1 && cs.sw == 1 && cs.ph == 1 && cs.pw == 1 &&
        (cs.H * cs.W) % 8 == 0 && (cs.H + 2) * (cs.W + 2) * 2 <= kPlaneSmem && ldx % 8 == 0 &&
        cs.H * cs.W <= 32767 && (reinterpret_cast<uintptr_t>(in) & 15u) == 0 &&
        (reinterpret_cast<uintptr_t>(xcol) & 15u) == 0 && cs.Nb <= 65535) {
        // channels per block: enough pixel groups for the 256 threads, within
        // the shared memory and the per-block channel tables
        const int64_t G = cs.H * cs.W / 8, psz = (cs.H + 2) * (cs.W + 2) * 2;
        int64_t ppb = (256 + G - 1) / G;
        if (ppb > kPlaneMaxChannels) ppb = kPlaneMaxChannels;
        if (ppb > kPlaneSmem / psz) ppb = kPlaneSmem / psz;
        if (ppb > cs.C) ppb = cs.C;
        const int64_t gx = (cs.C + ppb - 1) / ppb;
        if (gx <= 0x7fffffffLL) {
            im2col_3x3_plane_kernel<<<dim3((unsigned)gx, (unsigned)cs.Nb), 256,
                                      (size_t)(ppb * psz), s>>>(
                cs, ldx, (int)ppb, qmap, static_cast<const uint16_t *>(in),
                static_cast<uint16_t *>(xcol));
            return cudaGetLastError();
        }
    }
    if (cs.kh == 3 && cs.kw == 3 && cs.sh == 1 && cs.sw == 1 && cs.ph == 1 && cs.pw == 1 &&
        (cs.H * cs.W) % 8 != 0 && cs.H * cs.W >= 32 && cs.H * cs.W < 256 && ldx % 8 == 0 &&
        (reinterpret_cast<uintptr_t>(xcol) & 15u) == 0) {
        // H*W not a multiple of 8, 32 to 255 pixels (measured on ResNet-50:
        // 7x7 planes 62.3 -> 51.5 us on s4b2_3x3, 14x14 planes even with the
        // banded kernel at 51.5 us; planes under 32 pixels stay faster with the
        // rows kernel):
        // image groups with ig * H*W a multiple of 8, at least ~256 columns
        // per channel row, planes within the stage
        const int64_t HW = cs.H * cs.W, psz = (cs.H + 2) * (cs.W + 2) * 2;
        int64_t ig = 8;
        while (ig > 1 && (HW * (ig / 2)) % 8 == 0) ig /= 2;     // smallest aligned group
        while (ig * HW < 256 && ig * 2 * psz <= kPlaneSmem && ig < cs.Nb) ig *= 2;
        if (ig * psz <= kPlaneSmem) {
            const int64_t gpc = (ig * HW + 7) / 8;               // column groups per channel
            int64_t ppb = (512 + gpc - 1) / gpc;
            if (ppb > kPlaneMaxChannels) ppb = kPlaneMaxChannels;
            if (ppb > kPlaneSmem / (ig * psz)) ppb = kPlaneSmem / (ig * psz);
            if (ppb > cs.C) ppb = cs.C;
            if (ppb < 1) ppb = 1;
            const int64_t gx = (cs.C + ppb - 1) / ppb, gy = (cs.Nb + ig - 1) / ig;
            if (gx <= 0x7fffffffLL && gy <= 65535) {
                im2col_3x3_images_kernel<<<dim3((unsigned)gx, (unsigned)gy), 256,
                                           (size_t)(ppb * ig * psz), s>>>(
                    cs, ldx, (int)ppb, (int)ig, qmap, static_cast<const uint16_t *>(in),
                    static_cast<uint16_t *>(xcol));
                return cudaGetLastError();
            }
        }
    }
    // strided convolutions and planes of fewer than 32 output pixels: threads
    // along the rows (measured faster there: ResNet-50's stride-2 3x3 layers,
    // VGG-16's 2x2 layers); stride-1 layers on larger planes stage the input
    // rows of a band in shared memory once for all kernel positions
    if ((cs.sh != 1 || cs.sw != 1 || cs.Ho * cs.Wo < 32) && rows_kernel_ok(cs, ldx, xcol))
        return launch_im2col_rows(cs, ldx, in, xcol, qmap, s);
    constexpr int64_t kStage = 24 * 1024 / 2;     // staged values per block at most
    constexpr int64_t kTab = 4096;                 // table entries (output pixels) per block at most
    const int64_t wp = im2col_row_width(cs);
    // output rows per block (the band): as many as fit, at least one
    const int64_t max_rows = kStage / wp;
    if (max_rows < cs.kh) return cudaErrorInvalidValue;
    int64_t band = (max_rows - cs.kh) / cs.sh + 1;
    if (band > cs.Ho) band = cs.Ho;
    if (band * cs.Wo > kTab) band = kTab / cs.Wo > 0 ? kTab / cs.Wo : 1;
    const int64_t rows = (band - 1) * cs.sh + cs.kh;
    const int64_t nbands = (cs.Ho + band - 1) / band;
    const int64_t pix = band * cs.Wo;
    // images per block (whole images only): at least about 512 pixels per channel
    int64_t ig = 1;
    if (band == cs.Ho) {
        ig = (512 + pix - 1) / pix;
        if (ig > cs.Nb) ig = cs.Nb;
        if (ig > kTab / pix) ig = kTab / pix;
        if (ig > kStage / (rows * wp)) ig = kStage / (rows * wp);
        if (ig < 1) ig = 1;
    }
    // channels per block: about 2048 output pixels, within the stage
    int64_t cg = (2048 + ig * pix - 1) / (ig * pix);
    if (cg > kStage / (ig * rows * wp)) cg = kStage / (ig * rows * wp);
    if (cg > cs.C) cg = cs.C;
    if (cg < 1) cg = 1;
    auto smem_for = [&](int64_t g) {
        return (size_t)((4 * (ig * pix + g * cs.kh * cs.kw) + 15) & ~15) +
               (size_t)(g * ig * rows * wp * 2);
    };
    while (cg > 1 && smem_for(cg) > 48 * 1024) --cg;
    if (smem_for(cg) > 48 * 1024) return cudaErrorInvalidValue;
    const int64_t gx = (cs.C + cg - 1) / cg, gy = (cs.Nb + ig - 1) / ig;
    if (gx > 0x7fffffffLL || gy > 65535 || nbands > 65535) return cudaErrorInvalidValue;
    const size_t smem = smem_for(cg);
    im2col_kernel<<<dim3((unsigned)gx, (unsigned)gy, (unsigned)nbands), 256, smem, s>>>(
        cs, ldx, (int)band, (int)wp, (int)cg, (int)ig, qmap, static_cast<const uint16_t *>(in),
        static_cast<uint16_t *>(xcol));
    return cudaGetLastError();
}

}  // namespace bp
