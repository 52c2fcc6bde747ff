// Pruning kernels: per-unit squared norms (Eq. column / Eq. punched), the
// per-block keep of floor(P_b / r) best units, and the layer-wide selection of
// the remaining best units (a most-significant-digit radix select on the
// fp64 score bits, ties to the lower unit index), then the element mask.
//
// Units are numbered g = (rb*CB + cb)*P + u for block-punched layers,
// g = rb*K + column for block-based ones, and, for the row units of
// block-based layers, g = rb*bm*CB + cb*rows_rb + (r - rb*bm) (rows_rb = real
// rows of row-block rb: block-major, then row); the numbering is also the tie
// order.

#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "bp_common.cuh"

namespace bp {
namespace {

struct Part {
    int scheme;
    int64_t M, K, KK, C, bm, bk, RB, CB, U;
};

Part make_part(const bp_layout &l) {
    Part p;
    p.scheme = l.scheme;
    p.M = l.M;
    p.K = l.K;
    p.KK = (int64_t)l.kh * l.kw;
    p.C = l.K / p.KK;
    p.bm = l.bm;
    p.bk = l.bk;
    p.RB = (l.M + l.bm - 1) / l.bm;
    if (l.scheme == BP_BLOCK_BASED) {
        p.CB = (l.K + l.bk - 1) / l.bk;
        p.U = p.RB * l.K;
    } else if (l.scheme == kSchemeRows) {
        p.CB = (l.K + l.bk - 1) / l.bk;
        p.U = l.M * p.CB;
    } else if (l.scheme == kSchemePattern) {
        p.CB = p.C;
        p.U = l.M * p.C;
    } else {
        p.CB = (p.C + l.bk - 1) / l.bk;
        p.U = p.RB * p.CB * p.KK;
    }
    return p;
}

// Row unit g of a block-based layer -> (row, column-block), and the first
// unit and size of its block.
struct RowUnit {
    int64_t r, cb, first, P;
};
__device__ __forceinline__ RowUnit row_unit(const Part &p, int64_t g) {
    const int64_t rb = g / (p.bm * p.CB), r0 = rb * p.bm;
    const int64_t rows = min(p.bm, p.M - r0);
    const int64_t rem = g - r0 * p.CB, cb = rem / rows;
    RowUnit u;
    u.r = r0 + (rem - cb * rows);
    u.cb = cb;
    u.first = r0 * p.CB + cb * rows;
    u.P = rows;
    return u;
}

__device__ __forceinline__ float ld_half(const uint16_t *w, int64_t i, int dtype) {
    const uint16_t b = w[i];
    if (dtype == BP_BF16) return __bfloat162float(__ushort_as_bfloat16(b));
    return __half2float(__ushort_as_half(b));
}

// One thread per unit.  Block-based: the column's rows in ascending order;
// block-punched: filters ascending, then channels ascending.
__global__ void scores_kernel(Part p, int dtype, const uint16_t *__restrict__ W,
                              double *__restrict__ scores, int *__restrict__ nonfinite) {
    for (int64_t g = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; g < p.U;
         g += (int64_t)gridDim.x * blockDim.x) {
        double s = 0.0;
        bool bad = false;
        if (p.scheme == BP_BLOCK_BASED) {
            const int64_t rb = g / p.K, j = g % p.K;
            const int64_t r0 = rb * p.bm, r1 = min(r0 + p.bm, p.M);
            for (int64_t r = r0; r < r1; ++r) {
                const float f = ld_half(W, r * p.K + j, dtype);
                bad |= !isfinite(f);
                const double w = (double)f;
                s += w * w;
            }
        } else if (p.scheme == kSchemeRows) {
            // the row's segment in its column-block, columns ascending
            const RowUnit u = row_unit(p, g);
            const int64_t k0 = u.cb * p.bk, k1 = min(k0 + p.bk, p.K);
            for (int64_t k = k0; k < k1; ++k) {
                const float f = ld_half(W, u.r * p.K + k, dtype);
                bad |= !isfinite(f);
                const double w = (double)f;
                s += w * w;
            }
        } else {
            const int64_t pos = g % p.KK, b = g / p.KK;
            const int64_t rb = b / p.CB, cb = b % p.CB;
            const int64_t r0 = rb * p.bm, r1 = min(r0 + p.bm, p.M);
            const int64_t c0 = cb * p.bk, c1 = min(c0 + p.bk, p.C);
            for (int64_t f = r0; f < r1; ++f)
                for (int64_t c = c0; c < c1; ++c) {
                    const float v = ld_half(W, f * p.K + c * p.KK + pos, dtype);
                    bad |= !isfinite(v);
                    const double w = (double)v;
                    s += w * w;
                }
        }
        scores[g] = s;
        if (bad) atomicExch(nonfinite, 1);
    }
}

// keep[g] = 1 for the floor(P_b / rate) best units of each block (rank by
// score descending, then unit index ascending), else 0.
__global__ void base_select_kernel(Part p, double rate, const double *__restrict__ scores,
                                   uint8_t *__restrict__ keep) {
    for (int64_t g = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; g < p.U;
         g += (int64_t)gridDim.x * blockDim.x) {
        int64_t first, P;
        if (p.scheme == BP_BLOCK_BASED) {
            const int64_t rb = g / p.K, j = g % p.K, cb = j / p.bk;
            first = rb * p.K + cb * p.bk;
            P = min(p.bk, p.K - cb * p.bk);
        } else if (p.scheme == kSchemeRows) {
            const RowUnit u = row_unit(p, g);
            first = u.first;
            P = u.P;
        } else if (p.scheme == kSchemePattern) {
            first = g;            // each kernel is a block of one unit
            P = 1;
        } else {
            first = (g / p.KK) * p.KK;
            P = p.KK;
        }
        const int64_t base = (int64_t)floor((double)P / rate);
        const double s = scores[g];
        int64_t rank = 0;
        for (int64_t v = first; v < first + P; ++v) {
            const double t = scores[v];
            rank += (t > s) || (t == s && v < g);
        }
        keep[g] = rank < base ? 1 : 0;
    }
}

__device__ __forceinline__ uint64_t key_of(double s) {
    // scores are sums of squares (>= +0), so their bit patterns order like the values
    return (uint64_t)__double_as_longlong(s);
}

__global__ void radix_hist_kernel(int64_t U, const double *__restrict__ scores,
                                  const uint8_t *__restrict__ keep, uint64_t prefix, int shift,
                                  unsigned *__restrict__ hist) {
    __shared__ unsigned h[256];
    for (int i = threadIdx.x; i < 256; i += blockDim.x) h[i] = 0;
    __syncthreads();
    for (int64_t g = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; g < U;
         g += (int64_t)gridDim.x * blockDim.x) {
        if (keep[g]) continue;
        const uint64_t k = key_of(scores[g]);
        if (shift < 56 && (k >> (shift + 8)) != (prefix >> (shift + 8))) continue;
        atomicAdd(&h[(k >> shift) & 255u], 1u);
    }
    __syncthreads();
    for (int i = threadIdx.x; i < 256; i += blockDim.x)
        if (h[i]) atomicAdd(&hist[i], h[i]);
}

constexpr int kChunk = 4096;      // units per chunk of the ordered tie selection
constexpr int kSelThreads = 1024;

// Candidates above the threshold are kept; candidates equal to it are counted
// per chunk (they are resolved in unit order by the next two kernels).
__global__ void threshold_count_kernel(int64_t U, const double *__restrict__ scores,
                                       uint8_t *__restrict__ keep, uint64_t thr,
                                       int64_t *__restrict__ chunk_cnt) {
    __shared__ int cnt;
    if (threadIdx.x == 0) cnt = 0;
    __syncthreads();
    const int64_t c0 = (int64_t)blockIdx.x * kChunk;
    int local = 0;
    for (int64_t g = c0 + threadIdx.x; g < min(c0 + kChunk, U); g += blockDim.x) {
        if (keep[g]) continue;
        const uint64_t k = key_of(scores[g]);
        if (k > thr) keep[g] = 2;          // extra unit (2 = kept in the second step)
        else if (k == thr) ++local;
    }
    atomicAdd(&cnt, local);
    __syncthreads();
    if (threadIdx.x == 0) chunk_cnt[blockIdx.x] = cnt;
}

// exclusive scan of the chunk counts (one block)
__global__ void scan_chunks_kernel(int64_t n, int64_t *__restrict__ cnt) {
    __shared__ int64_t carry;
    __shared__ int64_t part[kSelThreads];
    if (threadIdx.x == 0) carry = 0;
    __syncthreads();
    for (int64_t base = 0; base < n; base += kSelThreads) {
        const int64_t i = base + threadIdx.x;
        const int64_t v = i < n ? cnt[i] : 0;
        part[threadIdx.x] = v;
        __syncthreads();
        for (int off = 1; off < kSelThreads; off <<= 1) {
            const int64_t t = threadIdx.x >= off ? part[threadIdx.x - off] : 0;
            __syncthreads();
            part[threadIdx.x] += t;
            __syncthreads();
        }
        if (i < n) cnt[i] = carry + part[threadIdx.x] - v;
        __syncthreads();
        if (threadIdx.x == kSelThreads - 1) carry += part[threadIdx.x];
        __syncthreads();
    }
}

// Among candidates equal to the threshold, keep the `need` with the lowest
// unit index: each thread owns kChunk / kSelThreads consecutive units.
__global__ void threshold_ties_kernel(int64_t U, const double *__restrict__ scores,
                                      uint8_t *__restrict__ keep, uint64_t thr, int64_t need,
                                      const int64_t *__restrict__ chunk_off) {
    constexpr int kPer = kChunk / kSelThreads;
    __shared__ int part[kSelThreads];
    const int64_t g0 = (int64_t)blockIdx.x * kChunk + (int64_t)threadIdx.x * kPer;
    bool eq[kPer];
    int mine = 0;
#pragma unroll
    for (int e = 0; e < kPer; ++e) {
        const int64_t g = g0 + e;
        eq[e] = g < U && keep[g] == 0 && key_of(scores[g]) == thr;
        mine += eq[e];
    }
    part[threadIdx.x] = mine;
    __syncthreads();
    for (int off = 1; off < kSelThreads; off <<= 1) {
        const int t = threadIdx.x >= off ? part[threadIdx.x - off] : 0;
        __syncthreads();
        part[threadIdx.x] += t;
        __syncthreads();
    }
    int64_t rank = chunk_off[blockIdx.x] + part[threadIdx.x] - mine;
#pragma unroll
    for (int e = 0; e < kPer; ++e)
        if (eq[e]) {
            if (rank < need) keep[g0 + e] = 2;
            ++rank;
        }
}

__global__ void write_mask_kernel(Part p, const uint8_t *__restrict__ keep,
                                  uint8_t *__restrict__ mask) {
    const int64_t total = p.M * p.K;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = i / p.K, k = i % p.K, rb = r / p.bm;
        int64_t g;
        if (p.scheme == BP_BLOCK_BASED) {
            g = rb * p.K + k;
        } else if (p.scheme == kSchemeRows) {
            // row units are ANDed into the mask already there
            const int64_t r0 = rb * p.bm, rows = min(p.bm, p.M - r0), cb = k / p.bk;
            g = r0 * p.CB + cb * rows + (r - r0);
            if (!keep[g]) mask[i] = 0;
            continue;
        } else {
            const int64_t c = k / p.KK, pos = k % p.KK;
            g = (rb * p.CB + c / p.bk) * p.KK + pos;
        }
        mask[i] = keep[g] ? 1 : 0;
    }
}

// Pattern units: kernel g = f*C + c.  Its squared weights (fp64), the kept
// norm of every pattern (positions ascending), the best pattern (ties to the
// lower index) into patsel and its norm into scores.
__global__ void pattern_scores_kernel(Part p, int dtype, const uint16_t *__restrict__ W,
                                      PatternSet ps, double *__restrict__ scores,
                                      uint8_t *__restrict__ patsel, int *__restrict__ nonfinite) {
    for (int64_t g = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; g < p.U;
         g += (int64_t)gridDim.x * blockDim.x) {
        const int64_t f = g / p.C, c = g - f * p.C;
        const uint16_t *k = W + f * p.K + c * 9;
        double sq[9];
        bool bad = false;
#pragma unroll
        for (int pos = 0; pos < 9; ++pos) {
            const float v = ld_half(k, pos, dtype);
            bad |= !isfinite(v);
            const double w = (double)v;
            sq[pos] = w * w;
        }
        double best = -1.0;
        int bq = 0;
        for (int q = 0; q < ps.n; ++q) {
            double e = 0.0;
#pragma unroll
            for (int pos = 0; pos < 9; ++pos)
                if ((ps.m[q] >> pos) & 1u) e += sq[pos];
            if (e > best) {
                best = e;
                bq = q;
            }
        }
        scores[g] = best;
        patsel[g] = (uint8_t)bq;
        if (bad) atomicExch(nonfinite, 1);
    }
}

// Element (f, 9c + pos) survives when kernel (f, c) survives and pos is in
// its pattern.
__global__ void pattern_mask_kernel(Part p, const uint8_t *__restrict__ keep,
                                    const uint8_t *__restrict__ patsel, PatternSet ps,
                                    uint8_t *__restrict__ mask) {
    const int64_t total = p.M * p.K;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t f = i / p.K, k = i - f * p.K, c = k / 9, pos = k - c * 9;
        const int64_t g = f * p.C + c;
        mask[i] = (keep[g] && ((ps.m[patsel[g]] >> pos) & 1u)) ? 1 : 0;
    }
}

int grid_for(int64_t n, int threads) {
    int64_t b = (n + threads - 1) / threads;
    const int64_t cap = (int64_t)num_sms() * 16;
    if (b > cap) b = cap;
    return (int)(b < 1 ? 1 : b);
}

}  // namespace

cudaError_t launch_scores(const bp_layout &lay, const void *W, double *scores, int *nonfinite,
                          cudaStream_t s) {
    const Part p = make_part(lay);
    scores_kernel<<<grid_for(p.U, 256), 256, 0, s>>>(p, lay.dtype,
                                                     static_cast<const uint16_t *>(W), scores,
                                                     nonfinite);
    return cudaGetLastError();
}

cudaError_t launch_base_select(const bp_layout &lay, const double *scores, double rate,
                               uint8_t *keep, cudaStream_t s) {
    const Part p = make_part(lay);
    base_select_kernel<<<grid_for(p.U, 256), 256, 0, s>>>(p, rate, scores, keep);
    return cudaGetLastError();
}

cudaError_t launch_radix_hist(int64_t U, const double *scores, const uint8_t *keep,
                              uint64_t prefix, int shift, unsigned *hist, cudaStream_t s) {
    radix_hist_kernel<<<grid_for(U, 512), 512, 0, s>>>(U, scores, keep, prefix, shift, hist);
    return cudaGetLastError();
}

int64_t threshold_chunks(int64_t U) { return (U + kChunk - 1) / kChunk; }

cudaError_t launch_threshold_select(int64_t U, const double *scores, uint8_t *keep,
                                    uint64_t thr, int64_t need, int64_t *chunk_cnt,
                                    cudaStream_t s) {
    const int64_t nch = threshold_chunks(U);
    threshold_count_kernel<<<(unsigned)nch, 256, 0, s>>>(U, scores, keep, thr, chunk_cnt);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    scan_chunks_kernel<<<1, kSelThreads, 0, s>>>(nch, chunk_cnt);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    if (need > 0)
        threshold_ties_kernel<<<(unsigned)nch, kSelThreads, 0, s>>>(U, scores, keep, thr, need,
                                                                   chunk_cnt);
    return cudaGetLastError();
}

cudaError_t launch_pattern_scores(const bp_layout &lay, const void *W, const PatternSet &ps,
                                  double *scores, uint8_t *patsel, int *nonfinite,
                                  cudaStream_t s) {
    const Part p = make_part(lay);
    pattern_scores_kernel<<<grid_for(p.U, 256), 256, 0, s>>>(
        p, lay.dtype, static_cast<const uint16_t *>(W), ps, scores, patsel, nonfinite);
    return cudaGetLastError();
}

cudaError_t launch_pattern_mask(const bp_layout &lay, const uint8_t *keep, const uint8_t *patsel,
                                const PatternSet &ps, uint8_t *mask, cudaStream_t s) {
    const Part p = make_part(lay);
    pattern_mask_kernel<<<grid_for(p.M * p.K, 256), 256, 0, s>>>(p, keep, patsel, ps, mask);
    return cudaGetLastError();
}

cudaError_t launch_write_mask(const bp_layout &lay, const uint8_t *keep, uint8_t *mask,
                              cudaStream_t s) {
    const Part p = make_part(lay);
    write_mask_kernel<<<grid_for(p.M * p.K, 256), 256, 0, s>>>(p, keep, mask);
    return cudaGetLastError();
}

}  // namespace bp
