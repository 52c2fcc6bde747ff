// Short path of bp_gemm for small layers with small row-blocks (bm <= 32).
//
// A layer of a few million kept multiply-adds (the 512 x 512 FC layer at 4x
// over 64 tokens: 4.2 M) is over before the tensor-core kernel's pipeline has
// filled: its persistent CTAs set up tensor memory, fetch chunk records, then
// the 128-row slab tiles and their gathered rows, each a dependent round trip
// to memory.  Here one CTA computes one row-block of bm rows for 32 tokens
// straight from the compact storage of Sec. 4.3 (values of the row-block,
// bm x K' row-major, and its kept-column list): per 128 listed columns it
// gathers those activation rows into shared memory (16-byte cp.async) and
// loads the row-block's weights for them, all loads of a step in flight
// together; the 8 warps split the columns, accumulate in fp32 on the CUDA
// cores and meet in shared memory; bias, ReLU and the round-to-nearest-even
// cast follow.  Only kept weights enter the product, row-block by row-block,
// as in the paper's own per-row-block kernels.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "bp_common.cuh"

namespace bp {
namespace {

constexpr int kSmallThreads = 256;
constexpr int kSmallWarps = kSmallThreads / 32;
constexpr int kSmallTok = 32;      // tokens per CTA
constexpr int kSmallK = 128;       // listed columns per step
constexpr int kSmallMaxBm = 32;

template <bool kBf16>
__device__ __forceinline__ float to_f(uint32_t v) {
    if (kBf16) return __uint_as_float(v << 16);
    return __half2float(__ushort_as_half((unsigned short)v));
}

template <bool kBf16>
__device__ __forceinline__ uint16_t from_f(float v) {
    if (kBf16) return __bfloat16_as_ushort(__float2bfloat16_rn(v));
    return __half_as_ushort(__float2half_rn(v));
}

struct SmallParams {
    const int64_t *rb_ptr;
    const int32_t *col_idx;
    const uint16_t *values;
    const uint16_t *X;
    uint16_t *Y;
    const float *bias;
    int64_t M, N, ldx, ldy;
    int bm, relu;
};

// grid: (row-blocks, token tiles of 32).  Warp w takes the listed columns
// i = w (mod 8) of each step; lane l: tokens 4 (l % 8) .. +3, rows l / 8 + 4 j.
template <bool kBf16>
__global__ void __launch_bounds__(kSmallThreads) bp_small_kernel(const __grid_constant__ SmallParams p) {
    __shared__ __align__(16) uint16_t xs[kSmallK][kSmallTok];      // gathered rows (8 KB)
    __shared__ __align__(16) uint16_t wsm[kSmallMaxBm][kSmallK];   // weights of the step (8 KB)
    __shared__ float out[kSmallMaxBm][kSmallTok];                   // the warps' sums
    const int64_t rb = blockIdx.x, n0 = (int64_t)blockIdx.y * kSmallTok;
    const int64_t r0 = rb * p.bm;
    const int rows = (int)min((int64_t)p.bm, p.M - r0);
    const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
    const int tq = (lane & 7) * 4, rq = lane >> 3;
    for (int e = t; e < kSmallMaxBm * kSmallTok; e += kSmallThreads) (&out[0][0])[e] = 0.f;
    __syncthreads();
    const int64_t c0 = p.rb_ptr[rb], kp = p.rb_ptr[rb + 1] - c0;    // K' of the row-block
    const uint16_t *wrb = p.values + (int64_t)p.bm * c0;             // rows x K' row-major
    float acc[kSmallMaxBm / 4][4];
#pragma unroll
    for (int j = 0; j < kSmallMaxBm / 4; ++j)
#pragma unroll
        for (int e = 0; e < 4; ++e) acc[j][e] = 0.f;
    for (int64_t k0 = 0; k0 < kp; k0 += kSmallK) {
        const int kn = (int)min((int64_t)kSmallK, kp - k0);
        // All loads of the step are issued before any is used (a loop that
        // consumes each load before issuing the next serialises the round
        // trips): the column indices and the weights, then the gathered rows.
        constexpr int kXU = kSmallK * (kSmallTok / 8) / kSmallThreads;     // 2 copies per thread
        constexpr int kWU = kSmallMaxBm * kSmallK / 8 / kSmallThreads;     // 2 per thread
        int32_t ci[kXU];
#pragma unroll
        for (int u = 0; u < kXU; ++u) {
            const int i = (t + kSmallThreads * u) >> 2;
            ci[u] = i < kn ? p.col_idx[c0 + k0 + i] : 0;
        }
        // weights: 8 consecutive columns of one row per thread and pass
        uint16_t wv[kWU][8];
#pragma unroll
        for (int u = 0; u < kWU; ++u) {
            const int e = t + kSmallThreads * u, r = e / (kSmallK / 8), i = (e % (kSmallK / 8)) * 8;
#pragma unroll
            for (int q = 0; q < 8; ++q)
                wv[u][q] = (r < rows && i + q < kn) ? wrb[(int64_t)r * kp + k0 + i + q] : (uint16_t)0;
        }
        // Launched as a programmatic dependent: the packed weights (written by
        // bp_pack, which synchronises) are read above while the previous
        // kernel may still run; the activations may come from that kernel, so
        // the first gather waits for it.
        if (k0 == 0) {
            grid_dependency_wait();
            grid_launch_dependents();
        }
#pragma unroll
        for (int u = 0; u < kXU; ++u) {
            const int e = t + kSmallThreads * u;
            const int i = e >> 2, q = (e & 3) * 8;
            const int64_t n = n0 + q;
            uint32_t nb = 0;
            const uint16_t *src = p.X;
            if (i < kn && n < p.N) {
                nb = (uint32_t)min((int64_t)16, (p.N - n) * 2);
                src = p.X + (int64_t)ci[u] * p.ldx + n;
            }
            cp_async_16(smem_u32(&xs[i][q]), src, nb);
        }
        cp_async_commit();
#pragma unroll
        for (int u = 0; u < kWU; ++u) {
            const int e = t + kSmallThreads * u, r = e / (kSmallK / 8), i = (e % (kSmallK / 8)) * 8;
            uint4 pk;
            pk.x = wv[u][0] | ((uint32_t)wv[u][1] << 16);
            pk.y = wv[u][2] | ((uint32_t)wv[u][3] << 16);
            pk.z = wv[u][4] | ((uint32_t)wv[u][5] << 16);
            pk.w = wv[u][6] | ((uint32_t)wv[u][7] << 16);
            *reinterpret_cast<uint4 *>(&wsm[r][i]) = pk;
        }
        cp_async_wait_all();
        __syncthreads();
        for (int i = warp; i < kn; i += kSmallWarps) {
            const uint2 xv = *reinterpret_cast<const uint2 *>(&xs[i][tq]);
            const float x0 = to_f<kBf16>(xv.x & 0xffffu), x1 = to_f<kBf16>(xv.x >> 16);
            const float x2 = to_f<kBf16>(xv.y & 0xffffu), x3 = to_f<kBf16>(xv.y >> 16);
#pragma unroll
            for (int j = 0; j < kSmallMaxBm / 4; ++j) {
                const float w = to_f<kBf16>(wsm[rq + 4 * j][i]);
                acc[j][0] = fmaf(w, x0, acc[j][0]);
                acc[j][1] = fmaf(w, x1, acc[j][1]);
                acc[j][2] = fmaf(w, x2, acc[j][2]);
                acc[j][3] = fmaf(w, x3, acc[j][3]);
            }
        }
        __syncthreads();
    }
    if (kp == 0) {              // nothing listed: the output is the bias alone
        grid_dependency_wait();
        grid_launch_dependents();
    }
    // the warps' partial sums meet in shared memory
#pragma unroll
    for (int j = 0; j < kSmallMaxBm / 4; ++j)
        if (rq + 4 * j < rows)
#pragma unroll
            for (int e = 0; e < 4; ++e) atomicAdd(&out[rq + 4 * j][tq + e], acc[j][e]);
    __syncthreads();
    // epilogue: + bias, ReLU, one rounding to the weight dtype; thread = (row, 4 tokens)
    for (int e = t; e < rows * (kSmallTok / 4); e += kSmallThreads) {
        const int r = e / (kSmallTok / 4), q = (e % (kSmallTok / 4)) * 4;
        const int64_t m = r0 + r, n = n0 + q;
        const float bv = p.bias ? p.bias[m] : 0.f;
        uint16_t o[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            float v = out[r][q + u] + bv;
            if (p.relu) v = fmaxf(v, 0.f);
            o[u] = from_f<kBf16>(v);
        }
        uint16_t *dst = p.Y + m * p.ldy + n;
        if (n + 4 <= p.N) {
            uint2 pk;
            pk.x = o[0] | ((uint32_t)o[1] << 16);
            pk.y = o[2] | ((uint32_t)o[3] << 16);
            *reinterpret_cast<uint2 *>(dst) = pk;
        } else {
            for (int u = 0; u < 4 && n + u < p.N; ++u) dst[u] = o[u];
        }
    }
}

}  // namespace

bool small_path_ok(const bp_packed &P, int64_t N) {
    // small row-blocks and few kept multiply-adds: the fixed latency of the
    // tensor-core pipeline would dominate (measured: the 512 x 512 FC layer at
    // 4x over 64 tokens takes ~17 us there)
    return P.lay.bm <= kSmallMaxBm && N > 0 && P.nnz_vals * N <= ((int64_t)1 << 24) &&
           P.num_rb <= 2147483647 && (N + kSmallTok - 1) / kSmallTok <= 65535;
}

cudaError_t launch_small(const bp_packed &P, const void *X, int64_t N, int64_t ldx,
                         const float *bias, int relu, void *Y, int64_t ldy, cudaStream_t s) {
    SmallParams p{};
    p.rb_ptr = P.rb_ptr;
    p.col_idx = P.col_idx;
    p.values = static_cast<const uint16_t *>(P.values);
    p.X = static_cast<const uint16_t *>(X);
    p.Y = static_cast<uint16_t *>(Y);
    p.bias = bias;
    p.M = P.lay.M;
    p.N = N;
    p.ldx = ldx;
    p.ldy = ldy;
    p.bm = P.lay.bm;
    p.relu = relu;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)P.num_rb, (unsigned)((N + kSmallTok - 1) / kSmallTok));
    cfg.blockDim = dim3(kSmallThreads);
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return P.lay.dtype == BP_BF16 ? cudaLaunchKernelEx(&cfg, bp_small_kernel<true>, p)
                                  : cudaLaunchKernelEx(&cfg, bp_small_kernel<false>, p);
}

}  // namespace bp
