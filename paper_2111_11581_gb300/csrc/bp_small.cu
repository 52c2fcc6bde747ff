// Short path of bp_gemm for small layers with small row-blocks (bm <= 32).
//
// A layer of a few million kept multiply-adds (the 512 x 512 FC layer at 4x
// over 64 tokens: 4.2 M) is over before the tensor-core kernel's pipeline has
// filled: its persistent CTAs set up tensor memory, fetch chunk records, then
// the 128-row slab tiles and their gathered rows, each a dependent round trip
// to memory.  Here one CTA computes one row-block of bm rows for 32 tokens
// straight from the compact storage of Sec. 4.3 (values of the row-block,
// bm x K' row-major, and its kept-column list), on the CUDA cores in fp32;
// only kept weights enter the product, row-block by row-block, as in the
// paper's own per-row-block kernels.  Bias, ReLU and the round-to-nearest-even
// cast follow.
//
// Such a launch is a chain of memory round trips, so the kernel keeps the
// chain short: the row-block's range, its column indices and weights are all
// requested at once, the range guessed as rb x (K' of an even split) -- a
// layer pruned at one rate keeps the same number of columns in every
// row-block -- and checked when the row-block pointers arrive (a wrong guess
// reloads); when K is at most kStageK the CTA's 32 tokens of every activation
// row are copied to shared memory in the same round trip, without waiting for
// the column indices, and the product indexes them there.  Longer rows are
// gathered by column index, 128 listed columns per step.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "bp_common.cuh"

// BP_TRACE (off by default; a build for measurement only): thread 0 of each
// of the first 256 CTAs records clock64() at its start (0), once its loads
// are issued (1), once the row-block range arrived (2), once the step's data
// landed (3), after the product (4) and at its end (5), and the global timer
// at its start (6) and end (7); read back with bp_debug_small_trace_read().
#ifdef BP_TRACE
namespace bp {
__device__ unsigned long long g_small_trace[256 * 8];
}  // namespace bp
#define BP_TS(ev, v)                                                      \
    do {                                                                  \
        if (threadIdx.x == 0 && blockIdx.y == 0 && blockIdx.x < 256)      \
            bp::g_small_trace[blockIdx.x * 8 + (ev)] = (v);               \
    } while (0)
#else
#define BP_TS(ev, v) \
    do {             \
    } while (0)
#endif

namespace bp {
namespace {

constexpr int kSmallThreads = 256;
constexpr int kSmallWarps = kSmallThreads / 32;
constexpr int kSmallTok = 32;      // tokens per CTA
constexpr int kSmallK = 128;       // listed columns per step
constexpr int kSmallMaxBm = 32;
constexpr int64_t kStageK = 1024;  // activation rows staged whole up to this K (64 KB)
// dynamic shared memory: weights of a step (rows padded to 136 values: the
// four rows a warp reads at once fall in different banks), each warp's partial
// sums, the step's column indices, then the activation rows (all K of them,
// or the step's gathered ones)
constexpr int kWPitch = kSmallK + 8;
constexpr int kOffW = 0, kOffRed = kOffW + kSmallMaxBm * kWPitch * 2;
constexpr int kOffIdx = kOffRed + kSmallWarps * kSmallMaxBm * kSmallTok * 4;
constexpr int kOffX = kOffIdx + kSmallK * 4;
constexpr int kMostSmem = kOffX + (int)kStageK * kSmallTok * 2;

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
    int64_t M, K, N, ldx, ldy;
    int64_t kp_even;     // K' of every row-block if they all kept the same count, else -1
    int bm, relu;
};

// 16-byte copies of token columns n .. n+7 of activation row k (zero past N)
__device__ __forceinline__ void copy_tokens(uint32_t dst, const SmallParams &p, int64_t k, int64_t n) {
    uint32_t nb = 0;
    const uint16_t *src = p.X;
    if (n < p.N) {
        nb = (uint32_t)min((int64_t)16, (p.N - n) * 2);
        src = p.X + k * p.ldx + n;
    }
    cp_async_16(dst, src, nb);
}

// grid: (row-blocks, token tiles of 32).  Warp w takes the column pairs
// (2q, 2q + 1), q = w (mod 8), of each step; lane l: tokens 4 (l % 8) .. +3,
// rows l / 8 + 4 j.  The warps' partial sums are added in warp order.
template <bool kBf16, bool kStage>
__global__ void __launch_bounds__(kSmallThreads) bp_small_kernel(const __grid_constant__ SmallParams p) {
    extern __shared__ __align__(16) uint8_t dsm[];
    uint16_t (*wsm)[kWPitch] = reinterpret_cast<uint16_t (*)[kWPitch]>(dsm + kOffW);
    float (*red)[kSmallMaxBm][kSmallTok] =
        reinterpret_cast<float (*)[kSmallMaxBm][kSmallTok]>(dsm + kOffRed);
    int32_t *cis = reinterpret_cast<int32_t *>(dsm + kOffIdx);
    uint16_t (*xs)[kSmallTok] = reinterpret_cast<uint16_t (*)[kSmallTok]>(dsm + kOffX);
    const int64_t rb = blockIdx.x, n0 = (int64_t)blockIdx.y * kSmallTok;
    const int64_t r0 = rb * p.bm;
    const int rows = (int)min((int64_t)p.bm, p.M - r0);
    const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
    const int tq = (lane & 7) * 4, rq = lane >> 3;
    BP_TS(0, clock64());
    BP_TS(6, globaltimer_ns());
    // this thread's outputs in the epilogue: row t / 8, tokens 4 (t % 8) ..;
    // its bias is requested now, with the other loads
    const int orow = t >> 3, oq = (t & 7) * 4;
    const float bv = (p.bias && orow < rows) ? p.bias[r0 + orow] : 0.f;
    // the row-block's range, requested now and used once the first step's
    // loads (issued for the guessed range) are in flight
    const int64_t ra = p.rb_ptr[rb], rz = p.rb_ptr[rb + 1];
    int64_t c0 = p.kp_even >= 0 ? rb * p.kp_even : ra;
    int64_t kp = p.kp_even >= 0 ? p.kp_even : rz - ra;
    bool first = true;
    float acc[kSmallMaxBm / 4][4];
#pragma unroll
    for (int j = 0; j < kSmallMaxBm / 4; ++j)
#pragma unroll
        for (int e = 0; e < 4; ++e) acc[j][e] = 0.f;
    for (int64_t k0 = 0; k0 < kp; k0 += kSmallK) {
        const int kn = (int)min((int64_t)kSmallK, kp - k0);
        const uint16_t *wrb = p.values + (int64_t)p.bm * c0;             // rows x K' row-major
        // All loads of the step are issued before any is used (a loop that
        // consumes each load before issuing the next serialises the round
        // trips): the column indices and the weights, then the rows.
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
        if (first) {
            first = false;
            // Launched as a programmatic dependent: the packed weights (written
            // by bp_pack, which synchronises) are read above while the previous
            // kernel may still run; the activations may come from that kernel,
            // so they are read after it.
            grid_dependency_wait();
            grid_launch_dependents();
            if (kStage) {
                for (int e = t; e < (int)p.K * (kSmallTok / 8); e += kSmallThreads)
                    copy_tokens(smem_u32(&xs[e >> 2][(e & 3) * 8]), p, e >> 2, n0 + (e & 3) * 8);
                cp_async_commit();
            }
            BP_TS(1, clock64());
            if (c0 != ra || kp != rz - ra) {
                // the row-blocks keep different counts: start over on the real range
                c0 = ra;
                kp = rz - ra;
                k0 = -kSmallK;
                continue;
            }
        }
        if (kStage) {
            // the step's column indices, from the copies already in registers
#pragma unroll
            for (int u = 0; u < kXU; ++u)
                if ((t & 3) == 0) cis[(t + kSmallThreads * u) >> 2] = ci[u];
        } else {
#pragma unroll
            for (int u = 0; u < kXU; ++u) {
                const int e = t + kSmallThreads * u;
                const int i = e >> 2, q = (e & 3) * 8;
                if (i < kn) copy_tokens(smem_u32(&xs[i][q]), p, ci[u], n0 + q);
                else cp_async_16(smem_u32(&xs[i][q]), p.X, 0u);
            }
            cp_async_commit();
        }
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
        BP_TS(2, clock64());
        cp_async_wait_all();
        __syncthreads();
        BP_TS(3, clock64());
        // column pairs: one 4-byte weight load per row serves two columns
#pragma unroll 2
        for (int i = 2 * warp; i + 1 < kn; i += 2 * kSmallWarps) {
            const int xa = kStage ? cis[i] : i, xb = kStage ? cis[i + 1] : i + 1;
            const uint2 va = *reinterpret_cast<const uint2 *>(&xs[xa][tq]);
            const uint2 vb = *reinterpret_cast<const uint2 *>(&xs[xb][tq]);
            const float a0 = to_f<kBf16>(va.x & 0xffffu), a1 = to_f<kBf16>(va.x >> 16);
            const float a2 = to_f<kBf16>(va.y & 0xffffu), a3 = to_f<kBf16>(va.y >> 16);
            const float b0 = to_f<kBf16>(vb.x & 0xffffu), b1 = to_f<kBf16>(vb.x >> 16);
            const float b2 = to_f<kBf16>(vb.y & 0xffffu), b3 = to_f<kBf16>(vb.y >> 16);
#pragma unroll
            for (int j = 0; j < kSmallMaxBm / 4; ++j) {
                if (rq + 4 * j < rows) {
                    const uint32_t w2 = *reinterpret_cast<const uint32_t *>(&wsm[rq + 4 * j][i]);
                    const float wa = to_f<kBf16>(w2 & 0xffffu), wb = to_f<kBf16>(w2 >> 16);
                    acc[j][0] = fmaf(wb, b0, fmaf(wa, a0, acc[j][0]));
                    acc[j][1] = fmaf(wb, b1, fmaf(wa, a1, acc[j][1]));
                    acc[j][2] = fmaf(wb, b2, fmaf(wa, a2, acc[j][2]));
                    acc[j][3] = fmaf(wb, b3, fmaf(wa, a3, acc[j][3]));
                }
            }
        }
        if ((kn & 1) && warp == ((kn - 1) >> 1) % kSmallWarps) {
            // odd count: the last column alone
            const int i = kn - 1, xa = kStage ? cis[i] : i;
            const uint2 va = *reinterpret_cast<const uint2 *>(&xs[xa][tq]);
            const float a0 = to_f<kBf16>(va.x & 0xffffu), a1 = to_f<kBf16>(va.x >> 16);
            const float a2 = to_f<kBf16>(va.y & 0xffffu), a3 = to_f<kBf16>(va.y >> 16);
#pragma unroll
            for (int j = 0; j < kSmallMaxBm / 4; ++j) {
                if (rq + 4 * j < rows) {
                    const float wa = to_f<kBf16>(wsm[rq + 4 * j][i]);
                    acc[j][0] = fmaf(wa, a0, acc[j][0]);
                    acc[j][1] = fmaf(wa, a1, acc[j][1]);
                    acc[j][2] = fmaf(wa, a2, acc[j][2]);
                    acc[j][3] = fmaf(wa, a3, acc[j][3]);
                }
            }
        }
        __syncthreads();
    }
    if (first) {                // nothing listed: the output is the bias alone
        grid_dependency_wait();
        grid_launch_dependents();
    }
    cp_async_wait_all();        // staged rows that no step read
    BP_TS(4, clock64());
    // each warp's partial sums to its own slice of shared memory
#pragma unroll
    for (int j = 0; j < kSmallMaxBm / 4; ++j)
        if (rq + 4 * j < rows)
            *reinterpret_cast<float4 *>(&red[warp][rq + 4 * j][tq]) =
                make_float4(acc[j][0], acc[j][1], acc[j][2], acc[j][3]);
    __syncthreads();
    // epilogue: the warps' sums in warp order, + bias, ReLU, one rounding to
    // the weight dtype; thread = (row, 4 tokens)
    if (orow < rows) {
        const int r = orow, q = oq;
        const int64_t m = r0 + r, n = n0 + q;
        float4 a = *reinterpret_cast<const float4 *>(&red[0][r][q]);
#pragma unroll
        for (int w = 1; w < kSmallWarps; ++w) {
            const float4 v = *reinterpret_cast<const float4 *>(&red[w][r][q]);
            a.x += v.x;
            a.y += v.y;
            a.z += v.z;
            a.w += v.w;
        }
        const float sum[4] = {a.x, a.y, a.z, a.w};
        uint16_t o[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            float v = sum[u] + bv;
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
    BP_TS(5, clock64());
    BP_TS(7, globaltimer_ns());
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
    p.K = P.lay.K;
    p.N = N;
    p.ldx = ldx;
    p.ldy = ldy;
    p.bm = P.lay.bm;
    p.relu = relu;
    // values hold bm x K' per row-block: an even split of the total is the
    // guess every row-block checks against its own range
    const int64_t per_rb = (int64_t)P.lay.bm * P.num_rb;
    p.kp_even = (per_rb > 0 && P.nnz_vals % per_rb == 0) ? P.nnz_vals / per_rb : -1;
    const bool stage = P.lay.K <= kStageK;
    const int smem = kOffX + (int)(stage ? P.lay.K : kSmallK) * kSmallTok * 2;     // > 48 KB
    const bool bf16 = P.lay.dtype == BP_BF16;
    const void *fn = stage ? (bf16 ? (const void *)bp_small_kernel<true, true> : (const void *)bp_small_kernel<false, true>)
                           : (bf16 ? (const void *)bp_small_kernel<true, false> : (const void *)bp_small_kernel<false, false>);
    // more than 48 KB of dynamic shared memory: allowed once per process (for
    // the largest K staged)
    static const cudaError_t raised = [] {
        const void *fns[4] = {(const void *)bp_small_kernel<true, true>,
                              (const void *)bp_small_kernel<false, true>,
                              (const void *)bp_small_kernel<true, false>,
                              (const void *)bp_small_kernel<false, false>};
        cudaError_t e = cudaSuccess;
        for (const void *f : fns)
            if (e == cudaSuccess)
                e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, kMostSmem);
        return e;
    }();
    if (raised != cudaSuccess) return raised;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)P.num_rb, (unsigned)((N + kSmallTok - 1) / kSmallTok));
    cfg.blockDim = dim3(kSmallThreads);
    cfg.dynamicSmemBytes = (size_t)smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
#ifdef BP_NO_PDL
    cfg.numAttrs = 0;       // (measurement build) an ordinary stream-ordered launch
#else
    cfg.numAttrs = 1;
#endif
    void *args[] = {&p};
    return cudaLaunchKernelExC(&cfg, fn, args);
}

}  // namespace bp

#ifdef BP_TRACE
extern "C" int bp_debug_small_trace_read(unsigned long long *host, int n) {
    if (n > 256 * 8) n = 256 * 8;
    return cudaMemcpyFromSymbol(host, bp::g_small_trace, n * sizeof(unsigned long long)) == cudaSuccess ? n : -1;
}
#endif
