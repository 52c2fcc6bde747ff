// Rates that bound the block-sparse product's design, measured on all SMs:
//   test 0: back-to-back tcgen05.mma 128 x N x 16 (bf16, fp32 accumulate) from
//           one thread per CTA, operands resident in shared memory, one commit
//           at the end: cycles per instruction against N;
//   test 1: TMA bulk copies of 16 KB global -> shared from 1..6 threads of a
//           CTA, four in flight per thread: bytes per cycle an SM ingests.
// Not part of libbp; built and run by `python -m paper_2111_11581_gb300.variants probe`.
#include <cuda.h>
#include <cstdio>
#include <cstdlib>
#include <vector>

#include "../csrc/bp_common.cuh"

using namespace bp;

constexpr uint64_t kLim = 1000000000ull;

struct PP {
    int test, iters, N, nthreads;
    const uint8_t *W;
    unsigned long long *out;
    unsigned *err;
};

__global__ void __launch_bounds__(256, 1) probe(const __grid_constant__ PP p) {
    extern __shared__ __align__(1024) uint8_t raw[];
    uint8_t *base = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(raw) + 1023) & ~(uintptr_t)1023);
    uint64_t *bars = reinterpret_cast<uint64_t *>(base + 6 * 16384 + 65536);
    uint32_t *tbase = reinterpret_cast<uint32_t *>(bars + 16);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int i = 0; i < 16; ++i) mbar_init(&bars[i], 1);
        fence_mbar_init();
    }
    for (int i = threadIdx.x; i < (6 * 16384 + 65536) / 16; i += blockDim.x)
        reinterpret_cast<uint4 *>(base)[i] = make_uint4(0, 0, 0, 0);
    fence_proxy_async_smem();
    if (warp == 0) {
        tmem_alloc(tbase, 512);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tbase;
    if (p.test == 0) {
        if (threadIdx.x == 0) {
            const uint32_t idesc = make_idesc(true, false, true, 128, p.N);
            const uint64_t a0 = make_sdesc_sw128(smem_u32(base), 16, 1024);
            const uint64_t b0 = make_sdesc_sw128(smem_u32(base + 16384), 8192, 1024);
            const unsigned long long t0 = clock64();
            for (int it = 0; it < p.iters; ++it) {
#pragma unroll
                for (int kk = 0; kk < 16; ++kk)
                    umma_f16_ss(tmem, a0 + (kk & 3) * 2, b0 + (kk & 3) * 128, idesc, 1u);
            }
            umma_commit(&bars[0]);
            const bool ok = mbar_wait(&bars[0], 0, kLim, nullptr);
            p.out[blockIdx.x] = clock64() - t0;
            if (!ok) atomicOr(p.err, 1u);
        }
    } else {
        const int t = warp;
        if (lane == 0 && t < p.nthreads) {
            uint64_t *b = &bars[t * 2];
            const uint32_t dst = smem_u32(base + (t % 6) * 16384);
            const unsigned long long t0 = clock64();
            bool ok = true;
            for (int it = 0; it < p.iters && ok; ++it) {
                mbar_arrive_expect_tx(b, 4 * 16384);
#pragma unroll
                for (int q = 0; q < 4; ++q)
                    bulk_g2s(dst, p.W + (((int64_t)blockIdx.x * 97 + it * 4 + q + t * 1000) % 512) * 16384,
                             16384, b);
                ok = mbar_wait(b, (uint32_t)(it & 1), kLim, nullptr);
            }
            if (t == 0) p.out[blockIdx.x] = clock64() - t0;
            if (!ok) atomicOr(p.err, 2u);
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 0) tmem_dealloc(tmem, 512);
}

int main(int argc, char **argv) {
    const int test = argc > 1 ? atoi(argv[1]) : 0;
    const int iters = argc > 2 ? atoi(argv[2]) : 512;
    const int N = argc > 3 ? atoi(argv[3]) : 256;
    const int nth = argc > 4 ? atoi(argv[4]) : 1;
    if (N < 16 || N > 256 || N % 16 || nth < 1 || nth > 6 || iters < 1) return 2;
    int sms = 0;
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, 0);
    uint8_t *W = nullptr;
    cudaMalloc(&W, 512 * 16384);
    cudaMemset(W, 0, 512 * 16384);
    unsigned long long *out = nullptr;
    unsigned *err = nullptr;
    cudaMalloc(&out, sms * 8);
    cudaMalloc(&err, 4);
    cudaMemset(err, 0, 4);
    PP p{test, iters, N, nth, W, out, err};
    const int smem = 1024 + 6 * 16384 + 65536 + 256;
    cudaFuncSetAttribute(probe, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    for (int w = 0; w < 2; ++w) probe<<<sms, 256, smem>>>(p);
    if (cudaDeviceSynchronize() != cudaSuccess) {
        printf("cuda error\n");
        return 4;
    }
    probe<<<sms, 256, smem>>>(p);
    if (cudaDeviceSynchronize() != cudaSuccess) {
        printf("cuda error\n");
        return 4;
    }
    std::vector<unsigned long long> h(sms);
    unsigned herr = 0;
    cudaMemcpy(h.data(), out, sms * 8, cudaMemcpyDeviceToHost);
    cudaMemcpy(&herr, err, 4, cudaMemcpyDeviceToHost);
    double avg = 0;
    for (int i = 0; i < sms; ++i) avg += h[i];
    avg /= sms;
    if (test == 0)
        printf("tcgen05.mma 128 x %d x 16: %.1f cycles per instruction (err %u)\n", N,
               avg / (iters * 16.0), herr);
    else
        printf("bulk copies from %d thread(s): %.1f bytes per cycle per SM (err %u)\n", nth,
               nth * 16384.0 * 4 * iters / avg, herr);
    return herr ? 5 : 0;
}
