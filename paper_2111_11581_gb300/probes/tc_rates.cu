// Rates that bound the block-sparse product's design, measured on all SMs:
//   test 0: back-to-back tcgen05.mma 128 x N x 16 (bf16, fp32 accumulate) from
//           one thread per CTA, operands resident in shared memory, one commit
//           at the end: cycles per instruction against N;
//   test 1: TMA bulk copies of 16 KB global -> shared from 1..6 threads of a
//           CTA, four in flight per thread: bytes per cycle an SM ingests;
//   test 2: the product's stage ring without data: a control thread releases
//           stage s (one arrival) once the tensor cores are done with it, the
//           MMA thread waits for the stage, optionally fences (flags: 1
//           tcgen05.fence::after_thread_sync, 2 fence.proxy.async), issues
//           four 128 x N x 16 MMAs (one 64-column chunk; flags bits 8-11: a
//           different count) and commits to the stage's empty barrier (flag
//           4: no waits at all, only the commits): cycles per stage against
//           stages, fences and MMAs per commit;
//   test 4: back-to-back MMAs in groups of 2, 4 or 8 with a commit after
//           each group (or none), one or two alternating accumulators: what a
//           commit costs the issue stream;
//   test 5: the cp.async row gather alone (8 KB batches, two in flight per
//           warp), rows at a given pitch over a given footprint: bytes per
//           cycle an SM ingests against the footprint;
//   test 6: the copy mix of the product without the tensor core: scattered
//           row gathers from several warps beside one thread streaming 16 KB
//           bulk copies: whether the two paths slow each other;
//   test 7: the product's stage ring with its data and without the tensor
//           core (weight tile bulk copy + 64 gathered activation rows per
//           chunk, two gather groups, a consumer that releases each stage):
//           cycles per chunk against the rows' spread, the tiles shared
//           between CTAs, the weight copies and the hold time;
//   test 8: groups of four 128 x N x 16 MMAs and a commit (one 64-column
//           chunk) with the tensor-core thread's per-chunk work between the
//           groups (flags: 1 tcgen05.fence::after_thread_sync, 2
//           fence.proxy.async, 4 try_wait on a completed barrier, 8 test_wait
//           on a completed barrier, 16 a dependent shared-memory load, 32 a
//           chain of 32 dependent integer operations, 64 a clock64 store to
//           global memory, 128 test_wait on an incomplete barrier; 256: that
//           work after the group's second MMA instead of before its first;
//           512: clock64 read before and after each group, to time its issue;
//           1024: meanwhile warps 2-9 poll a barrier that never completes;
//           2048: meanwhile warps 2-7 gather 512-byte rows with cp.async;
//           4096: the groups' operands rotate over four 48 KB stages, as in
//           the product, instead of one resident A and B; 8192: no work
//           function at all between the groups; 16384: eight rarely taken
//           branches between the groups, each around a nanosleep):
//           cycles per group (and how long the thread takes to issue one);
//   test 3: test 0's back-to-back MMAs while 1..6 other warps copy into a
//           separate shared-memory area (TMA bulk copies of 16 KB, or with
//           flag 4 one warp-wide 512-byte cp.async row per instruction, 16
//           rows per batch): cycles per MMA and bytes per cycle ingested, to
//           see whether operand reads and incoming copies slow each other.
// Not part of libbp; built and run by `python -m paper_2111_11581_gb300.variants probe`.
#include <cuda.h>
#include <cstdio>
#include <cstdlib>
#include <vector>

#include "../csrc/bp_common.cuh"

using namespace bp;

constexpr uint64_t kLim = 1000000000ull;
constexpr int kData = 4 * 49152;    // shared-memory data area (test 7: four 48 KB stages)

struct PP;
template <int kCode>
__device__ __forceinline__ void t8_loop(const PP &p, uint32_t tmem, uint64_t a0, uint64_t b0, uint32_t idesc,
                                        uint64_t *bars, const volatile uint32_t *vz, bool &ok);
struct PP {
    int test, iters, N, nthreads, flags;
    const uint8_t *W;
    unsigned long long *out;    // [2 * gridDim.x]: per CTA cycles (and test 3: bytes copied, cycles)
    unsigned *err;
};

// test 8 with nthreads = code >= 2: the groups with one kind of per-group code
// present in the loop, run when flag bit (code - 2) is set: 2 tcgen05 fence,
// 3 try_wait (bounded wait) on a completed barrier, 4 test_wait, 5 proxy
// fence, 6 a shared-memory load feeding the descriptor, 7 a clock64 store,
// 8 a 32-op integer chain; with the operands rotating over four 48 KB stages
// and the K step and first accumulate flag read at run time, as in the
// product: 9 descriptors formed between the MMAs, 10 the four MMAs from one
// asm block with their descriptors formed first
template <int kCode>
__device__ __forceinline__ void t8_loop(const PP &p, uint32_t tmem, uint64_t a0, uint64_t b0, uint32_t idesc,
                                        uint64_t *bars, const volatile uint32_t *vz, bool &ok) {
    const bool on = (p.flags >> (kCode - 2)) & 1;
    uint32_t x = 1;
    if constexpr (kCode >= 9) {
        const uint64_t da = 2 + (uint64_t)(p.flags & 1), db = 128 + (uint64_t)(p.flags & 2);
        for (int c = 0; c < p.iters; ++c) {
            const uint32_t so = (uint32_t)(c & 3) * (49152u >> 4);
            const uint64_t a = a0 + so, b = b0 + so;
            const uint32_t acc0 = (c & 15) ? 1u : (uint32_t)(p.flags >> 2) & 1u;
            if (kCode == 9) {
#pragma unroll
                for (int kk = 0; kk < 4; ++kk)
                    umma_f16_ss(tmem, a + kk * da, b + kk * db, idesc, kk > 0 ? 1u : acc0);
            } else {
                umma_f16_ss_x4(tmem, a, b, da, db, idesc, acc0);
            }
            umma_commit(&bars[c & 7]);
        }
    } else {
    for (int c = 0; c < p.iters; ++c) {
        uint32_t off = 0;
        if (on) {
            if (kCode == 2) tc_fence_after();
            if (kCode == 3) ok &= mbar_wait(&bars[14], 0, kLim, nullptr);
            if (kCode == 4) ok &= mbar_test_wait(&bars[14], 0);
            if (kCode == 5) fence_proxy_async_smem();
            if (kCode == 6) off += *vz;
            if (kCode == 7) p.out[4 * gridDim.x + (c & 255)] = clock64();
            if (kCode == 8) {
#pragma unroll
                for (int i = 0; i < 32; ++i)
                    asm volatile("mad.lo.u32 %0, %0, 3, %1;" : "+r"(x) : "r"((uint32_t)c));
                uint32_t z;
                asm volatile("and.b32 %0, %1, 0;" : "=r"(z) : "r"(x));
                off += z;
            }
        }
        umma_f16_ss(tmem, a0 + off, b0, idesc, 1u);
        umma_f16_ss(tmem, a0 + 2, b0 + 128, idesc, 1u);
        umma_f16_ss(tmem, a0 + 4, b0 + 256, idesc, 1u);
        umma_f16_ss(tmem, a0 + 6, b0 + 384, idesc, 1u);
        umma_commit(&bars[c & 7]);
    }
    }
}

__global__ void __launch_bounds__(320, 1) probe(const __grid_constant__ PP p) {
    extern __shared__ __align__(1024) uint8_t raw[];
    uint8_t *base = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(raw) + 1023) & ~(uintptr_t)1023);
    uint64_t *bars = reinterpret_cast<uint64_t *>(base + kData);
    uint32_t *tbase = reinterpret_cast<uint32_t *>(bars + 40);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int i = 0; i < 16; ++i) mbar_init(&bars[i], 1);
        // test 7: full[s] = bars[16 + s] (128 gather arrivals), wfull[s] = bars[24 + s],
        // empty[s] = bars[32 + s]
        {
            // test 7: arrivals per full barrier (per thread, or lane 0 of each warp)
            const int warps = (p.test == 7 && (p.flags & 16)) ? 8 : 4;
            const int per = (p.test == 7 && (p.flags & 192)) ? 1 : 32;
            for (int i = 16; i < 24; ++i) mbar_init(&bars[i], warps * per);
        }
        for (int i = 24; i < 40; ++i) mbar_init(&bars[i], 1);
        fence_mbar_init();
        tbase[1] = 0;           // test 3: the MMA thread's "done" flag
        tbase[2] = 0;           // test 8: a zero read from shared memory
    }
    for (int i = threadIdx.x; i < kData / 16; i += blockDim.x)
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
    } else if (p.test == 5) {
        // cp.async row gather alone: warps 0 .. nthreads-1 each keep two batches of
        // 16 rows x 512 bytes in flight; rows at a pitch of flags KB (0: 512 B,
        // contiguous rows) spread over N MB of global memory
        if (warp < p.nthreads) {
            const uint32_t dst = smem_u32(base + warp * 16384);
            const int64_t pitch = p.flags > 0 ? (int64_t)p.flags * 1024 : 512;
            const int64_t rows = ((int64_t)p.N << 20) / pitch;   // a power of two (checked on the host)
            const int64_t col = pitch > 512 ? (blockIdx.x % (pitch / 512)) * 512 : 0;
            const unsigned long long t0 = clock64();
            for (int it = 0; it < p.iters; ++it) {
#pragma unroll
                for (int r = 0; r < 16; ++r) {
                    const int64_t row =
                        ((int64_t)blockIdx.x * 7919 + (int64_t)it * 16 * 131 + r * 131 + warp * 104729) & (rows - 1);
                    cp_async_16_full(dst + (it & 1) * 8192 + r * 512 + lane * 16,
                                     p.W + row * pitch + col + lane * 16);
                }
                cp_async_commit();
                cp_async_wait_group<1>();
            }
            cp_async_wait_all();
            if (lane == 0) atomicAdd(&p.out[gridDim.x + blockIdx.x], (unsigned long long)p.iters * 8192);
            if (warp == 0 && lane == 0) p.out[2 * gridDim.x + blockIdx.x] = clock64() - t0;
        }
    } else if (p.test == 6) {
        // the product's copy mix without the tensor core: warps 0 .. nthreads-1
        // gather scattered 512-byte rows (as test 5, pitch 8 KB over N MB) while
        // warp 7 (one thread) streams 16 KB bulk copies, two in flight, until
        // the gathers finish (flag 1: no gathers, the bulk stream runs `iters`
        // x 8 copies; flag 2: no bulk copies).  out: bulk bytes, gather bytes,
        // gather cycles, bulk cycles.
        volatile int *done = reinterpret_cast<volatile int *>(tbase + 1);
        const bool gathers = !(p.flags & 1), bulks = !(p.flags & 2);
        if (warp < p.nthreads && gathers) {
            const uint32_t dst = smem_u32(base + warp * 16384);
            const int64_t pitch = 8192, rows = ((int64_t)p.N << 20) / pitch;
            const int64_t col = (blockIdx.x % 16) * 512;
            const unsigned long long t0 = clock64();
            for (int it = 0; it < p.iters; ++it) {
#pragma unroll
                for (int r = 0; r < 16; ++r) {
                    const int64_t row = ((int64_t)blockIdx.x * 7919 + (int64_t)it * 16 * 131 + r * 131 +
                                         warp * 104729) & (rows - 1);
                    cp_async_16_full(dst + (it & 1) * 8192 + r * 512 + lane * 16,
                                     p.W + row * pitch + col + lane * 16);
                }
                cp_async_commit();
                cp_async_wait_group<1>();
            }
            cp_async_wait_all();
            if (lane == 0) atomicAdd(&p.out[gridDim.x + blockIdx.x], (unsigned long long)p.iters * 8192);
            if (warp == 0 && lane == 0) {
                p.out[2 * gridDim.x + blockIdx.x] = clock64() - t0;
                *done = 1;
            }
        } else if (warp == 7 && lane == 0 && bulks) {
            const uint32_t dst = smem_u32(base + 7 * 16384);
            const int64_t tiles = ((int64_t)p.N << 20) / 16384;
            const int lim = gathers ? (1 << 22) : p.iters * 8;
            const unsigned long long t0 = clock64();
            bool ok = true;
            int n = 0;
            for (; n < lim && ok && (!gathers || !*done); ++n) {
                uint64_t *b = &bars[n & 1];
                if (n >= 2) ok = mbar_wait(b, (uint32_t)(((n >> 1) - 1) & 1), kLim, nullptr);
                if (!ok) break;
                mbar_arrive_expect_tx(b, 16384);
                bulk_g2s(dst, p.W + (((int64_t)blockIdx.x * 389 + (int64_t)n * 61) & (tiles - 1)) * 16384,
                         16384, b);
            }
            // the copies still in flight land before the CTA moves on
            for (int q = n > 2 ? n - 2 : 0; q < n; ++q)
                if (!mbar_wait(&bars[q & 1], (uint32_t)((q >> 1) & 1), kLim, nullptr)) ok = false;
            p.out[blockIdx.x] = (unsigned long long)n * 16384;
            p.out[3 * gridDim.x + blockIdx.x] = clock64() - t0;
            if (!ok) atomicOr(p.err, 128u);
        }
    } else if (p.test == 7) {
        // The product's stage ring without the tensor core, as the kernel runs
        // it: S stages of a weight tile (one bulk copy from a control thread) +
        // the chunk's activation rows of N tokens, gathered by one of two
        // groups of four warps (alternate chunks; 16 cp.async rows per warp
        // into the 128-byte-swizzled layout, cp.async.mbarrier.arrive.noinc),
        // and a consumer thread that waits for both and releases the stage.
        // X: 4096 rows x 4096 tokens, 16-bit.  Flags: 1 hold each stage 512
        // cycles (256 for half chunks) before releasing it, as the MMAs do;
        // 2 no weight copies; 4 rows anywhere (else sorted, about every fourth
        // row); 8 every CTA on token tile 0 (else blockIdx % 16); 16 all eight
        // warps gather every chunk; 32 half chunks (32 rows, 8 KB weight tile;
        // up to 8 stages); 64 / 128 other completion signals (below); 256
        // waits spin on test_wait; 512 / 1024 the gather warps poll for a free
        // stage from lane 0 only / with a back-off sleep; 2048 the consumer
        // releases a stage before its hold; 4096 it holds by sleeping in a
        // loop, 8192 with one sleep, 16384 with a chain of FMAs; 32768 two
        // chunks per stage (128 rows, 32 KB tile, 1,024-cycle hold, at most 2
        // stages).  Cycles per 64-row chunk.
        const int S = p.nthreads;
        const bool half = (p.flags & 32) != 0, all8 = (p.flags & 16) != 0;
        const bool dbl = (p.flags & 32768) != 0;          // two chunks per stage (128 rows)
        const int rows_per = half ? 32 : dbl ? 128 : 64;
        const uint32_t wbytes = half ? 8192u : dbl ? 32768u : 16384u;
        const uint32_t xbytes = half ? 16384u : dbl ? 65536u : 32768u;
        const uint32_t xcn = half ? 4096u : dbl ? 16384u : 8192u;   // bytes per 64-token group
        uint64_t *full = bars + 16, *wfull = bars + 24, *empty = bars + 32;
        const uint8_t *X = p.W;
        const int64_t n0 = (p.flags & 8) ? 0 : (int64_t)(blockIdx.x % 16) * 256;
        // a chunk's first row (one division per chunk, outside the row loop)
        const uint32_t span = (uint32_t)(4096 - 4 * rows_per);
        auto base_of = [&](int c) -> int64_t {
            return (int64_t)(((uint32_t)(c * 2654435761u) ^ (uint32_t)(blockIdx.x * 40503u)) % span);
        };
        auto row_of = [&](int c, int64_t b, int i) -> int64_t {
            const uint32_t h = (uint32_t)(c * 2654435761u) ^ (uint32_t)(blockIdx.x * 40503u) ^ (uint32_t)(i * 97u);
            if (p.flags & 4) return (int64_t)((h * 2246822519u) >> 20);                 // 0 .. 4095
            return b + 4 * i + ((h >> 7) & 3);                                            // < 4096
        };
        const int chunks = half ? 2 * p.iters : dbl ? p.iters / 2 : p.iters;
        // flag 256: every wait spins on mbarrier.test_wait instead of try_wait
        const bool spin = (p.flags & 256) != 0;
        auto wait = [&](uint64_t *bar, uint32_t parity) -> bool {
            if (!spin) return mbar_wait(bar, parity, kLim, nullptr);
            const uint64_t t0 = globaltimer_ns();
            for (uint32_t it = 1;; ++it) {
                if (mbar_test_wait(bar, parity)) return true;
                if ((it & 255u) == 0u && globaltimer_ns() - t0 > kLim) return false;
            }
        };
        if (warp < 8) {
            const int ngroups = all8 ? 1 : 2;
            const int g = all8 ? 0 : warp >> 2, gw = all8 ? warp : warp & 3, gwarps = all8 ? 8 : 4;
            const int cn = lane >> 3, jj = lane & 7;
            // signalling: arrive.noinc per thread (default); flag 64: commit
            // groups, the warp's previous chunk is signalled (one plain arrival
            // by lane 0) once wait_group<1> says it landed; flag 128: the warp
            // waits for its chunk's copies and signals it at once
            const bool lag = (p.flags & 64) != 0, sync = (p.flags & 128) != 0;
            bool ok = true;
            int prev = -1;
            for (int c = g; c < chunks && ok; c += ngroups) {
                const int s = c % S;
                if (c >= S) {
                    const uint32_t par = (uint32_t)(((c / S) & 1) ^ 1);
                    if (p.flags & 512) {
                        // lane 0 alone polls, the warp follows it
                        bool w = true;
                        if (lane == 0) w = wait(&empty[s], par);
                        ok = __shfl_sync(0xffffffffu, w ? 1 : 0, 0) != 0;
                        // every lane acquires the completed phase (no wait now)
                        if (ok) ok = __all_sync(0xffffffffu, wait(&empty[s], par));
                    } else if (p.flags & 1024) {
                        // polls with a back-off sleep between them
                        const uint64_t t0 = globaltimer_ns();
                        bool w = false;
                        for (uint32_t it = 1; !w; ++it) {
                            w = mbar_test_wait(&empty[s], par);
                            if (!w) __nanosleep(128);
                            if ((it & 255u) == 0u && globaltimer_ns() - t0 > kLim) break;
                        }
                        ok = __all_sync(0xffffffffu, w);
                    } else {
                        ok = __all_sync(0xffffffffu, wait(&empty[s], par));
                    }
                }
                if (!ok) break;
                unsigned long long *tr = p.out + 4 * gridDim.x + (int64_t)c * 4;
                const bool rec = blockIdx.x == 0 && gw == 0 && lane == 0 && c < 64;
                if (rec) tr[0] = clock64();
                const uint32_t xs = smem_u32(base + S * wbytes + s * xbytes);
                if (lane * 8 < p.N) {
                    const int64_t b = base_of(c);
                    for (int r = gw; r < rows_per; r += gwarps) {
                        const int64_t row = row_of(c, b, r);
                        cp_async_16_full(xs + cn * xcn + r * 128 + ((jj ^ (r & 7)) << 4),
                                         X + (row * 4096 + n0 + lane * 8) * 2);
                    }
                }
                if (rec) tr[1] = clock64();
                // every gather warp's issue time (CTA 0, first 32 chunks)
                if (blockIdx.x == 0 && lane == 0 && c < 32 && !all8)
                    p.out[4 * gridDim.x + 256 + c * 4 + gw] = clock64();
                if (lag) {
                    cp_async_commit();
                    cp_async_wait_group<1>();
                    __syncwarp();
                    if (prev >= 0 && lane == 0) mbar_arrive(&full[prev % S]);
                    prev = c;
                } else if (sync) {
                    cp_async_wait_all();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&full[s]);
                } else {
                    cp_async_arrive_noinc(&full[s]);
                }
            }
            cp_async_wait_all();
            __syncwarp();
            if (lag && prev >= 0 && lane == 0 && ok) mbar_arrive(&full[prev % S]);
            if (!ok) atomicOr(p.err, 256u);
        } else if (warp == 8 && lane == 0) {
            bool ok = true;
            for (int c = 0; c < chunks && ok; ++c) {
                const int s = c % S;
                if (c >= S) ok = wait(&empty[s], (uint32_t)(((c / S) & 1) ^ 1));
                if (!ok) break;
                if (p.flags & 2) {
                    mbar_arrive(&wfull[s]);
                } else {
                    mbar_arrive_expect_tx(&wfull[s], wbytes);
                    bulk_g2s(smem_u32(base + s * wbytes), X + ((int64_t)((c * 7 + blockIdx.x * 131) & 2047)) * 16384,
                             wbytes, &wfull[s]);
                }
            }
            if (!ok) atomicOr(p.err, 512u);
        } else if (warp == 9 && lane == 0) {
            bool ok = true;
            const long long hold = half ? 256 : dbl ? 1024 : 512;
            const unsigned long long t0 = clock64();
            for (int c = 0; c < chunks && ok; ++c) {
                const int s = c % S;
                const uint32_t ph = (uint32_t)((c / S) & 1);
                unsigned long long *tq = p.out + 4 * gridDim.x + 448 + (int64_t)c * 4;
                if (blockIdx.x == 0 && c < 64) tq[0] = clock64();
                ok = wait(&wfull[s], ph);
                if (blockIdx.x == 0 && c < 64) tq[1] = clock64();
                ok = ok && wait(&full[s], ph);
                if (blockIdx.x == 0 && c < 64) tq[2] = clock64();
                if (!ok) break;
                unsigned long long *tr = p.out + 4 * gridDim.x + (int64_t)c * 4;
                if (blockIdx.x == 0 && c < 64) tr[2] = clock64();
                // CTA 0: was the next stage's data already complete before this
                // stage's hold began (1), or only later (0)?
                if (blockIdx.x == 0 && c < 64 && c + 1 < chunks) {
                    const int s1 = (c + 1) % S;
                    const uint32_t ph1 = (uint32_t)(((c + 1) / S) & 1);
                    p.out[4 * gridDim.x + 384 + c] =
                        (mbar_test_wait(&wfull[s1], ph1) && mbar_test_wait(&full[s1], ph1)) ? 1ull : 0ull;
                }
                // flag 2048: release the stage first, then hold (the hold then
                // delays only the consumer); flag 4096: hold by sleeping
                if (p.flags & 2048) mbar_arrive(&empty[s]);
                if ((p.flags & 1) && (p.flags & 8192)) {
                    __nanosleep((unsigned)(hold / 2));          // one sleep of about the hold
                } else if ((p.flags & 1) && (p.flags & 16384)) {
                    // a dependent chain of ~hold / 4 FMAs, no clock reads
                    float a = (float)c;
                    for (int k = 0; k < (int)(hold / 4); ++k) a = fmaf(a, 1.0001f, 0.5f);
                    if (a == 12345.f) atomicOr(p.err, 0u);
                } else if (p.flags & 1) {
                    const long long h0 = clock64();
                    while (clock64() - h0 < hold) {
                        if (p.flags & 4096) __nanosleep(32);
                    }
                }
                if (blockIdx.x == 0 && c < 64) tr[3] = clock64();
                if (!(p.flags & 2048)) mbar_arrive(&empty[s]);
                if (blockIdx.x == 0 && c < 64) tq[3] = clock64();
            }
            p.out[blockIdx.x] = clock64() - t0;
            if (!ok) atomicOr(p.err, 1024u);
        }
    } else if (p.test == 4) {
        // back-to-back MMAs in groups of `per` (2, 4 or 8), a commit after each
        // group (flag 2: none), groups alternating between two accumulators
        // (flag 1); nothing waits on the commits until the end
        if (threadIdx.x == 0) {
            const uint32_t idesc = make_idesc(true, false, true, 128, p.N);
            const uint64_t a0 = make_sdesc_sw128(smem_u32(base), 16, 1024);
            const uint64_t b0 = make_sdesc_sw128(smem_u32(base + 16384), 8192, 1024);
            const int per = p.nthreads;
            const unsigned long long t0 = clock64();
            for (int c = 0; c < p.iters; ++c) {
                const uint32_t d = tmem + ((p.flags & 1) ? (uint32_t)(c & 1) * 256u : 0u);
                if (per == 2) {
#pragma unroll
                    for (int kk = 0; kk < 2; ++kk) umma_f16_ss(d, a0 + kk * 2, b0 + kk * 128, idesc, 1u);
                } else if (per == 4) {
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk) umma_f16_ss(d, a0 + kk * 2, b0 + kk * 128, idesc, 1u);
                } else {
#pragma unroll
                    for (int kk = 0; kk < 8; ++kk)
                        umma_f16_ss(d, a0 + (kk & 3) * 2, b0 + (kk & 3) * 128, idesc, 1u);
                }
                if (!(p.flags & 2)) umma_commit(&bars[c & 7]);
            }
            umma_commit(&bars[15]);
            const bool ok = mbar_wait(&bars[15], 0, kLim, nullptr);
            p.out[blockIdx.x] = clock64() - t0;
            if (!ok) atomicOr(p.err, 64u);
        }
    } else if (p.test == 8) {
        if (threadIdx.x == 0) {
            mbar_arrive(&bars[14]);     // completes its phase 0
            const uint32_t idesc = make_idesc(true, false, true, 128, p.N);
            const uint64_t a0 = make_sdesc_sw128(smem_u32(base), 16, 1024);
            const uint64_t b0 = make_sdesc_sw128(smem_u32(base + 16384), 8192, 1024);
            const volatile uint32_t *vz = tbase + 2;
            const int f = p.flags;
            uint32_t x = 1;
            bool ok = true;
            unsigned long long issue = 0;
            auto work = [&](int c, uint32_t &off) {
                if (f & 1) tc_fence_after();
                if (f & 2) fence_proxy_async_smem();
                if (f & 4) ok &= mbar_wait(&bars[14], 0, kLim, nullptr);
                if (f & 8) ok &= mbar_test_wait(&bars[14], 0);
                if (f & 16) off += *vz;
                if (f & 32) {
#pragma unroll
                    for (int i = 0; i < 32; ++i)
                        asm volatile("mad.lo.u32 %0, %0, 3, %1;" : "+r"(x) : "r"((uint32_t)c));
                    uint32_t z;
                    asm volatile("and.b32 %0, %1, 0;" : "=r"(z) : "r"(x));
                    off += z;
                }
                if (f & 64) p.out[4 * gridDim.x + (c & 255)] = clock64();
                if (f & 128) ok &= !mbar_test_wait(&bars[13], 0);
            };
            const unsigned long long t0 = clock64();
            if (p.nthreads >= 2) {
                switch (p.nthreads) {
                    case 2: t8_loop<2>(p, tmem, a0, b0, idesc, bars, vz, ok); break;
                    case 3: t8_loop<3>(p, tmem, a0, b0, idesc, bars, vz, ok); break;
                    case 4: t8_loop<4>(p, tmem, a0, b0, idesc, bars, vz, ok); break;
                    case 5: t8_loop<5>(p, tmem, a0, b0, idesc, bars, vz, ok); break;
                    case 6: t8_loop<6>(p, tmem, a0, b0, idesc, bars, vz, ok); break;
                    case 7: t8_loop<7>(p, tmem, a0, b0, idesc, bars, vz, ok); break;
                    case 8: t8_loop<8>(p, tmem, a0, b0, idesc, bars, vz, ok); break;
                    case 9: t8_loop<9>(p, tmem, a0, b0, idesc, bars, vz, ok); break;
                    default: t8_loop<10>(p, tmem, a0, b0, idesc, bars, vz, ok); break;
                }
            } else if (f & 256) {
                // the work between the group's second and third MMA
                for (int c = 0; c < p.iters; ++c) {
                    uint32_t off = 0;
                    umma_f16_ss(tmem, a0, b0, idesc, 1u);
                    umma_f16_ss(tmem, a0 + 2, b0 + 128, idesc, 1u);
                    work(c, off);
                    umma_f16_ss(tmem, a0 + 4 + off, b0 + 256, idesc, 1u);
                    umma_f16_ss(tmem, a0 + 6, b0 + 384, idesc, 1u);
                    umma_commit(&bars[c & 7]);
                }
            } else if (f & 512) {
                for (int c = 0; c < p.iters; ++c) {
                    uint32_t off = 0;
                    const unsigned long long ti = clock64();
                    work(c, off);
                    umma_f16_ss(tmem, a0 + off, b0, idesc, 1u);
                    umma_f16_ss(tmem, a0 + 2, b0 + 128, idesc, 1u);
                    umma_f16_ss(tmem, a0 + 4, b0 + 256, idesc, 1u);
                    umma_f16_ss(tmem, a0 + 6, b0 + 384, idesc, 1u);
                    umma_commit(&bars[c & 7]);
                    issue += clock64() - ti;
                }
            } else if (f & 8192) {
                for (int c = 0; c < p.iters; ++c) {
                    if (f & 16384) {
#pragma unroll
                        for (int k = 0; k < 8; ++k)
                            if (c == -1 - k * p.iters) asm volatile("nanosleep.u32 0;");
                    }
                    umma_f16_ss(tmem, a0, b0, idesc, 1u);
                    umma_f16_ss(tmem, a0 + 2, b0 + 128, idesc, 1u);
                    umma_f16_ss(tmem, a0 + 4, b0 + 256, idesc, 1u);
                    umma_f16_ss(tmem, a0 + 6, b0 + 384, idesc, 1u);
                    umma_commit(&bars[c & 7]);
                }
            } else if (f & 4096) {
                // stage st: A at st * 48 KB, B 16 KB after it (descriptor units of 16 B)
                for (int c = 0; c < p.iters; ++c) {
                    uint32_t off = 0;
                    work(c, off);
                    const uint32_t so = (uint32_t)(c & 3) * (49152u >> 4);
                    const uint64_t a = make_sdesc_sw128(smem_u32(base), 16, 1024) + so;
                    const uint64_t b = make_sdesc_sw128(smem_u32(base + 16384), 8192, 1024) + so;
                    umma_f16_ss(tmem, a + off, b, idesc, 1u);
                    umma_f16_ss(tmem, a + 2, b + 128, idesc, 1u);
                    umma_f16_ss(tmem, a + 4, b + 256, idesc, 1u);
                    umma_f16_ss(tmem, a + 6, b + 384, idesc, 1u);
                    umma_commit(&bars[c & 7]);
                }
            } else {
                for (int c = 0; c < p.iters; ++c) {
                    uint32_t off = 0;
                    work(c, off);
                    umma_f16_ss(tmem, a0 + off, b0, idesc, 1u);
                    umma_f16_ss(tmem, a0 + 2, b0 + 128, idesc, 1u);
                    umma_f16_ss(tmem, a0 + 4, b0 + 256, idesc, 1u);
                    umma_f16_ss(tmem, a0 + 6, b0 + 384, idesc, 1u);
                    umma_commit(&bars[c & 7]);
                }
            }
            umma_commit(&bars[15]);
            ok &= mbar_wait(&bars[15], 0, kLim, nullptr);
            p.out[blockIdx.x] = clock64() - t0;
            p.out[gridDim.x + blockIdx.x] = issue;
            *reinterpret_cast<volatile uint32_t *>(tbase + 1) = 1u;
            if (!ok) atomicOr(p.err, 128u);
        } else if (warp >= 2 && (p.flags & 1024)) {
            // pollers: a barrier nobody arrives on, until the MMA thread is done
            const volatile uint32_t *done = tbase + 1;
            const uint32_t a = smem_u32(&bars[12]);
            for (int it = 0; it < (1 << 24) && !*done; ++it) (void)mbar_try_wait(a, 0);
        } else if (warp >= 2 && warp <= 7 && (p.flags & 2048)) {
            // copiers: 16 rows of 512 B per batch into their own 8 KB areas
            const volatile uint32_t *done = tbase + 1;
            const uint32_t dst = smem_u32(base + 65536 + (warp - 2) * 8192);
            for (int it = 0; it < (1 << 20) && !*done; ++it) {
#pragma unroll
                for (int r = 0; r < 16; ++r) {
                    const int64_t row = ((int64_t)blockIdx.x * 131 + it * 16 + r + warp * 977) % 16384;
                    cp_async_16_full(dst + r * 512 + lane * 16, p.W + row * 512 + lane * 16);
                }
                cp_async_wait_all();
            }
        }
    } else if (p.test == 2) {
        // stage ring without data: full[s] = bars[s], empty[s] = bars[8 + s]
        const int S = p.nthreads;
        uint64_t *full = bars, *empty = bars + 8;
        if (threadIdx.x == 0) {
            const uint32_t idesc = make_idesc(true, false, true, 128, p.N);
            const uint64_t a0 = make_sdesc_sw128(smem_u32(base), 16, 1024);
            const uint64_t b0 = make_sdesc_sw128(smem_u32(base + 16384), 8192, 1024);
            const unsigned long long t0 = clock64();
            bool ok = true;
            const bool nowait = (p.flags & 4) != 0;
            const int per = (p.flags >> 8) & 15 ? (p.flags >> 8) & 15 : 4;   // MMAs per stage
            for (int c = 0; c < p.iters && ok; ++c) {
                const int s = c % S;
                if (!nowait) ok = mbar_wait(&full[s], (uint32_t)((c / S) & 1), kLim, nullptr);
                if (!ok) break;
                if (p.flags & 1) tc_fence_after();
                if (p.flags & 2) fence_proxy_async_smem();
                for (int kk = 0; kk < per; ++kk)
                    umma_f16_ss(tmem, a0 + (kk & 3) * 2, b0 + (kk & 3) * 128, idesc, 1u);
                umma_commit(&empty[s]);
            }
            const int last = p.iters - 1;
            if (ok) ok = mbar_wait(&empty[last % S], (uint32_t)((last / S) & 1), kLim, nullptr);
            p.out[blockIdx.x] = clock64() - t0;
            if (!ok) atomicOr(p.err, 4u);
        } else if (threadIdx.x == 32 && !(p.flags & 4)) {
            bool ok = true;
            for (int c = 0; c < p.iters && ok; ++c) {
                const int s = c % S;
                if (c >= S) ok = mbar_wait(&empty[s], (uint32_t)(((c / S) & 1) ^ 1), kLim, nullptr);
                if (ok) mbar_arrive(&full[s]);
            }
            if (!ok) atomicOr(p.err, 8u);
        }
    } else if (p.test == 3) {
        // back-to-back MMAs (warp 0) against copies from warps 1 .. nthreads
        volatile int *done = reinterpret_cast<volatile int *>(tbase + 1);
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
            umma_commit(&bars[15]);
            const bool ok = mbar_wait(&bars[15], 0, kLim, nullptr);
            p.out[blockIdx.x] = clock64() - t0;
            *done = 1;
            if (!ok) atomicOr(p.err, 16u);
        } else if (warp >= 1 && warp <= p.nthreads) {
            const int t = warp;
            // destination: 16 KB per copying warp in the area past the operands
            const uint32_t dst = smem_u32(base + 65536 + ((t - 1) & 3) * 16384);
            unsigned long long bytes = 0;
            const unsigned long long t0 = clock64();
            bool ok = true;
            if (p.flags & 4) {
                // cp.async rows: 16 rows of 512 bytes per batch, lanes 16 bytes each
                for (int it = 0; it < (1 << 20) && !*done; ++it) {
#pragma unroll
                    for (int r = 0; r < 16; ++r) {
                        const int64_t row = ((int64_t)blockIdx.x * 131 + it * 16 + r + t * 977) % 16384;
                        cp_async_16_full(dst + r * 512 + lane * 16, p.W + row * 512 + lane * 16);
                    }
                    cp_async_wait_all();
                    bytes += 16 * 512;
                }
            } else if (lane == 0) {
                uint64_t *b = &bars[t * 2 - 2];
                for (int it = 0; it < (1 << 20) && !*done && ok; ++it) {
                    mbar_arrive_expect_tx(b, 16384);
                    bulk_g2s(dst, p.W + (((int64_t)blockIdx.x * 97 + it + t * 1000) % 512) * 16384,
                             16384, b);
                    ok = mbar_wait(b, (uint32_t)(it & 1), kLim, nullptr);
                    bytes += 16384;
                }
            }
            if (lane == 0) atomicAdd(&p.out[gridDim.x + blockIdx.x], bytes);
            if (t == 1 && lane == 0) p.out[2 * gridDim.x + blockIdx.x] = clock64() - t0;
            if (!ok) atomicOr(p.err, 32u);
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
    const int flags = argc > 5 ? atoi(argv[5]) : 0;
    if (N < 16 || N > 256 || N % 16 || nth < 1 || nth > (test == 8 ? 10 : 8) || iters < 1 || test < 0 ||
        test > 8)
        return 2;
    if (test != 4 && test != 5 && test != 6 && test != 7 && test != 8 && nth > 6) return 2;
    if (test == 7 && (nth < 2 || nth > ((flags & 32) ? 8 : (flags & 32768) ? 2 : 4) ||
                      (N != 128 && N != 256) || flags < 0 || flags > 65535 || (flags & 192) == 192 ||
                      ((flags & 64) && nth < 4) || ((flags & 32) && (flags & 32768)))) return 2;
    if (test == 5 && (flags < 0 || flags > 64 || (flags & (flags - 1)) || (N & (N - 1)))) return 2;
    if (test == 6 && (nth > 6 || flags < 0 || flags > 2 || N < 64 || (N & (N - 1)))) return 2;
    if (test == 4 && nth != 2 && nth != 4 && nth != 8) return 2;   // MMAs per group
    if (test == 2 && (nth < 2 || nth > 6)) return 2;     // stages
    if (test == 8 && (flags < 0 || flags > 32767 || (flags & 3072) == 3072 ||
                      ((flags & 4096) && (flags & 2048)))) return 2;
    int sms = 0;
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, 0);
    uint8_t *W = nullptr;
    const size_t wbytes = (test == 5 || test == 6) ? ((size_t)N << 20)
                          : test == 7 ? ((size_t)32 << 20) : (size_t)512 * 16384;
    cudaMalloc(&W, wbytes);
    cudaMemset(W, 0, wbytes);
    unsigned long long *out = nullptr;
    unsigned *err = nullptr;
    cudaMalloc(&out, (4 * sms + 704) * 8);
    cudaMalloc(&err, 4);
    cudaMemset(err, 0, 4);
    PP p{test, iters, N, nth, flags, W, out, err};
    const int smem = 1024 + kData + 1024;
    cudaFuncSetAttribute(probe, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    for (int w = 0; w < 3; ++w) {
        cudaMemset(out, 0, (4 * sms + 704) * 8);
        probe<<<sms, 320, smem>>>(p);
        if (cudaDeviceSynchronize() != cudaSuccess) {
            printf("cuda error\n");
            return 4;
        }
    }
    std::vector<unsigned long long> h(4 * sms);
    unsigned herr = 0;
    cudaMemcpy(h.data(), out, 4 * sms * 8, cudaMemcpyDeviceToHost);
    cudaMemcpy(&herr, err, 4, cudaMemcpyDeviceToHost);
    double avg = 0, byt = 0, cyc = 0, bcyc = 0;
    for (int i = 0; i < sms; ++i) {
        avg += h[i];
        byt += h[sms + i];
        cyc += h[2 * sms + i];
        bcyc += h[3 * sms + i];
    }
    avg /= sms;
    if (test == 0)
        printf("tcgen05.mma 128 x %d x 16: %.1f cycles per instruction (err %u)\n", N,
               avg / (iters * 16.0), herr);
    else if (test == 1)
        printf("bulk copies from %d thread(s): %.1f bytes per cycle per SM (err %u)\n", nth,
               nth * 16384.0 * 4 * iters / avg, herr);
    else if (test == 2)
        printf("stage ring, %d stages, fences %d%s, %d x (128 x %d x 16) per stage: %.1f cycles per "
               "stage (err %u)\n", nth, flags & 3, (flags & 4) ? ", no waits" : "",
               (flags >> 8) & 15 ? (flags >> 8) & 15 : 4, N, avg / iters, herr);
    else if (test == 7) {
        printf("stage ring with data, %d stages, %d tokens, flags %d: %.1f cycles per chunk (err %u)\n",
               nth, N, flags, avg / iters, herr);
        if (getenv("TC_RING_TRACE")) {
            // CTA 0: per chunk, producer saw the stage free / issued, consumer saw the data / released
            std::vector<unsigned long long> t(704);
            cudaMemcpy(t.data(), out + 4 * sms, 704 * 8, cudaMemcpyDeviceToHost);
            // consumer: release -> (loop) -> wfull wait done -> full wait done
            for (int c = 10; c < 14; ++c)
                printf("  consumer chunk %d: arrive %lld, to next wait start %lld, wfull wait %lld, full wait %lld\n", c,
                       (long long)(t[448 + 4 * c + 3] - t[4 * c + 3]),
                       (long long)(t[448 + 4 * (c + 1)] - t[448 + 4 * c + 3]),
                       (long long)(t[448 + 4 * (c + 1) + 1] - t[448 + 4 * (c + 1)]),
                       (long long)(t[448 + 4 * (c + 1) + 2] - t[448 + 4 * (c + 1) + 1]));
            int ready = 0;
            for (int c = 8; c < 40; ++c) ready += (int)t[384 + c];
            printf("  next stage already complete before the hold: %d of 32 chunks\n", ready);
            const unsigned long long z = t[2];
            for (int c = 0; c < 32; ++c)
                printf("  chunk %2d: free %7lld issued %7lld data %7lld released %7lld; warps issued "
                       "%7lld %7lld %7lld %7lld\n", c,
                       (long long)(t[4 * c] - z), (long long)(t[4 * c + 1] - z),
                       (long long)(t[4 * c + 2] - z), (long long)(t[4 * c + 3] - z),
                       (long long)(t[256 + 4 * c] - z), (long long)(t[256 + 4 * c + 1] - z),
                       (long long)(t[256 + 4 * c + 2] - z), (long long)(t[256 + 4 * c + 3] - z));
        }
    }
    else if (test == 6)
        printf("copy mix over %d MB: %d gather warp(s)%s, %s: gathers %.1f, bulk %.1f bytes per "
               "cycle per SM (err %u)\n", N, (flags & 1) ? 0 : nth, "", (flags & 2) ? "no bulk stream"
               : "one bulk-copy thread", cyc > 0 ? byt / cyc : 0.0, bcyc > 0 ? avg * sms / bcyc : 0.0, herr);
    else if (test == 5)
        printf("cp.async rows of 512 B from %d warp(s), pitch %d B over %d MB: %.1f bytes per cycle "
               "per SM (err %u)\n", nth, flags > 0 ? flags * 1024 : 512, N, cyc > 0 ? byt / cyc : 0.0, herr);
    else if (test == 8)
        printf("mma groups of 4 x (128 x %d x 16) + commit, per-group work %d (code %d): %.1f cycles per "
               "group, %.1f to issue one (err %u)\n", N, flags, nth, avg / iters, byt / sms / iters, herr);
    else if (test == 4)
        printf("mma 128 x %d x 16 in groups of %d, %s, %s: %.1f cycles per instruction (err %u)\n",
               N, nth, (flags & 2) ? "no commits" : "a commit per group",
               (flags & 1) ? "two accumulators" : "one accumulator", avg / ((double)iters * nth), herr);
    else
        printf("mma 128 x %d x 16 with %d %s copier warp(s): %.1f cycles per instruction, "
               "%.1f bytes per cycle per SM copied (err %u)\n", N, nth,
               (flags & 4) ? "cp.async" : "bulk", avg / (iters * 16.0), cyc > 0 ? byt / cyc : 0.0,
               herr);
    return herr ? 5 : 0;
}
