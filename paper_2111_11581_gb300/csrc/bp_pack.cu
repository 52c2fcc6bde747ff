// Packing kernels: mask -> per-row-block kept-column counts (with the check
// that all rows of a row-block agree, the BCS occurrence property of
// Sec. 4.3), then col_idx / values (the canonical compact arrays) and the
// device image the tensor-core kernels stream: per row-block k-chunks of 64
// kept columns, each a (rows_pad x 64) K-major tile already in the 128-byte
// swizzled shared-memory order, plus the padded column list of every chunk.
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

// Padded column list of every k-chunk: entry r of chunk kc of row-block rb is
// its (kc*64 + r)-th kept column; past K'_rb it repeats the row-block's last
// kept column (a valid row to load, multiplied by the zero-padded weights).
__global__ void cidx_kernel(const int64_t *__restrict__ rb_ptr, const int64_t *__restrict__ kc_ptr,
                            const int32_t *__restrict__ col_idx, uint8_t *__restrict__ chunks,
                            int64_t tile_bytes, int64_t chunk_bytes) {
    const int64_t rb = blockIdx.x;
    const int64_t p0 = rb_ptr[rb], kp = rb_ptr[rb + 1] - p0;
    const int64_t c0 = kc_ptr[rb], nkc = kc_ptr[rb + 1] - c0;
    for (int64_t t = threadIdx.x; t < nkc * kBK; t += blockDim.x) {
        int32_t *cl = reinterpret_cast<int32_t *>(chunks + (c0 + t / kBK) * chunk_bytes + tile_bytes);
        cl[t % kBK] = col_idx[p0 + (t < kp ? t : kp - 1)];
    }
}

// Tiles: one thread per 16-byte unit (8 consecutive k of one row).
__global__ void tiles_kernel(int64_t M, int64_t bm, int64_t rows_pad,
                             const int64_t *__restrict__ rb_ptr,
                             const int64_t *__restrict__ kc_ptr,
                             const uint16_t *__restrict__ values, uint8_t *__restrict__ chunks,
                             int64_t chunk_bytes) {
    const int64_t rb = blockIdx.y;
    const int64_t p0 = rb_ptr[rb], kp = rb_ptr[rb + 1] - p0;
    const int64_t c0 = kc_ptr[rb], nkc = kc_ptr[rb + 1] - c0;
    const int64_t rows = min(bm, M - rb * bm);
    const int64_t units = nkc * rows_pad * (kBK / 8);
    for (int64_t u = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; u < units;
         u += (int64_t)gridDim.x * blockDim.x) {
        const int64_t kc = u / (rows_pad * (kBK / 8));
        const int64_t rem = u % (rows_pad * (kBK / 8));
        const uint32_t row = (uint32_t)(rem / (kBK / 8));
        const uint32_t ch = (uint32_t)(rem % (kBK / 8));
        uint16_t v[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const int64_t k = kc * kBK + ch * 8 + e;
            v[e] = (row < rows && k < kp) ? values[bm * p0 + row * kp + k] : (uint16_t)0;
        }
        uint4 pk;
        pk.x = v[0] | ((uint32_t)v[1] << 16);
        pk.y = v[2] | ((uint32_t)v[3] << 16);
        pk.z = v[4] | ((uint32_t)v[5] << 16);
        pk.w = v[6] | ((uint32_t)v[7] << 16);
        uint8_t *tile = chunks + (c0 + kc) * chunk_bytes;
        *reinterpret_cast<uint4 *>(tile + sw128_kmajor_offset(row, ch * 8)) = pk;
    }
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
    if (e != cudaSuccess || dl.orient == kNoTensorCore) return e;
    uint8_t *dev = static_cast<uint8_t *>(P.dev);
    const int64_t *kc_ptr = reinterpret_cast<const int64_t *>(dev);
    uint8_t *chunks = dev + dl.off_chunks;
    cidx_kernel<<<(unsigned)RB, 256, 0, s>>>(P.rb_ptr, kc_ptr, P.col_idx, chunks, dl.tile_bytes,
                                             dl.chunk_bytes);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    dim3 grid(8, (unsigned)RB);
    tiles_kernel<<<grid, 256, 0, s>>>(lay.M, lay.bm, dl.rows_pad, P.rb_ptr, kc_ptr,
                                      static_cast<const uint16_t *>(P.values), chunks,
                                      dl.chunk_bytes);
    return cudaGetLastError();
}

}  // namespace bp
