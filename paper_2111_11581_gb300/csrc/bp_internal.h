// Internal interfaces between the translation units of libbp (not exported).
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda_runtime.h>

#include "bp.h"

namespace bp {

// Device status bits recorded by kernels (read by bp_device_status).
constexpr unsigned kDevTimeout = 1u;

// Tile geometry of the tensor-core kernels.
constexpr int kBK = 64;            // GEMM-view columns per k-chunk (one 128-B swizzle row)
constexpr int kSlab = 128;         // weight rows per MMA when W is the A operand

// Which operand the compact weights are in the tensor-core product.
//   kWeightA: W rows are the MMA M dimension (bm a multiple of 128), the
//             gathered activations are the N = 256 operand.
//   kWeightB: 128 gathered activation columns (tokens / pixels) are the MMA M
//             dimension, W rows are N (bm <= 256, padded to a multiple of 16).
enum Orientation { kWeightA = 0, kWeightB = 1, kNoTensorCore = 2 };

// Device image inside bp_packed::dev (all offsets in bytes):
//   [0, 8*(num_rb+1))         int64 kc_ptr: first k-chunk of each row-block
//   off_chunks + c*chunk_bytes  k-chunk c: its (rows_pad x 64) 16-bit weight
//                               tile in K-major 128-byte-swizzled order,
//                               followed by its 64 int32 column indices
//                               (padding repeats the last kept column; its
//                               weights are zero).
struct DevLayout {
    Orientation orient;
    int64_t rows_pad;     // rows per k-chunk tile
    int64_t num_rb;
    int64_t kc_total;     // total k-chunks over all row-blocks (-1 if unknown)
    int64_t off_chunks;
    int64_t tile_bytes;   // rows_pad * 64 * 2
    int64_t chunk_bytes;  // tile_bytes + 64 * 4
    int64_t bytes;        // total image size (when kc_total is known)
};

Orientation orientation_for(int64_t bm);
int64_t rows_pad_for(int64_t bm);
// Image layout for a layout and its per-row-block kept-column counts
// (rb_ptr_host = host copy of rb_ptr, or nullptr to leave kc_total unknown).
DevLayout dev_layout(const bp_layout &lay, const int64_t *rb_ptr_host);

// Library-wide settings.
uint64_t watchdog_ns();
int64_t debug_drop_stage();     // -1 = no fault injection
unsigned *device_status_ptr();   // device address of the status word
int num_sms();
bool checked_mode();

// Launchers (return cudaError_t of the launch).
cudaError_t launch_scores(const bp_layout &lay, const void *W, double *scores, int *nonfinite,
                          cudaStream_t s);
cudaError_t launch_base_select(const bp_layout &lay, const double *scores, double rate,
                               uint8_t *keep, cudaStream_t s);
cudaError_t launch_radix_hist(int64_t U, const double *scores, const uint8_t *keep,
                              uint64_t prefix, int shift, unsigned *hist, cudaStream_t s);
cudaError_t launch_threshold_select(int64_t U, const double *scores, uint8_t *keep,
                                    uint64_t thr, int64_t need, int64_t *chunk_cnt,
                                    cudaStream_t s);
cudaError_t launch_write_mask(const bp_layout &lay, const uint8_t *keep, uint8_t *mask,
                              cudaStream_t s);
int64_t threshold_chunks(int64_t U);

cudaError_t launch_rb_counts(const bp_layout &lay, const uint8_t *mask, int64_t *rb_ptr,
                             int *bad, cudaStream_t s);
cudaError_t launch_pack(const bp_layout &lay, const void *W, const uint8_t *mask,
                        const bp_packed &P, const DevLayout &dl, cudaStream_t s);

struct ConvShape {
    int64_t Nb, C, H, W, Ho, Wo;
    int kh, kw, ph, pw, sh, sw;
};
cudaError_t launch_mma(const bp_packed &P, const DevLayout &dl, const void *X, int64_t N,
                       int64_t ldx, const float *bias, int relu, void *Y, int64_t ldy,
                       const ConvShape *conv, cudaStream_t s);

}  // namespace bp
