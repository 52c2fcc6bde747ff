// Internal interfaces between the translation units of libbp (not exported).
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include "bp.h"

namespace bp {

// Internal scheme value of the prune kernels: the row units of a block-based
// layout (rows of each bm x bk block; written into the mask with AND).
constexpr int kSchemeRows = 2;
// ... and the kernels of a 3x3 layer for pattern-based pruning (one unit per
// (filter, channel) kernel, scored by its best pattern's kept norm).
constexpr int kSchemePattern = 3;
constexpr int kMaxPatterns = 16;
struct PatternSet {
    uint16_t m[kMaxPatterns];   // 9-bit masks, 4 bits set, pos = 3i + j
    int n;
};

// Device status bits recorded by kernels (read by bp_device_status).
constexpr unsigned kDevTimeout = 1u;

// Tile geometry of the tensor-core kernel.
constexpr int kBK = 64;            // GEMM-view columns per k-chunk (one 128-B swizzle row)
constexpr int kSlab = 128;         // weight rows per slab (the MMA's M)

constexpr int kDenseMin = 48;      // a 64-column block whose union keeps >= this many columns is stored whole
constexpr int64_t kMaxSlabs = 8192;  // 128-row slabs per layer (M <= 1,048,576)
constexpr int kListBytes = kBK * 4;  // a chunk's 64 int32 column indices
constexpr int kPlanBytes = 64;       // a chunk's load plan
constexpr int kMetaBytes = kListBytes + kPlanBytes;   // list + plan record of a chunk
constexpr int kMaxBoxes = 8;         // tile loads in a chunk's plan at most

// Device image inside bp_packed::dev, the form the tensor-core kernel streams.
// Rows are grouped in slabs of 128 (slab s = rows 128s .. 128s+127); a slab's
// column list is the union of the kept columns of its rows (all rows of a
// row-block keep the same columns, so for bm a multiple of 128 it is exactly
// the row-block's list).  Aligned 64-column blocks whose union holds at least
// kDenseMin columns are listed whole (64 consecutive columns, weights zero
// where a row prunes them); the other union columns follow in ascending
// order, 64 per k-chunk.  All offsets in bytes, C = total k-chunks:
//   [0, 8*(S+1))                 int64 kc_ptr: first k-chunk of each slab
//   [8*(S+1), 8*(S+2))           int64 Kc: number of columns any slab lists
//   off_tiles + c*16384          k-chunk c's 128 x 64 16-bit weight tile in
//                                K-major 128-byte-swizzled order
//   off_meta + c*kMetaBytes      k-chunk c's record:
//     [0, 256)                   its 64 int32 column indices (a partial last
//                                chunk repeats its last index; the weights of
//                                such repeats are zero);
//     [256, 320)                 its load plan, int32 words: [0] = number of
//                                tile loads B (0: gather the rows one by one),
//                                [1 + b] = first column of load b, [9], [10] =
//                                one byte per load: bits 0-2 = first list
//                                position / 8, bits 4-5 = log2(rows / 8); the
//                                loads cover the 64 list positions in order,
//                                and each live entry of a load's range is its
//                                first column plus its offset (repeats read
//                                other rows, against zero weights).
//   off_meta2 + c*kMetaBytes     the same record in compacted coordinates: list
//                                entries replaced by their rank among the Kc
//                                listed columns (qmap), plan built from those,
//                                with no load reaching past row Kc - 1.  A
//                                convolution writes only the Kc listed rows of
//                                its im2col matrix, in that order.
//   off_qmap + 4*k               int32 qmap[k]: rank of column k among the
//                                listed columns, -1 if no slab lists it.
//
//
// Layers with kh * kw > 1 carry a third section, the same slabs in the form
// the implicit convolution streams.  There a chunk is one K-group: 64
// consecutive input channels at one kernel position, (c64, i, j), i.e. the
// GEMM-view columns (64 c64 + u) kh kw + i kw + j, u < 64 (channels past C
// have zero weights).  Per slab, the K-groups any of its rows keeps are listed
// position-major ((i, j), then c64).  The section is sized for every K-group
// listed (c3max chunks), so its size follows from the layout:
//   off_sec3                     int64 kc3_ptr[S+1]: first chunk of each slab
//   off_tiles3 + c*16384         chunk c's 128 x 64 weight tile, K-major with
//                                the 128-byte swizzle; column u = channel
//                                64 c64 + u
//   off_meta3 + c*kMetaBytes     chunk c's record: int32 word [0] its K-group
//                                (c64 << 16 | i << 8 | j), [64] = 1 (every
//                                chunk is loaded with TMA)
struct DevLayout {
    int64_t num_slabs;
    int64_t kc_total;     // total k-chunks (-1 if unknown)
    int64_t off_tiles;
    int64_t off_meta;     // (this and the following when kc_total is known)
    int64_t off_meta2;
    int64_t off_qmap;
    int64_t tile_bytes;   // 128 * 64 * 2
    int64_t c3max;        // section 3: chunks it has room for (0: no section)
    int64_t off_sec3;     // (these three when kc_total is known and c3max > 0)
    int64_t off_tiles3;
    int64_t off_meta3;
    int64_t bytes;        // total image size (when kc_total is known)
};
// K-groups of a layout's section 3, and the section's size
int64_t kgroups(const bp_layout &lay);
int64_t sec3_bytes(const bp_layout &lay);
constexpr int64_t kChunkBytes = 128 * kBK * 2 + 2 * kMetaBytes;   // per k-chunk, all parts

// Image layout; slab_chunks_host = per-slab chunk counts (host) or nullptr.
DevLayout dev_layout(const bp_layout &lay, const int64_t *slab_chunks_host);

// Library-wide settings.
uint64_t watchdog_ns();
int64_t debug_drop_stage();     // -1 = no fault injection
unsigned *device_status_ptr();   // device address of the status word
int num_sms();
PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder();   // nullptr if the driver lacks it
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
cudaError_t launch_pattern_scores(const bp_layout &lay, const void *W, const PatternSet &ps,
                                  double *scores, uint8_t *patsel, int *nonfinite,
                                  cudaStream_t s);
cudaError_t launch_pattern_mask(const bp_layout &lay, const uint8_t *keep, const uint8_t *patsel,
                                const PatternSet &ps, uint8_t *mask, cudaStream_t s);
cudaError_t launch_write_mask(const bp_layout &lay, const uint8_t *keep, uint8_t *mask,
                              cudaStream_t s);
int64_t threshold_chunks(int64_t U);

// Reweighted regulariser: per unit s = ||W_u||^2, alpha = 1/(s + eps),
// R = lambda * sum alpha^2 s, grad = 2 lambda alpha^2 W (fp32).  The
// workspace holds a completion counter (zero between calls) at offset 0 and
// the per-block partial sums of R from offset 256.
size_t penalty_workspace_bytes(const bp_layout &lay, int groups);
cudaError_t launch_penalty(const bp_layout &lay, int groups, const void *W, double eps,
                           double lambda, double *alpha, double *R, float *grad, void *ws,
                           cudaStream_t s);

cudaError_t launch_rb_counts(const bp_layout &lay, const uint8_t *mask, int64_t *rb_ptr,
                             int *bad, cudaStream_t s);
// Per slab: number of whole (dense) 64-column blocks and of remaining union
// columns, written to info[2*s], info[2*s+1] (device).
cudaError_t launch_slab_counts(const bp_layout &lay, const uint8_t *mask, int64_t *info,
                               cudaStream_t s);
cudaError_t launch_pack(const bp_layout &lay, const void *W, const uint8_t *mask,
                        const bp_packed &P, const DevLayout &dl, cudaStream_t s);
// Section 3 of the device image (see DevLayout); scratch: 8 * (S + 1) bytes of
// device memory for the per-slab counts.
cudaError_t launch_pack_sec3(const bp_layout &lay, const void *W, const uint8_t *mask,
                             const bp_packed &P, const DevLayout &dl, int64_t *scratch,
                             cudaStream_t s);

struct ConvShape {
    int64_t Nb, C, H, W, Ho, Wo;
    int kh, kw, ph, pw, sh, sw;
};
// im2col of an NCHW input: Xcol[k][n] (K x N row-major, leading dimension ldx),
// k = c*kh*kw + i*kw + j, n = b*Ho*Wo + oh*Wo + ow, zero outside the image.
// qmap: for row k of the full im2col matrix its row in xcol, or -1 to skip it
// (nullptr: row k is row k).
cudaError_t launch_im2col(const ConvShape &cs, int64_t ldx, const void *in, void *xcol,
                          const int32_t *qmap, cudaStream_t s);
int64_t im2col_row_width(const ConvShape &cs);   // staged input row length (elements)
// NCHW input -> NHWC with the channels padded to a multiple of 8 (zeros):
// out[b][h][w][c], C8 = roundup(C, 8) channels per pixel.  Stride-2 layers
// (cs.sh == 2): the four phases of the input (pixels (2h + a, 2w + c)), each
// ceil(H/2) x ceil(W/2), phase (a, c) of image b at image (2a + c) * Nb + b.
cudaError_t launch_nhwc8(const ConvShape &cs, const void *in, void *out, cudaStream_t s);
// Implicit convolution (stride 1, kh * kw > 1): output tiles of whole output
// rows.  ipt > 0: tiles of ipt whole images; else tiles of rpt rows of one
// image (tpi tiles per image).  nt = the tile's pixels rounded up to 32.
struct ImplicitTiles {
    int64_t ipt, rpt, tpi, tiles;
    int nt;
    bool ok;
};
ImplicitTiles implicit_tiles(const ConvShape &cs);
bool implicit_conv_ok(const bp_packed &P, const ConvShape &cs);
// The block-sparse product on the tensor cores: Y = act(W_packed X + bias).
// conv == nullptr: Y is M x N row-major (ldy).  Otherwise Y is the NCHW output
// of the convolution and X its im2col matrix.
// Split of the product into work units.  Persistent CTAs take (slab, column
// tile) items in waves; when the last wave is partial (or there are fewer
// items than SMs), its items are split along their k-chunks into `split`
// units each, whose fp32 partial tiles meet in a workspace: the last unit of
// an item to finish sums them and writes the output.
// Balanced launches (enough items for every SM, but a last wave that would
// leave many SMs idle): the chunks of all items are cut into one equal range
// per CTA; an item cut by a range boundary meets its parts through fp32
// partial tiles, one per CTA, and per-(CTA, quadrant) flags in the workspace.
struct SplitPlan {
    int nt;             // activation columns per tile
    int64_t items;      // (slab, column tile) items
    int64_t full;       // items computed whole (the first `full`)
    int split;          // units per remaining item (1: no split)
    int64_t units;      // full + (items - full) * split; balanced: the CTA count
    bool balanced;      // balanced launch
    int64_t total;      // balanced: chunks of all items
    size_t bytes;       // workspace: partial tiles + counters / flags (0 if none)
};
// Short path of bp_gemm (small layers with row-blocks of at most 64 rows): one
// CTA per (row-block, 64 tokens) on the compact storage, CUDA-core fp32.
bool small_path_ok(const bp_packed &P, int64_t N);
cudaError_t launch_small(const bp_packed &P, const void *X, int64_t N, int64_t ldx,
                         const float *bias, int relu, void *Y, int64_t ldy, cudaStream_t s);

// it: the implicit convolution's tiles (nullptr: tiles of nt consecutive columns)
SplitPlan plan_split(const DevLayout &dl, int64_t N, bool allow_split,
                     const ImplicitTiles *it = nullptr);

// With conv, X holds only the listed rows (see DevLayout::off_meta2), or
// with direct, X is the NCHW input of a 1 x 1 stride-1 layer read in place
// (ldx = H*W, a multiple of 8).  ws: at least plan_split(dl, N, true).bytes of
// 256-byte-aligned device memory, or nullptr (no split).
cudaError_t launch_mma(const bp_packed &P, const DevLayout &dl, const void *X, int64_t N,
                       int64_t ldx, const float *bias, int relu, void *Y, int64_t ldy,
                       const ConvShape *conv, void *ws, cudaStream_t s,
                       bool implicit = false, bool direct = false);
// 1 x 1 stride-1 layers without padding whose H*W is a multiple of 8: the
// product gathers the input's channel planes in place (no im2col)
bool direct_conv_ok(const ConvShape &cs);

}  // namespace bp
