/*
 * bp.h -- C ABI of libbp.so: inference of layers pruned with the block-based
 * (FC / GEMM view) and block-punched (CONV) schemes of arXiv 2111.11581,
 * on one NVIDIA GB300 (sm_103a).
 *
 *   bp_prune     keep the highest-norm columns / kernel positions of every
 *                block at a given rate                (Sec. 4.1, Eq. column,
 *                                                       Eq. punched, Sec. 5.1)
 *   bp_pack      dense weight + mask -> compact per-row-block storage (Sec. 4.3)
 *   bp_gemm      block-sparse GEMM  Y = (W o mask) X, fused bias/ReLU/cast
 *   bp_conv2d    block-sparse convolution (implicit GEMM for stride-1 and stride-2
 *                k x k layers, 1 x 1 stride-1 layers read in place, im2col + the
 *                same product otherwise), same epilogue
 *
 * Conventions shared by every call:
 *   - All tensor pointers are DEVICE pointers allocated by the caller; the
 *     library never allocates device memory.  Host pointers are only the
 *     scalar outputs named "host" below.
 *   - 16-bit float tensors are fp16 or bf16 per bp_layout.dtype.  Weights,
 *     activations and outputs of one call all use that dtype; biases are fp32.
 *   - `stream` is a cudaStream_t (NULL = legacy default stream).  Calls are
 *     asynchronous on it unless they say they synchronize.
 *   - Every call returns a bp_status.  Argument, shape and alignment problems
 *     are reported synchronously and launch nothing.  A kernel whose bounded
 *     wait ran out (it never hangs) records BP_ERR_TIMEOUT in a device status
 *     word that bp_device_status() reads.  CUDA launch errors map to
 *     BP_ERR_CUDA.
 *   - Pointers passed to bp_gemm / bp_conv2d must be 16-byte aligned and the
 *     leading dimensions multiples of 8 elements.
 */
#ifndef BP_H_
#define BP_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    BP_OK = 0,
    BP_ERR_INVALID_ARG = 1,   /* bad pointer, size, rate, alignment or mask */
    BP_ERR_UNSUPPORTED = 2,   /* valid but beyond the implemented limits (e.g. M > 1,048,576) */
    BP_ERR_NONFINITE = 3,     /* bp_prune: a weight is Inf or NaN */
    BP_ERR_WORKSPACE = 4,     /* workspace missing or smaller than bp_workspace_size() */
    BP_ERR_CUDA = 5,          /* a CUDA runtime call or launch failed */
    BP_ERR_TIMEOUT = 6        /* a kernel's bounded wait expired; its output is invalid */
} bp_status;

typedef enum { BP_F16 = 0, BP_BF16 = 1 } bp_dtype;

typedef enum {
    BP_BLOCK_BASED = 0,   /* Sec. 4.1.1: bm x bk blocks of the M x K matrix keep whole columns */
    BP_BLOCK_PUNCHED = 1  /* Sec. 4.1.2: bm filters x bk channels keep the same kh*kw positions */
} bp_scheme;

/* Shape of a prunable layer in GEMM view (Sec. 4.2: W_i is P x Q for FC,
 * P x Q x Kh x Kw for CONV; here M = P filters / out-features and
 * K = Q*Kh*Kw, the OIHW weight flattened so column k = c*kh*kw + i*kw + j).
 * Block-based: row-blocks of bm rows, column-blocks of bk columns of the
 *   M x K matrix (kh, kw only describe the conv for bp_conv2d).
 * Block-punched: blocks of bm filters x bk input channels; a block's units
 *   are its kh*kw kernel positions.
 * Partial last blocks keep their real size. */
typedef struct {
    int32_t scheme;   /* bp_scheme */
    int32_t dtype;    /* bp_dtype */
    int64_t M;        /* rows (filters / out-features), >= 1 */
    int64_t K;        /* columns = C*kh*kw, >= 1 */
    int32_t kh, kw;   /* kernel size, 1 x 1 for FC layers */
    int32_t bm;       /* rows per row-block, >= 1 */
    int32_t bk;       /* columns (block-based) or channels (punched) per block, >= 1 */
} bp_layout;

/* Compact storage of a pruned weight (Blocked Compressed Storage, Sec. 4.3).
 * All rows of a row-block keep the same columns, so one column list per
 * row-block replaces BCS's per-row column stride + occurrence arrays.
 * Filled by bp_pack_size (rb_ptr) and bp_pack (the rest); all arrays are
 * device memory owned by the caller and must stay alive while used.
 *   rb_ptr [num_rb+1]  int64: row-block rb's columns are col_idx[rb_ptr[rb] .. rb_ptr[rb+1])
 *   col_idx[nnz_cols]  int32: kept GEMM-view columns, ascending within a row-block
 *   values [nnz_vals]  16-bit: row-block rb is a bm_rb x K'_rb row-major block
 *                      starting at element bm*rb_ptr[rb] (bm_rb = rows of rb)
 *   dev    [dev_bytes] the same weights re-tiled for the tensor-core kernel:
 *                      slabs of 128 rows, each with the union of its rows'
 *                      kept columns in chunks of 64 (pre-swizzled tiles, zero
 *                      weights where a row prunes a column), their index lists
 *                      and load plans, and for layers with kh * kw > 1 a
 *                      second set of the slabs' tiles for the implicit
 *                      convolution (chunks of 64 channels at one kernel
 *                      position); opaque to callers, its size fixed by the
 *                      layout and the mask (bp_pack_size). */
typedef struct {
    bp_layout lay;
    int64_t num_rb;
    int64_t nnz_cols;
    int64_t nnz_vals;
    int64_t *rb_ptr;
    int32_t *col_idx;
    void *values;
    void *dev;
    int64_t dev_bytes;
} bp_packed;

/* Human-readable name of a status code (static string, never NULL). */
const char *bp_status_string(int status);

/* Library ABI version: (major << 16) | minor. */
int bp_version(void);

/* Device workspace bytes bp_prune needs for `lay` (host output); for
 * block-based layouts the same workspace also serves bp_prune_rows, for
 * block-punched 3x3 layouts bp_prune_pattern. */
bp_status bp_workspace_size(const bp_layout *lay, size_t *bytes);

/* One-shot magnitude pruning by block (Sec. 5.1 with the block regularities
 * of Sec. 4.1).  Scores are the squared L2 norms of Eq. (column) (block-based:
 * each column of each block) and Eq. (punched) (each kernel position of each
 * filters x channels block), accumulated in fp64 in ascending row (resp.
 * filter, then channel) order.  Rate r >= 1 is the parameter-reduction
 * factor: block b with P_b units keeps its floor(P_b / r) best units, and the
 * T - sum floor(P_b / r) best remaining units of the whole layer are kept as
 * well, T = floor(sum P_b / r + 0.5).  Ties prefer the lower unit index
 * (row-block, then column-block, then column / position).
 *   W     device, M x K 16-bit weights (OIHW for convolutions)
 *   rate  >= 1, finite
 *   mask  device, M x K uint8 output, 1 = kept
 *   ws    device workspace of at least bp_workspace_size() bytes, 256-B aligned
 * Synchronizes `stream` (it reads back counts); returns BP_ERR_NONFINITE if a
 * weight is Inf/NaN (mask then undefined). */
bp_status bp_prune(const bp_layout *lay, const void *W, double rate, uint8_t *mask, void *ws,
                   size_t ws_bytes, void *stream);

/* Row pruning of a block-based layer (Sec. 4.1.1: the rows and the columns of
 * each block are pruned independently; the rows are the groups of Eq. row).
 * The units of block (rb, cb) are its rows r -- the segments
 * W[r, cb*bk .. min(cb*bk + bk, K) - 1] -- scored by their squared norm in fp64
 * (columns ascending) and selected as bp_prune selects columns: floor(P_b / r)
 * per block of P_b rows, plus the best remaining units of the layer up to
 * T = floor(M * ceil(K/bk) / r + 0.5).  Units are ordered block-major (row-block,
 * then column-block), then by row; ties prefer the lower.  The result is ANDed
 * into `mask` (device, M x K uint8, in/out), so bp_prune followed by
 * bp_prune_rows, both on the same W, gives independent row and column pruning.
 * Rows of a row-block then keep different columns: pack such a mask with
 * bm = 1 (every row its own list).  Same workspace, synchronisation and errors
 * as bp_prune; BP_ERR_INVALID_ARG for block-punched layouts. */
bp_status bp_prune_rows(const bp_layout *lay, const void *W, double rate, uint8_t *mask,
                        void *ws, size_t ws_bytes, void *stream);

/* Pattern-based pruning of a 3x3 CONV layer (Sec. 2: kernel pattern pruning
 * plus connectivity pruning), the alternative the paper maps to 3x3 layers
 * for large datasets.  lay: block-punched, kh = kw = 3 (bm, bk unused).
 * Kernel (f, c) keeps the 4 positions (pos = 3i + j) of the pattern, among
 * `patterns` (host, npatterns 9-bit masks with 4 bits set, 1..16 of them),
 * whose kept squared norm (fp64, positions ascending) is largest, ties to the
 * lower pattern index; then the T = floor(9 F C / (4 rate) + 0.5) kernels
 * with the largest kept norms survive (connectivity pruning, ties to the
 * lower kernel index f*C + c) and the rest are removed.  rate >= 9/4 is the
 * parameter-reduction factor.  Filters then keep different columns: pack the
 * mask with bm = bk = 1.  Same workspace (bp_workspace_size of the layout),
 * synchronisation and errors as bp_prune. */
bp_status bp_prune_pattern(const bp_layout *lay, const void *W, double rate,
                           const uint16_t *patterns, int npatterns, uint8_t *mask, void *ws,
                           size_t ws_bytes, void *stream);

/* First half of packing: checks that every row of each row-block keeps the
 * same columns as the row-block's first row (BP_ERR_INVALID_ARG otherwise)
 * and writes rb_ptr (device, num_rb+1 int64, caller-allocated).  Host
 * outputs: nnz_cols, nnz_vals and dev_bytes, the sizes the caller allocates
 * for col_idx, values and dev.  Synchronizes `stream`. */
bp_status bp_pack_size(const bp_layout *lay, const uint8_t *mask, int64_t *rb_ptr,
                       int64_t *nnz_cols, int64_t *nnz_vals, int64_t *dev_bytes, void *stream);

/* Second half: fills out->col_idx, out->values and out->dev from W and mask.
 * `out` must carry lay, rb_ptr (from bp_pack_size), the sizes returned by
 * bp_pack_size and caller-allocated arrays of those sizes (dev 16-B aligned).
 * num_rb, nnz_cols, nnz_vals and dev_bytes are checked against the layout. */
bp_status bp_pack(const bp_layout *lay, const void *W, const uint8_t *mask, bp_packed *out,
                  void *stream);

/* Block-sparse GEMM (the FC layer of Sec. 4.2 with pruned weights skipped,
 * Sec. 4.3):  Y[m, n] = act( sum over kept k of W[m,k] * X[k,n] + bias[m] ),
 * fp32 accumulation on the tensor cores, one round-to-nearest-even cast.
 *   X     device, K x N row-major (leading dimension ldx >= N, multiple of 8)
 *   N     >= 0 columns (tokens)
 *   bias  device fp32 [M] or NULL
 *   relu  0 / 1
 *   Y     device, M x N row-major (ldy >= N, multiple of 8)
 *   ws    device workspace of bp_gemm_workspace_size() bytes (256-B aligned),
 *         or NULL: with it, a launch with fewer (128-row slab, column tile)
 *         items than SMs splits each item along k and its units add their
 *         fp32 partial sums into one accumulator tile per item in the
 *         workspace (atomic vector adds, so the order of those fp32 adds, and
 *         rarely the last bit of the rounded output, can differ from call to
 *         call); without it nothing is split (same result up to fp32
 *         summation order).  Zero-fill a new workspace (and again after a
 *         BP_ERR_TIMEOUT); the kernel leaves it zeroed for the next call.
 *         Calls that may overlap on the GPU need separate workspaces.
 * Any bm: weights are processed in slabs of 128 rows (see bp_packed::dev).
 * Small layers with row-blocks of at most 32 rows (nnz_vals * N <= 2^24) take
 * a short path instead: one CTA per (row-block, 32 tokens) on the compact
 * arrays (rb_ptr, col_idx, values), fp32 accumulation on the CUDA cores; `ws`
 * is not used there.
 * X must be finite: rows of X that a slab lists may meet zero weights of rows
 * that prune them (0 * Inf is NaN).  The launch is a programmatic dependent
 * of the previous kernel in `stream` (its set-up overlaps that kernel's end;
 * it reads X and writes Y only after that kernel has completed; the short
 * path reads the packed weights before, so they must not be written by that
 * kernel -- bp_pack synchronises its stream). */
bp_status bp_gemm(const bp_packed *P, const void *X, int64_t N, int64_t ldx, const float *bias,
                  int relu, void *Y, int64_t ldy, void *ws, size_t ws_bytes, void *stream);

/* Workspace bytes bp_gemm may use for this packed weight and N (host output;
 * 0 when nothing would be split). */
bp_status bp_gemm_workspace_size(const bp_packed *P, int64_t N, size_t *bytes);

/* Block-sparse convolution over the GEMM view of bp_layout (kept column
 * k = c*kh*kw + i*kw + j), NCHW input and output:
 *   out[b,f,oh,ow] = act( sum over kept (c,i,j) of W[f,c,i,j] *
 *                         in[b, c, oh*stride_h + i - pad_h, ow*stride_w + j - pad_w]
 *                         + bias[f] ),  zero outside the input.
 *   in    device, Nb x C x H x W;   out  device, Nb x M x Ho x Wo with
 *   Ho = (H + 2 pad_h - kh) / stride_h + 1, Wo likewise.
 *   ws    device workspace of at least bp_conv2d_workspace_size() bytes
 *         (256-B aligned), and the partial sums of the product's split work
 *         (see bp_gemm: zero-fill a new workspace).  Stride-1 layers with
 *         kh * kw > 1, W and Wo <= 256 (implicit GEMM): the input copied once
 *         to NHWC with the channels padded to a multiple of 8; the product
 *         loads, per k-chunk (64 channels at one kernel position), one TMA box
 *         of those channels for its tile of output rows, shifted by the kernel
 *         position, zeros outside the input being the padding.  Stride 2 in
 *         both directions, kh * kw > 1: the same, from the input's four
 *         phases (even / odd rows x even / odd columns, each ceil(H/2) x
 *         ceil(W/2) pixels, NHWC), a kernel position reading one phase.
 *         1 x 1 stride-1 layers without padding and with H*W a multiple of 8:
 *         the product reads the input's channel planes in place (the
 *         workspace holds only the split partial sums).  Other layers: the
 *         listed rows of the input expanded to the K x (Nb*Ho*Wo) matrix
 *         (im2col), which the product then reads.
 * Requires C*kh*kw == lay.K; dilation and groups are not supported.  The
 * input must be finite (see bp_gemm).  BP_ERR_UNSUPPORTED when kh input
 * rows padded to W + 2 pad_w exceed 12288 values, when Wo > 4096, Nb > 65535
 * or Nb*Ho*Wo >= 2^31. */
bp_status bp_conv2d(const bp_packed *P, const void *in, int64_t Nb, int64_t C, int64_t H,
                    int64_t W, int pad_h, int pad_w, int stride_h, int stride_w,
                    const float *bias, int relu, void *out, void *ws, size_t ws_bytes,
                    void *stream);

/* Device workspace bytes bp_conv2d needs for this packed weight and input
 * shape (host output): the implicit GEMM's NHWC copy, 2 * Nb * H * W *
 * (C rounded up to 8) (stride 2: 2 * 4 Nb * ceil(H/2) * ceil(W/2) * (C
 * rounded up to 8)), nothing for 1 x 1 layers read in place, or the im2col
 * matrix, 2 * K * (Nb*Ho*Wo rounded up to 8), rounded up to 256; plus the
 * split product's share. */
bp_status bp_conv2d_workspace_size(const bp_packed *P, int64_t Nb, int64_t C, int64_t H,
                                   int64_t W, int pad_h, int pad_w, int stride_h, int stride_w,
                                   size_t *bytes);

/* Groups of the reweighted regulariser (Sec. 4.2).  BP_GROUPS_LAYOUT: the
 * layout's pruning units -- the columns of each block for block-based layouts
 * (Eq. column), the kernel positions of each filters x channels block for
 * block-punched ones (Eq. punched).  BP_GROUPS_ROWS: the rows of each block of
 * a block-based layout (Eq. row); unit u = r * ceil(K / bk) + cb is the
 * segment W[r, cb*bk .. min(cb*bk + bk, K) - 1] (bm does not enter). */
typedef enum { BP_GROUPS_LAYOUT = 0, BP_GROUPS_ROWS = 1 } bp_groups;

/* Number of groups (host output) -- the length of bp_reweighted_penalty's
 * alpha: ceil(M/bm) * K (block-based), ceil(M/bm) * ceil(C/bk) * kh*kw
 * (block-punched), M * ceil(K/bk) (row groups).  BP_ERR_INVALID_ARG for row
 * groups of a block-punched layout. */
bp_status bp_penalty_units(const bp_layout *lay, int groups, int64_t *units);

/* Reweighted group-Lasso regulariser of one layer and its gradient (Sec. 4.2:
 * Eq. prob_block with the groups above; the reweighting of Candes et al. for
 * the factors):
 *   s_u     = squared Frobenius norm of group u's weights,
 *   alpha_u = 1 / (s_u + eps),
 *   R       = lambda * sum_u ||alpha_u o W_u||_F^2 = lambda * sum_u alpha_u^2 s_u,
 *   grad    = dR/dW = 2 lambda alpha_u^2 W  (the factors held fixed, as in
 *             one reweighting step).
 *   groups  a bp_groups value
 *   W       device, M x K 16-bit weights (OIHW for convolutions), 16-B aligned
 *   eps     > 0 (see the range below), lambda finite
 *   alpha   device fp64 [bp_penalty_units] output
 *   R       device fp64 scalar output
 *   grad    device fp32 M x K output, 16-B aligned
 *   ws      device workspace of bp_penalty_workspace_size() bytes, 256-B
 *           aligned, zero-filled before its first use; every call leaves it
 *           zeroed again.  Calls that may run concurrently need separate
 *           workspaces.
 * Precision (fp32, as in the paper's training): s_u is summed in fp32 (each
 * square of a 16-bit weight is exact in fp32; relative error at most
 * (n-1) 2^-24 for a group of n weights); alpha_u, the group's term
 * alpha_u^2 s_u and the factor 2 lambda alpha_u^2 are formed in fp32 from
 * fp32(eps) and fp32(2 lambda), and the gradient is that factor times each
 * weight in fp32; alpha is stored widened to fp64 and R is the fp64 sum of the
 * fp32 terms times lambda, in a fixed order (the same bits run to run on one
 * GPU).  Non-finite weights, and groups whose squared norm leaves the fp32
 * range (|w| above about 1.8e19), give non-finite outputs.  Asynchronous.
 * BP_ERR_UNSUPPORTED when M*K >= 2^31, or when eps is outside [2^-60, 2^60]
 * or 2 |lambda| / eps^2 >= 2^127 (the largest factor must be a finite fp32). */
bp_status bp_reweighted_penalty(const bp_layout *lay, int groups, const void *W, double eps,
                                double lambda, double *alpha, double *R, float *grad, void *ws,
                                size_t ws_bytes, void *stream);

/* Device workspace bytes bp_reweighted_penalty needs (host output):
 * 256 + 8 * (the number of blocks the launch uses, at most 2048). */
bp_status bp_penalty_workspace_size(const bp_layout *lay, int groups, size_t *bytes);

/* Synchronizes `stream`, then returns BP_ERR_TIMEOUT if any kernel of this
 * library recorded an expired wait since the previous call (and clears the
 * record), else BP_OK. */
bp_status bp_device_status(void *stream);

/* Upper bound, in nanoseconds, on every wait inside the kernels launched
 * after this call (default 2e9).  0 restores the default. */
bp_status bp_set_watchdog_ns(uint64_t ns);

/* bp_prune without a caller-provided workspace, for callers that cannot
 * allocate device memory (code running under a no-allocation rule after
 * start-up, plug-ins whose host framework owns all device memory, callers
 * that must not trigger the synchronisation cudaMalloc can cause).  The
 * paper has no counterpart: this is an interface convenience of this library.
 * Same arguments, result and synchronisation as bp_prune; the workspace is a
 * fixed 8 MiB array inside the library's device memory (held on every GPU
 * that loads the library until it is unloaded).  Layouts whose
 * bp_workspace_size() exceeds 8 MiB are rejected with BP_ERR_WORKSPACE before
 * anything is launched.  Like bp_prune it synchronises `stream` (the
 * selection reads counts back), so it cannot run inside a stream capture.
 * All calls share the array: calls that may overlap on the GPU race and must
 * be serialised by the caller.  Allocates nothing. */
bp_status bp_prune_noalloc(const bp_layout *lay, const void *W, double rate, uint8_t *mask,
                           void *stream);

/* Fault injection for tests of the bounded waits: from the next launch on,
 * CTA 0 of every bp_gemm / bp_conv2d kernel skips filling its pipeline stage
 * number `stage` (0-based, counted over the CTA's whole run), so the tensor-
 * core warp waits for data that never comes, its wait expires after the
 * watchdog budget, the kernel records BP_ERR_TIMEOUT and returns (the output
 * is then invalid).  -1 (the default) turns it off.  Nothing faults. */
bp_status bp_debug_drop_stage(int64_t stage);

#ifdef __cplusplus
}
#endif
#endif /* BP_H_ */
