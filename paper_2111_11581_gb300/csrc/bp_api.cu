// C ABI of libbp (declared in include/bp.h): argument checking, host-side
// counting and the launch sequences of bp_prune / bp_pack_size / bp_pack /
// bp_gemm / bp_conv2d.  No call allocates device memory.
#include <cmath>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <vector>

#include "bp_common.cuh"

namespace bp {

// Device status word: kernels OR kDevTimeout into it when a bounded wait ran
// out; bp_device_status() reads and clears it.
__device__ unsigned g_dev_status;
// Flag word of bp_pack_size's row-block consistency check and per-slab block
// counts of the device image (pack calls are serialised by g_mu).
__device__ int g_pack_bad;
__device__ int64_t g_slab_info[2 * kMaxSlabs];

namespace {
constexpr uint64_t kDefaultWatchdogNs = 2000000000ull;
uint64_t g_watchdog_ns = kDefaultWatchdogNs;
int64_t g_drop_stage = -1;
std::mutex g_mu;            // guards the per-device caches and g_pack_bad
constexpr int kMaxDev = 64;
int g_sms[kMaxDev];

int cur_dev() {
    int d = 0;
    cudaGetDevice(&d);
    return d < 0 || d >= kMaxDev ? 0 : d;
}

int64_t cdiv(int64_t a, int64_t b) { return (a + b - 1) / b; }

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

bp_status cuda_status(cudaError_t e) { return e == cudaSuccess ? BP_OK : BP_ERR_CUDA; }

bool layout_ok(const bp_layout *l) {
    if (!l) return false;
    if (l->scheme != BP_BLOCK_BASED && l->scheme != BP_BLOCK_PUNCHED) return false;
    if (l->dtype != BP_F16 && l->dtype != BP_BF16) return false;
    if (l->M < 1 || l->K < 1 || l->kh < 1 || l->kw < 1 || l->bm < 1 || l->bk < 1) return false;
    if (l->K % ((int64_t)l->kh * l->kw) != 0) return false;
    if (l->M > (int64_t)1 << 40 || l->K > ((int64_t)1 << 31) - 1) return false;
    return true;
}

// units and per-layer keep counts (Sec. 4.1 / 5.1 reading: floor(P_b / r) per
// block, T = floor(sum P_b / r + 0.5) per layer)
struct Counts {
    int64_t U, sum_base, T, E;
};

Counts host_counts(const bp_layout &l, double rate) {
    Counts c{};
    const int64_t RB = cdiv(l.M, l.bm);
    const int64_t KK = (int64_t)l.kh * l.kw;
    int64_t per_rb_base = 0, per_rb_units = 0;
    if (l.scheme == kSchemePattern) {
        // one unit per kernel, each a block of its own, kept at the kernel
        // rate 4 r / 9 (r = the weight rate): T = floor(9 F C / (4 r) + 0.5)
        c.U = l.M * (l.K / 9);
        c.sum_base = c.U * (int64_t)std::floor(1.0 / (4.0 * rate / 9.0));
        c.T = (int64_t)std::floor(9.0 * (double)c.U / (4.0 * rate) + 0.5);
        c.E = c.T - c.sum_base;
        return c;
    }
    if (l.scheme == kSchemeRows) {
        // row units: every block of row-block rb has rows_rb units
        const int64_t CB = cdiv(l.K, l.bk), last = l.M - (RB - 1) * l.bm;
        c.U = l.M * CB;
        c.sum_base = CB * ((RB - 1) * (int64_t)std::floor((double)l.bm / rate) +
                           (int64_t)std::floor((double)last / rate));
        c.T = (int64_t)std::floor((double)c.U / rate + 0.5);
        c.E = c.T - c.sum_base;
        return c;
    }
    if (l.scheme == BP_BLOCK_BASED) {
        const int64_t full = l.K / l.bk, tail = l.K % l.bk;
        per_rb_base = full * (int64_t)std::floor((double)l.bk / rate) +
                      (tail ? (int64_t)std::floor((double)tail / rate) : 0);
        per_rb_units = l.K;
    } else {
        const int64_t CB = cdiv(l.K / KK, l.bk);
        per_rb_base = CB * (int64_t)std::floor((double)KK / rate);
        per_rb_units = CB * KK;
    }
    c.U = RB * per_rb_units;
    c.sum_base = RB * per_rb_base;
    c.T = (int64_t)std::floor((double)c.U / rate + 0.5);
    c.E = c.T - c.sum_base;
    return c;
}

struct PruneWs {
    int64_t off_scores, off_hist, off_chunks, off_flag, off_keep, off_patsel, total;
};

int64_t align_up(int64_t v, int64_t a) { return (v + a - 1) / a * a; }

PruneWs prune_ws(const bp_layout &l) {
    Counts c = host_counts(l, 1.0);
    if (l.scheme == BP_BLOCK_BASED) {
        // one workspace serves bp_prune and bp_prune_rows
        bp_layout rows = l;
        rows.scheme = (bp_scheme)kSchemeRows;
        c.U = std::max(c.U, host_counts(rows, 1.0).U);
    }
    const bool k3 = l.scheme == BP_BLOCK_PUNCHED && l.kh == 3 && l.kw == 3;
    if (k3) c.U = std::max(c.U, l.M * (l.K / 9));   // ... and bp_prune_pattern
    PruneWs w;
    w.off_scores = 0;
    w.off_hist = align_up(c.U * 8, 256);
    w.off_chunks = w.off_hist + 1024;
    w.off_flag = align_up(w.off_chunks + 8 * threshold_chunks(c.U), 256);
    w.off_keep = w.off_flag + 256;
    w.off_patsel = align_up(w.off_keep + c.U, 256);
    w.total = k3 ? align_up(w.off_patsel + c.U, 256) : w.off_patsel;
    return w;
}

// The pruning pipeline over the units of `lay` (scheme may be kSchemeRows):
// scores, per-block keep, layer-wide extras by radix select, mask.
bp_status prune_units(const bp_layout &lay, const void *W, double rate, uint8_t *mask,
                      void *ws, const PruneWs &w, cudaStream_t s,
                      const PatternSet *ps = nullptr) {
    uint8_t *base = static_cast<uint8_t *>(ws);
    double *scores = reinterpret_cast<double *>(base + w.off_scores);
    unsigned *hist = reinterpret_cast<unsigned *>(base + w.off_hist);
    int64_t *chunks = reinterpret_cast<int64_t *>(base + w.off_chunks);
    int *flag = reinterpret_cast<int *>(base + w.off_flag);
    uint8_t *keep = base + w.off_keep;
    const Counts c = host_counts(lay, rate);

    uint8_t *patsel = base + w.off_patsel;
    cudaError_t e = cudaMemsetAsync(flag, 0, sizeof(int), s);
    if (e == cudaSuccess)
        e = ps ? launch_pattern_scores(lay, W, *ps, scores, patsel, flag, s)
               : launch_scores(lay, W, scores, flag, s);
    // pattern units are blocks of one kernel: floor(1 / (4 r / 9)) of each
    if (e == cudaSuccess) e = launch_base_select(lay, scores, ps ? 4.0 * rate / 9.0 : rate, keep, s);
    int nonfinite = 0;
    if (e == cudaSuccess) e = cudaMemcpyAsync(&nonfinite, flag, sizeof(int), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return BP_ERR_CUDA;
    if (nonfinite) return BP_ERR_NONFINITE;

    if (c.E > 0) {
        // most-significant-digit radix select of the E-th best remaining unit
        uint64_t prefix = 0;
        int64_t need = c.E;
        unsigned h[256];
        for (int shift = 56; shift >= 0; shift -= 8) {
            e = cudaMemsetAsync(hist, 0, 256 * sizeof(unsigned), s);
            if (e == cudaSuccess) e = launch_radix_hist(c.U, scores, keep, prefix, shift, hist, s);
            if (e == cudaSuccess) e = cudaMemcpyAsync(h, hist, sizeof(h), cudaMemcpyDeviceToHost, s);
            if (e == cudaSuccess) e = cudaStreamSynchronize(s);
            if (e != cudaSuccess) return BP_ERR_CUDA;
            int d = 255;
            for (; d > 0; --d) {
                if ((int64_t)h[d] >= need) break;
                need -= h[d];
            }
            prefix |= (uint64_t)d << shift;
        }
        e = launch_threshold_select(c.U, scores, keep, prefix, need, chunks, s);
        if (e != cudaSuccess) return BP_ERR_CUDA;
    }
    e = ps ? launch_pattern_mask(lay, keep, patsel, *ps, mask, s)
           : launch_write_mask(lay, keep, mask, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    return cuda_status(e);
}

}  // namespace

uint64_t watchdog_ns() { return g_watchdog_ns; }
int64_t debug_drop_stage() { return g_drop_stage; }

// Looked up on every call (a host-side lookup, no allocation): an address
// cached across calls would go stale when the device's context is reset.
unsigned *device_status_ptr() {
    void *p = nullptr;
    if (cudaGetSymbolAddress(&p, g_dev_status) != cudaSuccess) return nullptr;
    return static_cast<unsigned *>(p);
}

int num_sms() {
    const int d = cur_dev();
    if (!g_sms[d]) {
        int v = 0;
        cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, d);
        g_sms[d] = v > 0 ? v : 1;
    }
    return g_sms[d];
}

bool checked_mode() {
    const char *e = std::getenv("BP_CHECKED");
    return e && e[0] == '1';
}

static int64_t qmap_bytes(const bp_layout &lay) { return align_up(4 * lay.K, 16); }

int64_t kgroups(const bp_layout &lay) {
    if ((int64_t)lay.kh * lay.kw <= 1) return 0;
    const int64_t C = lay.K / ((int64_t)lay.kh * lay.kw);
    return cdiv(C, 64) * lay.kh * lay.kw;
}

static int64_t sec3_chunks(const bp_layout &lay) {
    return cdiv(lay.M, kSlab) * kgroups(lay);
}

int64_t sec3_bytes(const bp_layout &lay) {
    const int64_t c3 = sec3_chunks(lay);
    if (c3 == 0) return 0;
    return align_up(8 * (cdiv(lay.M, kSlab) + 1), 256) + c3 * ((int64_t)kSlab * kBK * 2 + kMetaBytes);
}

static void set_chunks(DevLayout &d, const bp_layout &lay, int64_t kc) {
    d.kc_total = kc;
    d.off_meta = d.off_tiles + kc * d.tile_bytes;
    d.off_meta2 = d.off_meta + kc * kMetaBytes;
    d.off_qmap = d.off_meta2 + kc * kMetaBytes;
    d.bytes = d.off_qmap + qmap_bytes(lay);
    if (d.c3max > 0) {
        d.off_sec3 = align_up(d.bytes, 256);
        d.off_tiles3 = d.off_sec3 + align_up(8 * (d.num_slabs + 1), 256);
        d.off_meta3 = d.off_tiles3 + d.c3max * d.tile_bytes;
        d.bytes = d.off_sec3 + sec3_bytes(lay);
    }
}

DevLayout dev_layout(const bp_layout &lay, const int64_t *slab_chunks_host) {
    DevLayout d{};
    d.num_slabs = cdiv(lay.M, kSlab);
    d.off_tiles = align_up(8 * (d.num_slabs + 2), 256);
    d.tile_bytes = (int64_t)kSlab * kBK * 2;
    d.kc_total = -1;
    d.off_meta = d.off_meta2 = d.off_qmap = -1;
    d.c3max = sec3_chunks(lay);
    d.off_sec3 = d.off_tiles3 = d.off_meta3 = -1;
    d.bytes = -1;
    if (slab_chunks_host) {
        int64_t kc = 0;
        for (int64_t s = 0; s < d.num_slabs; ++s) kc += slab_chunks_host[s];
        set_chunks(d, lay, kc);
    }
    return d;
}

// Per-slab chunk counts of the device image (device pass + read-back; syncs).
static bp_status slab_chunk_counts(const bp_layout &lay, const uint8_t *mask, cudaStream_t s,
                                   std::vector<int64_t> &chunks) {
    const int64_t S = cdiv(lay.M, kSlab);
    int64_t *info = nullptr;
    if (cudaGetSymbolAddress(reinterpret_cast<void **>(&info), g_slab_info) != cudaSuccess)
        return BP_ERR_CUDA;
    std::vector<int64_t> h(2 * S);
    cudaError_t e = launch_slab_counts(lay, mask, info, s);
    if (e == cudaSuccess) e = cudaMemcpyAsync(h.data(), info, 16 * S, cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return BP_ERR_CUDA;
    chunks.resize(S);
    for (int64_t i = 0; i < S; ++i) chunks[i] = h[2 * i] + cdiv(h[2 * i + 1], kBK);
    return BP_OK;
}

ImplicitTiles implicit_tiles(const ConvShape &cs) {
    ImplicitTiles t{};
    t.ok = false;
    if (cs.Wo < 1 || cs.Ho < 1 || cs.Wo > 256 || cs.W > 256 || cs.Nb < 1) return t;
    const int64_t HoWo = cs.Ho * cs.Wo;
    int64_t px;
    if (HoWo <= 256) {
        // tiles of whole images (box: 64 channels x Wo x Ho x ipt)
        t.ipt = std::min<int64_t>(256 / HoWo, cs.Nb);
        t.rpt = cs.Ho;
        t.tpi = 1;
        t.tiles = cdiv(cs.Nb, t.ipt);
        px = t.ipt * HoWo;
    } else {
        // tiles of rpt whole rows of one image (box: 64 channels x Wo x rpt x 1);
        // rpt * Wo a multiple of 8 where possible, so that every tile starts
        // 16-byte aligned in the NCHW output (its TMA box stores need that)
        t.ipt = 0;
        t.rpt = 256 / cs.Wo;
        for (int64_t r = t.rpt; r >= 1; --r)
            if ((r * cs.Wo) % 8 == 0) {
                t.rpt = r;
                break;
            }
        t.tpi = cdiv(cs.Ho, t.rpt);
        t.tiles = cs.Nb * t.tpi;
        px = t.rpt * cs.Wo;
    }
    t.nt = (int)align_up(px, 32);
    t.ok = t.nt <= 256 && t.tiles < INT32_MAX;
    return t;
}

// The implicit convolution serves stride-1 and stride-2 layers with a kh x kw
// > 1 window (the image's section 3); other strides and 1 x 1 layers take the
// im2col path.
bool implicit_conv_ok(const bp_packed &P, const ConvShape &cs) {
    // stride 1, or stride 2 in both directions (the input staged by phases)
    if ((int64_t)cs.kh * cs.kw <= 1 || cs.sh != cs.sw || (cs.sh != 1 && cs.sh != 2)) return false;
    if (sec3_bytes(P.lay) == 0) return false;
    if (cs.ph > 255 || cs.pw > 255 || cs.kh > 255 || cs.kw > 255) return false;
    if ((cs.C + 63) / 64 > 32767) return false;
    return implicit_tiles(cs).ok;
}

bool direct_conv_ok(const ConvShape &cs) {
    return cs.kh == 1 && cs.kw == 1 && cs.sh == 1 && cs.sw == 1 && cs.ph == 0 && cs.pw == 0 &&
           (cs.H * cs.W) % 8 == 0;
}

size_t nhwc8_bytes(const ConvShape &cs) {
    if (cs.sh == 2)     // four phases of ceil(H/2) x ceil(W/2) pixels
        return (size_t)align_up(4 * cs.Nb * cdiv(cs.H, 2) * cdiv(cs.W, 2) * align_up(cs.C, 8) * 2, 256);
    return (size_t)align_up(cs.Nb * cs.H * cs.W * align_up(cs.C, 8) * 2, 256);
}

}  // namespace bp

using namespace bp;

extern "C" {

const char *bp_status_string(int status) {
    switch (status) {
    case BP_OK: return "ok";
    case BP_ERR_INVALID_ARG: return "invalid argument";
    case BP_ERR_UNSUPPORTED: return "unsupported configuration";
    case BP_ERR_NONFINITE: return "non-finite weight";
    case BP_ERR_WORKSPACE: return "workspace too small";
    case BP_ERR_CUDA: return "CUDA error";
    case BP_ERR_TIMEOUT: return "kernel wait timed out";
    default: return "unknown status";
    }
}

int bp_version(void) { return (2 << 16) | 4; }

bp_status bp_workspace_size(const bp_layout *lay, size_t *bytes) {
    if (!layout_ok(lay) || !bytes) return BP_ERR_INVALID_ARG;
    *bytes = (size_t)prune_ws(*lay).total;
    return BP_OK;
}

bp_status bp_prune(const bp_layout *lay, const void *W, double rate, uint8_t *mask, void *ws,
                   size_t ws_bytes, void *stream) {
    if (!layout_ok(lay) || !W || !mask) return BP_ERR_INVALID_ARG;
    if (!(rate >= 1.0) || !std::isfinite(rate)) return BP_ERR_INVALID_ARG;
    const PruneWs w = prune_ws(*lay);
    if (!ws || ws_bytes < (size_t)w.total || (reinterpret_cast<uintptr_t>(ws) & 255u))
        return BP_ERR_WORKSPACE;
    return prune_units(*lay, W, rate, mask, ws, w, static_cast<cudaStream_t>(stream));
}

bp_status bp_prune_pattern(const bp_layout *lay, const void *W, double rate,
                           const uint16_t *patterns, int npatterns, uint8_t *mask, void *ws,
                           size_t ws_bytes, void *stream) {
    if (!layout_ok(lay) || !W || !mask || !patterns) return BP_ERR_INVALID_ARG;
    if (lay->scheme != BP_BLOCK_PUNCHED || lay->kh != 3 || lay->kw != 3)
        return BP_ERR_INVALID_ARG;
    if (!(rate >= 2.25) || !std::isfinite(rate)) return BP_ERR_INVALID_ARG;
    if (npatterns < 1 || npatterns > kMaxPatterns) return BP_ERR_INVALID_ARG;
    PatternSet ps{};
    ps.n = npatterns;
    for (int q = 0; q < npatterns; ++q) {
        if ((patterns[q] >> 9) || __builtin_popcount(patterns[q]) != 4) return BP_ERR_INVALID_ARG;
        ps.m[q] = patterns[q];
    }
    const PruneWs w = prune_ws(*lay);
    if (!ws || ws_bytes < (size_t)w.total || (reinterpret_cast<uintptr_t>(ws) & 255u))
        return BP_ERR_WORKSPACE;
    bp_layout pl = *lay;
    pl.scheme = (bp_scheme)kSchemePattern;
    return prune_units(pl, W, rate, mask, ws, w, static_cast<cudaStream_t>(stream), &ps);
}

bp_status bp_prune_rows(const bp_layout *lay, const void *W, double rate, uint8_t *mask,
                        void *ws, size_t ws_bytes, void *stream) {
    if (!layout_ok(lay) || !W || !mask || lay->scheme != BP_BLOCK_BASED)
        return BP_ERR_INVALID_ARG;
    if (!(rate >= 1.0) || !std::isfinite(rate)) return BP_ERR_INVALID_ARG;
    const PruneWs w = prune_ws(*lay);
    if (!ws || ws_bytes < (size_t)w.total || (reinterpret_cast<uintptr_t>(ws) & 255u))
        return BP_ERR_WORKSPACE;
    bp_layout rows = *lay;
    rows.scheme = (bp_scheme)kSchemeRows;
    return prune_units(rows, W, rate, mask, ws, w, static_cast<cudaStream_t>(stream));
}

bp_status bp_pack_size(const bp_layout *lay, const uint8_t *mask, int64_t *rb_ptr,
                       int64_t *nnz_cols, int64_t *nnz_vals, int64_t *dev_bytes, void *stream) {
    if (!layout_ok(lay) || !mask || !rb_ptr || !nnz_cols || !nnz_vals || !dev_bytes)
        return BP_ERR_INVALID_ARG;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const int64_t RB = cdiv(lay->M, lay->bm);
    if (RB > 65535) return BP_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> lk(g_mu);
    int *bad = nullptr;
    if (cudaGetSymbolAddress(reinterpret_cast<void **>(&bad), g_pack_bad) != cudaSuccess)
        return BP_ERR_CUDA;
    std::vector<int64_t> h(RB + 1);
    int hbad = 0;
    cudaError_t e = cudaMemsetAsync(bad, 0, sizeof(int), s);
    if (e == cudaSuccess) e = launch_rb_counts(*lay, mask, rb_ptr, bad, s);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(h.data(), rb_ptr, 8 * (RB + 1), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaMemcpyAsync(&hbad, bad, sizeof(int), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return BP_ERR_CUDA;
    if (hbad) return BP_ERR_INVALID_ARG;
    int64_t nv = 0;
    for (int64_t rb = 0; rb < RB; ++rb) {
        const int64_t rows = std::min<int64_t>(lay->bm, lay->M - rb * lay->bm);
        nv += rows * (h[rb + 1] - h[rb]);
    }
    if (cdiv(lay->M, kSlab) > kMaxSlabs) return BP_ERR_UNSUPPORTED;
    std::vector<int64_t> sc;
    const bp_status st = slab_chunk_counts(*lay, mask, s, sc);
    if (st != BP_OK) return st;
    *nnz_cols = h[RB];
    *nnz_vals = nv;
    *dev_bytes = dev_layout(*lay, sc.data()).bytes;
    return BP_OK;
}

bp_status bp_pack(const bp_layout *lay, const void *W, const uint8_t *mask, bp_packed *out,
                  void *stream) {
    if (!layout_ok(lay) || !W || !mask || !out || !out->rb_ptr) return BP_ERR_INVALID_ARG;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const int64_t RB = cdiv(lay->M, lay->bm);
    if (RB > 65535) return BP_ERR_UNSUPPORTED;
    if (out->num_rb != RB) return BP_ERR_INVALID_ARG;
    std::vector<int64_t> h(RB + 1);
    cudaError_t e = cudaMemcpyAsync(h.data(), out->rb_ptr, 8 * (RB + 1), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return BP_ERR_CUDA;
    if (h[0] != 0) return BP_ERR_INVALID_ARG;
    int64_t nv = 0;
    for (int64_t rb = 0; rb < RB; ++rb) {
        const int64_t kp = h[rb + 1] - h[rb];
        if (kp < 0 || kp > lay->K) return BP_ERR_INVALID_ARG;
        nv += std::min<int64_t>(lay->bm, lay->M - rb * lay->bm) * kp;
    }
    if (out->nnz_cols != h[RB] || out->nnz_vals != nv) return BP_ERR_INVALID_ARG;
    if ((h[RB] > 0 && !out->col_idx) || (nv > 0 && !out->values)) return BP_ERR_INVALID_ARG;
    if (cdiv(lay->M, kSlab) > kMaxSlabs) return BP_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> lk(g_mu);
    std::vector<int64_t> sc;
    const bp_status st = slab_chunk_counts(*lay, mask, s, sc);
    if (st != BP_OK) return st;
    const DevLayout dl = dev_layout(*lay, sc.data());
    if (out->dev_bytes != dl.bytes) return BP_ERR_INVALID_ARG;
    if (!out->dev || !aligned16(out->dev)) return BP_ERR_INVALID_ARG;
    out->lay = *lay;
    std::vector<int64_t> kc(dl.num_slabs + 2, 0);
    for (int64_t i = 0; i < dl.num_slabs; ++i) kc[i + 1] = kc[i] + sc[i];
    e = cudaMemcpyAsync(out->dev, kc.data(), 8 * (dl.num_slabs + 2), cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess) e = launch_pack(*lay, W, mask, *out, dl, s);
    if (e == cudaSuccess && dl.c3max > 0) {
        int64_t *scratch = nullptr;   // the slab-count words (under g_mu)
        e = cudaGetSymbolAddress(reinterpret_cast<void **>(&scratch), g_slab_info);
        if (e == cudaSuccess) e = launch_pack_sec3(*lay, W, mask, *out, dl, scratch, s);
    }
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    return cuda_status(e);
}

static bp_status check_packed(const bp_packed *P, DevLayout *dl) {
    if (!P || !layout_ok(&P->lay) || !P->dev || !aligned16(P->dev)) return BP_ERR_INVALID_ARG;
    if (P->num_rb != cdiv(P->lay.M, P->lay.bm)) return BP_ERR_INVALID_ARG;
    if (cdiv(P->lay.M, kSlab) > kMaxSlabs) return BP_ERR_UNSUPPORTED;
    *dl = dev_layout(P->lay, nullptr);
    // the chunk count follows from the image size: tiles + two record sets + qmap
    // (+ section 3, whose size the layout fixes; it starts 256-byte aligned)
    const int64_t s3 = sec3_bytes(P->lay);
    for (int64_t pad = 0; pad < (s3 ? 256 : 1); pad += 16) {
        const int64_t rest = P->dev_bytes - s3 - pad - dl->off_tiles - qmap_bytes(P->lay);
        if (rest < 0 || rest % kChunkBytes) continue;
        set_chunks(*dl, P->lay, rest / kChunkBytes);
        if (dl->bytes == P->dev_bytes) return BP_OK;
    }
    return BP_ERR_INVALID_ARG;
}

static bp_status finish_launch(cudaError_t e, cudaStream_t s) {
    if (e != cudaSuccess) return BP_ERR_CUDA;
    if (checked_mode()) return bp_device_status(s);
    return BP_OK;
}

bp_status bp_gemm_workspace_size(const bp_packed *P, int64_t N, size_t *bytes) {
    DevLayout dl;
    if (!bytes || N < 0) return BP_ERR_INVALID_ARG;
    const bp_status st = check_packed(P, &dl);
    if (st != BP_OK) return st;
    *bytes = N > 0 ? plan_split(dl, N, true).bytes : 0;
    return BP_OK;
}

bp_status bp_gemm(const bp_packed *P, const void *X, int64_t N, int64_t ldx, const float *bias,
                  int relu, void *Y, int64_t ldy, void *ws, size_t ws_bytes, void *stream) {
    DevLayout dl;
    bp_status st = check_packed(P, &dl);
    if (st != BP_OK) return st;
    if (N < 0 || !X || !Y || ldx < N || ldy < N || ldx % 8 || ldy % 8) return BP_ERR_INVALID_ARG;
    if (!aligned16(X) || !aligned16(Y)) return BP_ERR_INVALID_ARG;
    if (bias && (reinterpret_cast<uintptr_t>(bias) & 3u)) return BP_ERR_INVALID_ARG;
    if (ws && ((reinterpret_cast<uintptr_t>(ws) & 255u) || ws_bytes < plan_split(dl, N, true).bytes))
        return BP_ERR_WORKSPACE;
    if (N == 0) return BP_OK;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (small_path_ok(*P, N)) {
        if ((P->nnz_cols > 0 && !P->col_idx) || (P->nnz_vals > 0 && !P->values) || !P->rb_ptr)
            return BP_ERR_INVALID_ARG;
        return finish_launch(launch_small(*P, X, N, ldx, bias, relu, Y, ldy, s), s);
    }
    return finish_launch(launch_mma(*P, dl, X, N, ldx, bias, relu, Y, ldy, nullptr, ws, s), s);
}

static bp_status conv_shape(const bp_packed *P, int64_t Nb, int64_t C, int64_t H, int64_t W,
                            int pad_h, int pad_w, int stride_h, int stride_w, ConvShape *cs,
                            DevLayout *dl) {
    bp_status st = check_packed(P, dl);
    if (st != BP_OK) return st;
    const bp_layout &l = P->lay;
    if (Nb < 0 || C < 1 || H < 1 || W < 1) return BP_ERR_INVALID_ARG;
    if (pad_h < 0 || pad_w < 0 || stride_h < 1 || stride_w < 1) return BP_ERR_INVALID_ARG;
    if (C * l.kh * l.kw != l.K) return BP_ERR_INVALID_ARG;
    if (H + 2 * pad_h < l.kh || W + 2 * pad_w < l.kw) return BP_ERR_INVALID_ARG;
    if (H > (1 << 28) || W > (1 << 28)) return BP_ERR_UNSUPPORTED;

    // 32-bit pixel indexing in the im2col pass
    const int64_t Ho = (H + 2 * pad_h - l.kh) / stride_h + 1, Wo = (W + 2 * pad_w - l.kw) / stride_w + 1;
    if (Nb * Ho * Wo > INT32_MAX - 8 || Nb * C * H * W > ((int64_t)1 << 40)) return BP_ERR_UNSUPPORTED;
    cs->Nb = Nb;
    cs->C = C;
    cs->H = H;
    cs->W = W;
    cs->Ho = (H + 2 * pad_h - l.kh) / stride_h + 1;
    cs->Wo = (W + 2 * pad_w - l.kw) / stride_w + 1;
    cs->kh = l.kh;
    cs->kw = l.kw;
    cs->ph = pad_h;
    cs->pw = pad_w;
    cs->sh = stride_h;
    cs->sw = stride_w;
    // the im2col pass stages kh padded input rows in 24 KB of shared memory
    if (im2col_row_width(*cs) * l.kh > 12288 || cs->Wo > 4096 || Nb > 65535)
        return BP_ERR_UNSUPPORTED;
    return BP_OK;
}

bp_status bp_conv2d_workspace_size(const bp_packed *P, int64_t Nb, int64_t C, int64_t H,
                                   int64_t W, int pad_h, int pad_w, int stride_h, int stride_w,
                                   size_t *bytes) {
    ConvShape cs;
    DevLayout dl;
    if (!bytes) return BP_ERR_INVALID_ARG;
    const bp_status st = conv_shape(P, Nb, C, H, W, pad_h, pad_w, stride_h, stride_w, &cs, &dl);
    if (st != BP_OK) return st;
    const int64_t N = Nb * cs.Ho * cs.Wo;
    if (implicit_conv_ok(*P, cs)) {
        const ImplicitTiles it = implicit_tiles(cs);
        *bytes = nhwc8_bytes(cs) + plan_split(dl, N, true, &it).bytes;
        return BP_OK;
    }
    if (direct_conv_ok(cs)) {
        *bytes = plan_split(dl, N, true).bytes;
        return BP_OK;
    }
    *bytes = (size_t)align_up(P->lay.K * align_up(N, 8) * 2, 256) + plan_split(dl, N, true).bytes;
    return BP_OK;
}

bp_status bp_conv2d(const bp_packed *P, const void *in, int64_t Nb, int64_t C, int64_t H,
                    int64_t W, int pad_h, int pad_w, int stride_h, int stride_w,
                    const float *bias, int relu, void *out, void *ws, size_t ws_bytes,
                    void *stream) {
    ConvShape cs;
    DevLayout dl;
    const bp_status st =
        conv_shape(P, Nb, C, H, W, pad_h, pad_w, stride_h, stride_w, &cs, &dl);
    if (st != BP_OK) return st;
    if (!in || !out || !aligned16(in) || !aligned16(out)) return BP_ERR_INVALID_ARG;
    if (bias && (reinterpret_cast<uintptr_t>(bias) & 3u)) return BP_ERR_INVALID_ARG;
    const int64_t N = Nb * cs.Ho * cs.Wo;
    if (N == 0) return BP_OK;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (implicit_conv_ok(*P, cs)) {
        // implicit GEMM: the input goes to NHWC (channels padded to 8) in the
        // workspace; the product loads its B operand from it with TMA boxes
        const ImplicitTiles it = implicit_tiles(cs);
        const size_t xb = nhwc8_bytes(cs);
        const size_t sb = plan_split(dl, N, true, &it).bytes;
        if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) || ws_bytes < xb + sb)
            return BP_ERR_WORKSPACE;
        void *split_ws = sb ? static_cast<uint8_t *>(ws) + xb : nullptr;
        cudaError_t e = launch_nhwc8(cs, in, ws, s);
        if (e != cudaSuccess) return BP_ERR_CUDA;
        return finish_launch(
            launch_mma(*P, dl, ws, N, 0, bias, relu, out, 0, &cs, split_ws, s, true), s);
    }
    if (direct_conv_ok(cs)) {
        // 1 x 1, stride 1: the channel planes are the activation rows
        const size_t sb = plan_split(dl, N, true).bytes;
        if (sb && (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) || ws_bytes < sb))
            return BP_ERR_WORKSPACE;
        return finish_launch(launch_mma(*P, dl, in, N, cs.H * cs.W, bias, relu, out, 0, &cs,
                                        sb ? ws : nullptr, s, false, true),
                             s);
    }
    const int64_t ldx = align_up(N, 8);
    // workspace: the im2col matrix, then the split product's partial tiles
    const size_t xbytes = (size_t)align_up(P->lay.K * ldx * 2, 256);
    const size_t sbytes = plan_split(dl, N, true).bytes;
    if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) || ws_bytes < xbytes + sbytes)
        return BP_ERR_WORKSPACE;
    void *split_ws = sbytes ? static_cast<uint8_t *>(ws) + xbytes : nullptr;
    const int32_t *qmap =
        reinterpret_cast<const int32_t *>(static_cast<const uint8_t *>(P->dev) + dl.off_qmap);
    cudaError_t e = launch_im2col(cs, ldx, in, ws, qmap, s);
    if (e != cudaSuccess) return BP_ERR_CUDA;
    return finish_launch(launch_mma(*P, dl, ws, N, ldx, bias, relu, out, 0, &cs, split_ws, s), s);
}

static bool groups_ok(const bp_layout *lay, int groups) {
    if (groups == BP_GROUPS_LAYOUT) return true;
    return groups == BP_GROUPS_ROWS && lay->scheme == BP_BLOCK_BASED;
}

bp_status bp_penalty_units(const bp_layout *lay, int groups, int64_t *units) {
    if (!layout_ok(lay) || !units || !groups_ok(lay, groups)) return BP_ERR_INVALID_ARG;
    const int64_t RB = cdiv(lay->M, lay->bm);
    if (groups == BP_GROUPS_ROWS) {
        *units = lay->M * cdiv(lay->K, lay->bk);
    } else if (lay->scheme == BP_BLOCK_BASED) {
        *units = RB * lay->K;
    } else {
        const int64_t KK = (int64_t)lay->kh * lay->kw;
        *units = RB * cdiv(lay->K / KK, lay->bk) * KK;
    }
    return BP_OK;
}

bp_status bp_penalty_workspace_size(const bp_layout *lay, int groups, size_t *bytes) {
    if (!layout_ok(lay) || !bytes || !groups_ok(lay, groups)) return BP_ERR_INVALID_ARG;
    if (lay->M * lay->K >= INT32_MAX) return BP_ERR_UNSUPPORTED;
    *bytes = penalty_workspace_bytes(*lay, groups);
    return BP_OK;
}

bp_status bp_reweighted_penalty(const bp_layout *lay, int groups, const void *W, double eps,
                                double lambda, double *alpha, double *R, float *grad, void *ws,
                                size_t ws_bytes, void *stream) {
    if (!layout_ok(lay) || !W || !alpha || !R || !grad || !groups_ok(lay, groups))
        return BP_ERR_INVALID_ARG;
    if (!aligned16(W) || !aligned16(grad) || (reinterpret_cast<uintptr_t>(alpha) & 7u) ||
        (reinterpret_cast<uintptr_t>(R) & 7u))
        return BP_ERR_INVALID_ARG;
    if (!(eps > 0.0) || !std::isfinite(eps) || !std::isfinite(lambda)) return BP_ERR_INVALID_ARG;
    if (lay->M * lay->K >= INT32_MAX) return BP_ERR_UNSUPPORTED;
    // the fp32 factors: eps and 1/eps representable, 2 |lambda| / eps^2 finite
    if (eps < 0x1p-60 || eps > 0x1p60 || 2.0 * std::fabs(lambda) / (eps * eps) >= 0x1p127)
        return BP_ERR_UNSUPPORTED;
    if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) ||
        ws_bytes < penalty_workspace_bytes(*lay, groups))
        return BP_ERR_WORKSPACE;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    return cuda_status(launch_penalty(*lay, groups, W, eps, lambda, alpha, R, grad, ws, s));
}

bp_status bp_device_status(void *stream) {
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (cudaStreamSynchronize(s) != cudaSuccess) return BP_ERR_CUDA;
    unsigned *p = device_status_ptr();
    if (!p) return BP_ERR_CUDA;
    unsigned v = 0;
    if (cudaMemcpy(&v, p, sizeof(v), cudaMemcpyDeviceToHost) != cudaSuccess) return BP_ERR_CUDA;
    if (v) {
        const unsigned zero = 0;
        if (cudaMemcpy(p, &zero, sizeof(zero), cudaMemcpyHostToDevice) != cudaSuccess)
            return BP_ERR_CUDA;
        return BP_ERR_TIMEOUT;
    }
    return BP_OK;
}

bp_status bp_set_watchdog_ns(uint64_t ns) {
    g_watchdog_ns = ns ? ns : kDefaultWatchdogNs;
    return BP_OK;
}

bp_status bp_debug_drop_stage(int64_t stage) {
    if (stage < -1) return BP_ERR_INVALID_ARG;
    g_drop_stage = stage;
    return BP_OK;
}

}  // extern "C"
