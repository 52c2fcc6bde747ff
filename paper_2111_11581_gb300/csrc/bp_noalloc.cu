// bp_prune_noalloc: bp_prune for callers that cannot allocate device memory.
//
// bp_prune needs a device workspace from its caller (fp64 scores, keep flags
// and selection tables).  Some callers cannot provide one: code that runs
// under a no-allocation rule once it has started (real-time inference loops,
// plug-ins hosted by a framework that owns all device memory, code that must
// not call cudaMalloc because that call can synchronise the device).  This
// entry point gives them pruning without any allocation: the workspace is a
// fixed array in the library's own device memory, declared below.
//
// The array costs kNoAllocScratchBytes of device memory on every GPU that
// loads the library, for as long as the library stays loaded.  Its device
// address is looked up on every call, with the caller's device current (a
// host-side lookup that allocates nothing), so no address outlives a reset
// of the device's context.  Like bp_prune, the call synchronises its stream
// (the selection reads counts back), so it cannot be used inside a stream
// capture.  Every call uses the same array: calls that can overlap on the GPU
// (different streams, different host threads) race on it and must be
// serialised by the caller.  The array keeps whatever the previous call left;
// bp_prune clears every table it reads before use, so no state carries over
// between calls.
#include "bp_common.cuh"

namespace bp {
namespace {

constexpr size_t kNoAllocScratchBytes = 8u << 20;   // 8 MiB

static __device__ __align__(256) uint8_t g_noalloc_scratch[kNoAllocScratchBytes];

// Device address of the scratch array in the current device's context.  In
// host code g_noalloc_scratch names a host-side stand-in, never the device
// array, so the address must come from the runtime.
bp_status scratch_for_current_device(void **out) {
    void *p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return BP_ERR_CUDA;
    *out = p;
    return BP_OK;
}

}  // namespace
}  // namespace bp

extern "C" bp_status bp_prune_noalloc(const bp_layout *lay, const void *W, double rate,
                                      uint8_t *mask, void *stream) {
    size_t need = 0;
    const bp_status st = bp_workspace_size(lay, &need);
    if (st != BP_OK) return st;
    if (need > bp::kNoAllocScratchBytes) return BP_ERR_WORKSPACE;
    void *scratch = nullptr;
    const bp_status s2 = bp::scratch_for_current_device(&scratch);
    if (s2 != BP_OK) return s2;
    return bp_prune(lay, W, rate, mask, scratch, bp::kNoAllocScratchBytes, stream);
}
