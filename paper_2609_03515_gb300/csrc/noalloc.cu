// Workspace-free variant of ikv_decode_attend_score for callers that cannot
// allocate device memory.
//
// Some callers have no way to obtain scratch memory: a serving runtime that
// hands out all device memory at start-up and forbids later cudaMalloc calls,
// an operator hook running inside a host framework that owns the allocator,
// or a latency-critical loop that must avoid cudaMalloc's implicit device
// synchronisation.  For them this file keeps the scratch of one attention +
// score call in a fixed, library-owned device array.
//
// The array lives for as long as the library is loaded on a device (every GPU
// that loads the library holds kStaticScratchBytes of it until the process
// exits).  Its device address is looked up once per device, with that device
// current, on the first call made on it, and kept for the life of the process
// (a cudaDeviceReset would leave the kept address stale, so the entry point is
// not for use after one).  All calls share the array and it
// keeps the last call's contents; the attention path fully writes every
// scratch word before reading it, so nothing needs clearing between calls.
// Two calls whose work overlaps on the GPU (different streams, or different
// host threads on one device) race on the array and must be serialised by the
// caller.
#include <mutex>

#include "ikv_internal.cuh"

namespace {

constexpr size_t kStaticScratchBytes = size_t(16) << 20;  // 16 MiB per device

static __device__ __align__(256) unsigned char g_static_scratch[kStaticScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
void *g_scratch_ptr[kMaxDevices] = {nullptr};

// Device address of g_static_scratch on the current device (set up on first use).
cudaError_t scratch_address(void **out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_mu);
    if (!g_scratch_ptr[dev]) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_static_scratch);
        if (e != cudaSuccess) return e;
        g_scratch_ptr[dev] = p;
    }
    *out = g_scratch_ptr[dev];
    return cudaSuccess;
}

}  // namespace

extern "C" {

size_t ikv_static_scratch_bytes(void) { return kStaticScratchBytes; }

ikv_status ikv_decode_attend_score_static(const ikv_shape *shape, const ikv_cache *cache, int32_t layer,
                                          const void *q, void *out, float *score, float *ema, float alpha,
                                          cudaStream_t stream) {
    size_t need = 0;
    ikv_status st = ikv_attend_workspace_size(shape, cache, &need);
    if (st != IKV_OK) return st;
    if (need > kStaticScratchBytes)
        return ikv::report(IKV_ERR_WORKSPACE,
                           "ikv_decode_attend_score_static: this shape needs %zu bytes of scratch, more than the "
                           "fixed %zu-byte array; use ikv_decode_attend_score with a caller workspace",
                           need, kStaticScratchBytes);
    void *scratch = nullptr;
    cudaError_t e = scratch_address(&scratch);
    if (e != cudaSuccess)
        return ikv::report(IKV_ERR_CUDA, "ikv_decode_attend_score_static: cudaGetSymbolAddress: %s",
                           cudaGetErrorString(e));
    return ikv_decode_attend_score(shape, cache, layer, q, out, score, ema, alpha, scratch, kStaticScratchBytes,
                                   stream);
}

}  // extern "C"
