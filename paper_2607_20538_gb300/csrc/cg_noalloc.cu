// cg_noalloc.cu -- cg_kivi_append_static: the KIVI stream append for callers that cannot
// allocate device memory.
//
// cg_kivi_append stages the tokens of a completed key group in a workspace that the caller
// allocates. Some callers cannot allocate: code that runs inside a framework's memory pool
// with no hook for extra buffers, a process whose device memory is reserved up front, or a
// real-time loop where an allocation could block or fail at the wrong moment. This entry
// point takes the workspace from a fixed array in the library's own device memory instead.
//
// The array holds CG_KIVI_APPEND_STATIC_BYTES (32 MiB). Its address is looked up once per
// device, on the first call made with that device current; make that first call before any
// stream capture. No call allocates or frees memory. All calls share the one array: calls
// whose kernels overlap on the GPU (different streams, or graphs replayed concurrently)
// race on it, so serialize them. Nothing in the array needs to start at zero: an append
// writes every byte of it that it reads, before reading it.
#include <mutex>

#include "cg_launch.h"

#define CG_EXPORT __attribute__((visibility("default")))

namespace cg {
namespace {

__device__ __align__(256) unsigned char g_append_scratch[CG_KIVI_APPEND_STATIC_BYTES];

// Device address of the array on the current device (set up once per device).
int append_scratch(void** out) {
    static std::mutex mu;
    static void* ptrs[64] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return set_error(CG_ECUDA, "cudaGetDevice failed");
    if (dev < 0 || dev >= 64) return set_error(CG_EUNSUPPORTED, "device ordinal out of range");
    std::lock_guard<std::mutex> lk(mu);
    if (!ptrs[dev]) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_append_scratch);
        if (e != cudaSuccess) return set_error(CG_ECUDA, "cudaGetSymbolAddress of the append scratch failed");
        ptrs[dev] = p;
    }
    *out = ptrs[dev];
    return CG_OK;
}

}  // namespace
}  // namespace cg

extern "C" CG_EXPORT int cg_kivi_append_static(const cg_shape* shape, const cg_params* params, const void* kv_new_bf16,
                                               const float* gauges, void* codes, void* scales, void* ring,
                                               void* stream) {
    size_t need = 0;
    int rc = cg_kivi_stream_bytes(shape, params, nullptr, nullptr, nullptr, &need);
    if (rc) return rc;
    if (need > (size_t)CG_KIVI_APPEND_STATIC_BYTES)
        return cg::set_error(CG_ERANGE, "cg_kivi_append_static: this shape stages up to %zu bytes per append, more "
                             "than the %zu-byte static workspace; call it per layer (L = 1) or use cg_kivi_append",
                             need, (size_t)CG_KIVI_APPEND_STATIC_BYTES);
    void* scratch = nullptr;
    if ((rc = cg::append_scratch(&scratch))) return rc;
    return cg_kivi_append(shape, params, kv_new_bf16, gauges, codes, scales, ring, scratch,
                          (size_t)CG_KIVI_APPEND_STATIC_BYTES, stream);
}
