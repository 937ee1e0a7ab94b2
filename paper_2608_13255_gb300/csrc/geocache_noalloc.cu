// geocache_transport_step_noalloc: the cached step without a caller-provided
// workspace.  Its scratch is a fixed array in the library's device image, so
// a call needs no device allocation by anybody.
//
// Who needs this: callers that cannot hand the library a scratch buffer at
// the point where they run a step -- for example code whose device memory is
// owned by another component (a framework's caching allocator or a fixed
// arena) with no way to obtain a temporary buffer there, or serving loops
// that must not allocate once they are running because cudaMalloc can
// synchronise the device and stall for milliseconds.
#include <cuda_runtime.h>

#include <cstdint>
#include <mutex>

#include "geocache.h"
#include "geocache_internal.h"

namespace {

// Scratch shared by every call of the entry point on a device; loaded with
// the library and held until the process exits.
constexpr int64_t kNoallocFloats = GEOCACHE_NOALLOC_MAX_WORKSPACE_FLOATS;
static __device__ __align__(256) float g_noalloc_scratch[kNoallocFloats];

constexpr int kMaxDevices = 64;
std::mutex g_setup_mutex;
float* g_scratch_ptr[kMaxDevices] = {};

// Device address of the scratch array on the current device, looked up once
// per device (the host-side name g_noalloc_scratch is not a device address).
cudaError_t scratch_address(float** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_setup_mutex);
    if (!g_scratch_ptr[dev]) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess) return e;
        g_scratch_ptr[dev] = static_cast<float*>(p);
    }
    *out = g_scratch_ptr[dev];
    return cudaSuccess;
}

}  // namespace

extern "C" int geocache_transport_step_noalloc(const geocache_corr* corr, const int32_t* anchors, int a, int C,
                                               const float* x0_anchor_new, const float* x0_prev, float* x0_out,
                                               const void* x_t, void* x_next, geocache_dtype lat_dtype,
                                               const geocache_recon* recon, void* stream) {
    // only a sparse-mode step with a view outside the anchor set uses scratch,
    // at least max_records * C floats (the whole array is passed, so the
    // increment-plane path runs whenever the array also holds the plane)
    const int64_t need = (corr && a < corr->N && corr->mode == GEOCACHE_CORR_SPARSE && corr->max_records > 0 && C > 0)
                             ? corr->max_records * (int64_t)C
                             : 0;
    if (need > kNoallocFloats)
        return geocache::set_error(GEOCACHE_ESHAPE,
                                   "geocache_transport_step_noalloc: this step needs %lld floats of scratch but the "
                                   "built-in array holds %lld; use geocache_transport_step with a workspace",
                                   (long long)need, (long long)kNoallocFloats);
    float* scratch = nullptr;
    if (need > 0) {
        const cudaError_t e = scratch_address(&scratch);
        if (e != cudaSuccess)
            return geocache::set_error(GEOCACHE_ECUDA,
                                       "geocache_transport_step_noalloc: looking up the scratch array: %s (%s)",
                                       cudaGetErrorName(e), cudaGetErrorString(e));
    }
    return geocache_transport_step(corr, anchors, a, C, x0_anchor_new, x0_prev, x0_out, x_t, x_next, lat_dtype, recon,
                                   scratch, need > 0 ? kNoallocFloats : 0, stream);
}
