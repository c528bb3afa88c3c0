// flarepp_route_fwd_noalloc: the routing chain for callers that cannot allocate device
// memory when they call it. Examples are a plugin whose host application owns every device
// allocation and gives it no allocator, and a latency-critical loop where cudaMalloc or
// cudaFree would synchronise the device. Such callers cannot provide the workspace that
// flarepp_route_fwd needs.
//
// This entry point uses a fixed scratch area instead: a file-scope __device__ array of
// kNoAllocScratchBytes (64 MiB), which every GPU that loads the library holds until the
// process exits. Host code cannot use the array's name as a device address (in host code
// it names a host-side stand-in), so the first call on each device, with that device
// current, looks the address up once with cudaGetSymbolAddress and caches it. That first
// call should therefore come before any stream capture. The call itself allocates nothing.
#include <cuda_runtime.h>
#include <mutex>

#include "flarepp_internal.h"

namespace flarepp {
namespace {

constexpr size_t kNoAllocScratchBytes = size_t(64) << 20;
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

std::mutex g_noalloc_mu;
void* g_noalloc_addr[kMaxDevices] = {};

// Device address of the scratch array on the current device (looked up once per device).
cudaError_t scratch_address(void** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    if (!g_noalloc_addr[dev]) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess) return e;
        g_noalloc_addr[dev] = p;
    }
    *out = g_noalloc_addr[dev];
    return cudaSuccess;
}

}  // namespace
}  // namespace flarepp

extern "C" flarepp_status flarepp_route_fwd_noalloc(const flarepp_shape* shape, const void* seeds,
                                                    const void* Kt, const void* Vt, const void* K,
                                                    const void* V, float scale, void* Y,
                                                    void* stream) {
    // An invalid shape needs no workspace; flarepp_route_fwd then reports why it is invalid.
    const size_t need = flarepp_route_workspace_bytes(shape);
    if (need > flarepp::kNoAllocScratchBytes) return FLAREPP_ERR_WORKSPACE;
    // The scratch address is the current device's; a stream of another device would run
    // the kernels there against this device's array.
    if (need > 0) {
        int cur = 0, sdev = 0;
        if (cudaGetDevice(&cur) != cudaSuccess ||
            cudaStreamGetDevice((cudaStream_t)stream, &sdev) != cudaSuccess)
            return FLAREPP_ERR_CUDA;
        if (sdev != cur) return FLAREPP_ERR_INVALID_ARGUMENT;
    }
    void* scratch = nullptr;
    if (need > 0 && flarepp::scratch_address(&scratch) != cudaSuccess) return FLAREPP_ERR_CUDA;
    return flarepp_route_fwd(shape, seeds, Kt, Vt, K, V, scale, Y, scratch,
                             need > 0 ? flarepp::kNoAllocScratchBytes : 0, stream);
}
