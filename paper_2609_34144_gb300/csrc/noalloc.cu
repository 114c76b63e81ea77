// Routing entry point that needs no device allocation from its caller.
//
// Some callers cannot call cudaMalloc (or any allocator) at the point where they route:
// plugins that run inside a host framework which owns every device allocation and forbids
// allocating during execution, real-time loops that must not take the allocator's locks or
// its implicit synchronisation, and fixed-budget embedded runtimes.  For them the routing
// scratch lives in a file-scope device array of a fixed size that the library reserves on
// every GPU where the library is loaded, for the life of the process.
#include <cuda_runtime.h>

#include <mutex>

#include "internal.h"

namespace cast {
namespace {

constexpr size_t kNoAllocScratchBytes = size_t(16) << 20;   // 16 MiB
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_route_scratch[kNoAllocScratchBytes];

std::mutex g_setup_mu;
void* g_scratch_ptr[kMaxDevices] = {};

// Device address of g_route_scratch on the current device, looked up once per device and kept
// for the life of the process (a context torn down by cudaDeviceReset would invalidate it; the
// header tells callers not to use this entry point after a reset).
cast_status scratch_for_current_device(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(CAST_ERR_CUDA, "cast_route_topk_noalloc: %s", cudaGetErrorString(e));
  if (dev < 0 || dev >= kMaxDevices)
    return fail(CAST_ERR_UNSUPPORTED, "cast_route_topk_noalloc: device %d above %d", dev, kMaxDevices);
  std::lock_guard<std::mutex> lock(g_setup_mu);
  if (!g_scratch_ptr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_route_scratch);
    if (e != cudaSuccess || !p)
      return fail(CAST_ERR_CUDA, "cast_route_topk_noalloc: cudaGetSymbolAddress failed: %s",
                  cudaGetErrorString(e));
    g_scratch_ptr[dev] = p;
  }
  *out = g_scratch_ptr[dev];
  return CAST_OK;
}

}  // namespace
}  // namespace cast

extern "C" cast_status cast_route_topk_noalloc(const cast_route_args* a, void* stream) {
  using namespace cast;
  if (!a) return fail(CAST_ERR_INVALID_ARG, "cast_route_topk_noalloc: args is NULL");
  const size_t need = cast_route_workspace_size(a);
  if (need > kNoAllocScratchBytes)
    return fail(CAST_ERR_UNSUPPORTED,
                "cast_route_topk_noalloc: this problem needs %zu B of scratch, above the fixed "
                "%zu B (16 MiB) limit; use cast_route_topk with a caller workspace",
                need, kNoAllocScratchBytes);
  void* scratch = nullptr;
  const cast_status s = scratch_for_current_device(&scratch);
  if (s != CAST_OK) return s;
  // The routing kernels overwrite every scratch word they read, so nothing needs clearing.
  return cast_route_topk(a, scratch, kNoAllocScratchBytes, stream);
}
