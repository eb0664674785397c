// moe_decode_layer_noalloc: the fused decode layer with its scratch memory in
// a fixed device array owned by this library, for callers that must not
// allocate device memory when they run the layer.
//
// Some callers cannot allocate at call time: an inference engine's plugin
// "enqueue" path is given a stream and its tensors but no allocator and must
// not grow the process's memory, and a latency-critical serving loop cannot
// afford cudaMalloc, which may synchronise the device.  This entry point takes
// only inputs and outputs; its scratch is the file-scope array below.
#include <cuda_runtime.h>

#include <mutex>

#include "../../include/moe.h"
#include "common.cuh"

namespace {

// Scratch of moe_decode_layer_noalloc.  Every GPU that loads this library
// holds these 16 MiB until the process exits.
constexpr size_t kNoAllocBytes = size_t(16) << 20;
__device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocBytes];

struct DevScratch {
  std::once_flag once;
  void* ptr = nullptr;
  cudaError_t err = cudaSuccess;
};
DevScratch g_scratch[64];

}  // namespace

extern "C" int moe_decode_layer_noalloc(const void* x, const float* router_w,
                                        const float* router_bias, const moe_expert_weights_t* w,
                                        int T, int k, int flags, const void* residual, void* out,
                                        void* stream) {
  size_t need = 0;
  int rc = moe_workspace_size(w, T, k, &need);
  if (rc != MOE_OK) return rc;
  if (need > kNoAllocBytes) return MOE_ERR_WORKSPACE_TOO_SMALL;
  if (T == 0) return MOE_OK;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return MOE_ERR_CUDA;
  // Host code cannot use the array's name as a device address: look the
  // address up once per device, with that device current.
  DevScratch& d = g_scratch[dev];
  std::call_once(d.once, [&] {
    d.err = cudaGetSymbolAddress(&d.ptr, g_noalloc_scratch);
  });
  if (d.err != cudaSuccess || d.ptr == nullptr) return MOE_ERR_CUDA;
  // The array keeps the previous call's contents; clear what must start at
  // zero: the device status word and the router's ticket counters, which lie
  // in front of the routing logits in the workspace layout.
  const size_t control = moe::ws_layout(T, k, w->E, w->H, w->I).logits;
  if (cudaMemsetAsync(d.ptr, 0, control, static_cast<cudaStream_t>(stream)) != cudaSuccess)
    return MOE_ERR_CUDA;
  return moe_decode_layer(x, router_w, router_bias, w, T, k, flags, residual, out, d.ptr,
                          kNoAllocBytes, stream);
}
