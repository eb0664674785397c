// moe_decode_layer_noalloc: the fused decode layer with its scratch memory in
// a fixed device array owned by this library, for callers that must not
// allocate device memory when they run the layer.
//
// Some callers cannot allocate at call time: an inference engine's plugin
// "enqueue" path is given a stream and its tensors but no allocator and must
// not grow the process's memory, and a latency-critical serving loop cannot
// afford cudaMalloc, which may synchronise the device.  This entry point takes
// only inputs and outputs; its scratch is the file-scope array below.
// moe_noalloc_read_status reads the device status word kept in that array.
#include <cuda_runtime.h>

#include <atomic>
#include <mutex>

#include "../../include/moe.h"
#include "common.cuh"

namespace {

// Scratch of moe_decode_layer_noalloc.  Every GPU that loads this library
// holds these 16 MiB until the process exits.
constexpr size_t kNoAllocBytes = size_t(16) << 20;
__device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocBytes];

// Device address of the array, per device.  It stays null until a lookup
// succeeds, so a lookup that failed (for example inside a stream capture)
// is tried again by the next call.
constexpr int kMaxDevices = 64;
std::mutex g_scratch_mu;
void* g_scratch_ptr[kMaxDevices] = {};
std::atomic<bool> g_status_cleared[kMaxDevices] = {};

// The array's device address on the current device, or null.  Host code
// cannot use the array's name as a device address: the address is looked up
// with that device current.
void* scratch_for_current_device(int* dev_out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  *dev_out = dev;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (g_scratch_ptr[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr) {
      cudaGetLastError();  // leave no sticky error from the failed lookup behind
      return nullptr;
    }
    g_scratch_ptr[dev] = p;
  }
  return g_scratch_ptr[dev];
}

}  // namespace

extern "C" int moe_decode_layer_noalloc(const void* x, const float* router_w,
                                        const float* router_bias, const moe_expert_weights_t* w,
                                        int T, int k, int flags, const void* residual, void* out,
                                        void* stream) {
  size_t need = 0;
  int rc = moe_workspace_size_flags(w, T, k, flags, &need);
  if (rc != MOE_OK) return rc;
  if (need > kNoAllocBytes) return MOE_ERR_WORKSPACE_TOO_SMALL;
  if (T == 0) return MOE_OK;
  int dev = 0;
  void* scratch = scratch_for_current_device(&dev);
  if (scratch == nullptr) return MOE_ERR_CUDA;
  // The array keeps the previous call's contents; clear what must start at
  // zero: the router's ticket counters, the per-expert assignment counters
  // and the shared-tail counters, which lie between the status word and the
  // routing logits in the workspace layout.  The status word is cleared by
  // the first call on a device only, so that moe_noalloc_read_status reports
  // an error of any call since the last read.
  const moe::WsLayout L = moe::ws_layout(T, k, w->E, w->H, w->I);
  const size_t from = g_status_cleared[dev] ? L.acnt : 0;
  if (cudaMemsetAsync(static_cast<char*>(scratch) + from, 0, L.logits - from,
                      static_cast<cudaStream_t>(stream)) != cudaSuccess)
    return MOE_ERR_CUDA;
  g_status_cleared[dev] = true;
  return moe_decode_layer(x, router_w, router_bias, w, T, k, flags, residual, out, scratch,
                          kNoAllocBytes, stream);
}

extern "C" int moe_noalloc_read_status(int* status, void* stream) {
  if (!status) return MOE_ERR_INVALID_ARG;
  int dev = 0;
  void* scratch = scratch_for_current_device(&dev);
  if (scratch == nullptr) return MOE_ERR_CUDA;
  return moe_read_status(scratch, kNoAllocBytes, status, stream);
}
