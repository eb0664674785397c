// Expert FFN kernels for FP8 E4M3 weights with 128x128 fp32 block scales.
#include "ffn_launch.cuh"

namespace moe {
MOE_DEFINE_FFN_LAUNCH(1)
MOE_DEFINE_SWIGLU_LAUNCH(1)
cudaError_t launch_finalize(int sms, const FfnParams& p, cudaStream_t st) {
  size_t blocks = ((size_t)p.T * p.H / 4 + 255) / 256;
  if (blocks > (size_t)(4 * sms)) blocks = 4 * sms;
  if (blocks < 1) blocks = 1;
  return launch_pdl(finalize_kernel, dim3((unsigned)blocks), dim3(256), 0, st, p);
}
}  // namespace moe
