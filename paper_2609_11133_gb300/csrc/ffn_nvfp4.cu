// Expert FFN kernels for NVFP4 weights (E2M1 codes, per-16 E4M3 scales,
// fp32 tensor scale).
#include "ffn_launch.cuh"

namespace moe {
MOE_DEFINE_FFN_LAUNCH(2)
MOE_DEFINE_SWIGLU_LAUNCH(2)
}  // namespace moe
