// Expert FFN kernels for FP8 E4M3 weights with 128x128 fp32 block scales.
#include "ffn_launch.cuh"

namespace moe {
MOE_DEFINE_FFN_LAUNCH(1)
MOE_DEFINE_FFN_TC_LAUNCH(1)
}  // namespace moe
