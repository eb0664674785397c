// The FP8 tcgen05 engine (ffn_f8.cuh) and the SwiGLU step that feeds its down
// projection.
#include "ffn_f8.cuh"
#include "ffn_launch.cuh"

namespace moe {

template <int NT, int PHASE>
static cudaError_t launch_ffn_f8_ph(int grid, const FfnMaps& m, const FfnParams& p,
                                    cudaStream_t st) {
  auto kern = p.det ? ffn_f8_kernel<NT, PHASE, true> : ffn_f8_kernel<NT, PHASE, false>;
  const int smem = F8Geom<NT, PHASE>::SMEM;
  static std::atomic<unsigned long long> done[2] = {{0}, {0}};  // per variant
  cudaError_t err = set_smem_once(kern, smem, done[p.det ? 1 : 0]);
  if (err != cudaSuccess) return err;
  return launch_k(kern, dim3(grid), dim3(F8Geom<NT, PHASE>::THREADS), smem, st, expert_pdl(p),
                  m.a0, m.a1, m.b, p);
}

template <int NT>
static cudaError_t launch_ffn_f8_nt(int grid, const FfnMaps& m, const FfnParams& p,
                                    cudaStream_t st) {
  return p.phase == 1 ? launch_ffn_f8_ph<NT, 1>(grid, m, p, st)
                      : launch_ffn_f8_ph<NT, 2>(grid, m, p, st);
}

cudaError_t launch_ffn_f8(int nt, int grid, const FfnMaps& m, const FfnParams& p,
                          cudaStream_t st) {
  switch (nt) {
    case 8:
      return launch_ffn_f8_nt<8>(grid, m, p, st);
    case 16:
      return launch_ffn_f8_nt<16>(grid, m, p, st);
    case 32:
      return launch_ffn_f8_nt<32>(grid, m, p, st);
    default:
      return cudaErrorInvalidValue;
  }
}

cudaError_t launch_swiglu_e4m3(int rows, int sms, const FfnParams& p, cudaStream_t st) {
  int blocks = rows;
  if (blocks > 8 * sms) blocks = 8 * sms;
  if (blocks < 1) blocks = 1;
  return launch_pdl(swiglu_e4m3_kernel, dim3(blocks), dim3(128), 0, st, p, rows);
}

}  // namespace moe
