// The NVFP4 prefill engine (ffn_pf.cuh): launches of both phases.
#include "ffn_launch.cuh"
#include "ffn_pf.cuh"

namespace moe {

template <int PHASE>
static cudaError_t launch_ffn_pf_ph(int grid, const FfnMaps& m, const FfnParams& p,
                                    cudaStream_t st) {
  auto kern = ffn_pf_kernel<PHASE>;
  constexpr int smem = PfGeom::SMEM;
  static std::atomic<unsigned long long> done{0};
  cudaError_t err = set_smem_once(kern, smem, done);
  if (err != cudaSuccess) return err;
  return launch_k(kern, dim3(grid), dim3(kPfThreads), smem, st, expert_pdl(p), m.a0, m.a1,
                  m.s0, m.s1, m.b, m.sb, p);
}

cudaError_t launch_ffn_pf(int grid, const FfnMaps& m, const FfnParams& p, cudaStream_t st) {
  return p.phase == 1 ? launch_ffn_pf_ph<1>(grid, m, p, st) : launch_ffn_pf_ph<2>(grid, m, p, st);
}

}  // namespace moe
