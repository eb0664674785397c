// The block-scaled tcgen05 engine for NVFP4 weights (ffn_bs.cuh) and the
// SwiGLU step that feeds its down projection.
#include "ffn_bs.cuh"
#include "ffn_launch.cuh"

namespace moe {

template <int NT, int PHASE>
static cudaError_t launch_ffn_bs_ph(int grid, const FfnMaps& m, const FfnParams& p,
                                    cudaStream_t st) {
  auto kern = p.det ? ffn_bs_kernel<NT, PHASE, true> : ffn_bs_kernel<NT, PHASE, false>;
  const int smem = BsGeom<NT>::SMEM;
  static std::atomic<unsigned long long> done[2] = {{0}, {0}};  // per variant
  cudaError_t err = set_smem_once(kern, smem, done[p.det ? 1 : 0]);
  if (err != cudaSuccess) return err;
  return launch_k(kern, dim3(grid), dim3(kBsThreads), smem, st, expert_pdl(p), m.a0, m.a1,
                  m.s0, m.s1, m.b, p);
}

template <int NT>
static cudaError_t launch_ffn_bs_nt(int grid, const FfnMaps& m, const FfnParams& p,
                                    cudaStream_t st) {
  return p.phase == 1 ? launch_ffn_bs_ph<NT, 1>(grid, m, p, st)
                      : launch_ffn_bs_ph<NT, 2>(grid, m, p, st);
}

cudaError_t launch_ffn_bs(int nt, int grid, const FfnMaps& m, const FfnParams& p,
                          cudaStream_t st) {
  switch (nt) {
    case 8:
      return launch_ffn_bs_nt<8>(grid, m, p, st);
    case 16:
      return launch_ffn_bs_nt<16>(grid, m, p, st);
    default:
      return cudaErrorInvalidValue;
  }
}

// One wave of the rows kernel: every resident CTA takes the same number of
// rows (within one), so none of them is left running alone at the end.  It
// is launched after the gate/up kernel, not as its programmatic dependent:
// launched early, the wave's CTAs pile up on the SMs whose gate/up CTAs end
// first, and the rest of the SMs get none (measured on the 235B-shaped layer
// at 2048 tokens: 818 us a layer with the early launch, 750 us without).
template <typename K>
static int resident_blocks(K kern, int sms, std::atomic<int>& cache) {
  int per = cache.load();
  if (per <= 0) {
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per, kern, 128, 0) != cudaSuccess ||
        per < 1)
      per = 4;
    cache.store(per);
  }
  return per * sms;
}

template <int G, int NTERM>
static cudaError_t launch_rows_g(int sms, int rows, const FfnParams& p, cudaStream_t st) {
  static std::atomic<int> per{0};
  auto kern = swiglu_terms_rows_kernel<G, NTERM>;
  int blocks = resident_blocks(kern, sms, per);
  if (blocks > rows) blocks = rows;
  return launch_k(kern, dim3(blocks), dim3(128), 0, st, false, p, rows);
}

template <int NTERM>
static cudaError_t launch_rows(int sms, int rows, const FfnParams& p, cudaStream_t st) {
  if (p.I <= 2048) return launch_rows_g<1, NTERM>(sms, rows, p, st);
  if (p.I <= 4096) return launch_rows_g<2, NTERM>(sms, rows, p, st);
  return launch_rows_g<4, NTERM>(sms, rows, p, st);
}

cudaError_t launch_swiglu_terms(int rows, int sms, const FfnParams& p, cudaStream_t st,
                                int nterms) {
  int blocks = rows;
  if (blocks > 8 * sms) blocks = 8 * sms;
  if (blocks < 1) blocks = 1;
  if (rows > kSwigluQuadMaxRows)
    return nterms == kPfTerms ? launch_rows<kPfTerms>(sms, rows, p, st)
                              : launch_rows<kTerms>(sms, rows, p, st);
  return launch_pdl(swiglu_terms_kernel, dim3(blocks), dim3(kSwigluThreads), 0, st, p, rows);
}

}  // namespace moe
