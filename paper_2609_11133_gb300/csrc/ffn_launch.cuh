// Host-side launchers of the expert FFN kernels (one translation unit per
// weight format keeps compile times short).
#pragma once

#include "ffn.cuh"

namespace moe {

// Launch `kern` as a programmatic dependent of the previous kernel on the
// stream (pdl: its blocks may start while that kernel finishes; the kernel
// calls griddepcontrol.wait before reading what the previous kernel wrote),
// or after it (!pdl).
template <typename... KArgs, typename... Args>
cudaError_t launch_k(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem,
                     cudaStream_t st, bool pdl, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, args...);
}

template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t st, Args... args) {
  return launch_k(kern, grid, block, smem, st, true, args...);
}

// Whether an expert kernel of the tensor-core engines starts as a programmatic
// dependent of the kernel before it.  The persistent grid divides its stages
// by CTA index and assumes every CTA starts at once; launched early behind a
// large gather (at least 2048 assignment rows), its CTAs start as the
// gather's SMs free up and the last ones finish late.  Measured in graphs of
// layer calls, gate/up without / with the early start: FP8 480B-shaped T=512
// 1511 / 1539 us a layer, FP8 Zipf T=256 1280 / 1286; below 2048 rows the
// early start pays (FP8 Zipf T=128 819 / 809 us; the NVFP4 94-layer stack at
// T=128 26.40 / 26.14 ms, of which 0.19 ms came from the down kernel).
inline bool expert_pdl(const FfnParams& p) {
  return !(p.phase == 1 && p.b_compact && (long long)p.T * p.k >= 2048);
}

struct FfnMaps {
  CUtensorMap a0, a1, s0, s1, b;
  CUtensorMap sb;  // prefill engine: the activation terms' scales
};

// Instantiated in ffn_fp8.cu (FMT = 1) and ffn_nvfp4.cu (FMT = 2).
template <int FMT>
cudaError_t launch_ffn(int nt, int grid, const FfnMaps& maps, const FfnParams& p,
                       cudaStream_t st, bool pdl);

template <int FMT>
int ffn_smem_bytes(int nt);

// SwiGLU between the phases and the bf16 conversion after them.
template <int FMT>
cudaError_t launch_swiglu(int rows, int sms, const FfnParams& p, bool perm, cudaStream_t st);
cudaError_t launch_finalize(int sms, const FfnParams& p, cudaStream_t st);

// The block-scaled tcgen05 engine for NVFP4 (ffn_bs.cuh, instantiated in
// ffn_bs.cu); nt in {8, 16}.  SwiGLU into NVFP4 terms for its down step.
cudaError_t launch_ffn_bs(int nt, int grid, const FfnMaps& maps, const FfnParams& p,
                          cudaStream_t st);
// SwiGLU into NVFP4 terms; batches of more than kSwigluQuadMaxRows rows may
// write only the first `nterms` of the four terms (the prefill engine reads
// kPfTerms).
cudaError_t launch_swiglu_terms(int rows, int sms, const FfnParams& p, cudaStream_t st,
                                int nterms = 4);

// The FP8 tcgen05 engine (ffn_f8.cuh, instantiated in ffn_f8tc.cu); nt in
// {8, 16, 32}.  SwiGLU into E4M3 terms for its down step.
cudaError_t launch_ffn_f8(int nt, int grid, const FfnMaps& maps, const FfnParams& p,
                          cudaStream_t st);
cudaError_t launch_swiglu_e4m3(int rows, int sms, const FfnParams& p, cudaStream_t st);

// The NVFP4 prefill engine (ffn_pf.cuh, instantiated in ffn_pf.cu): maps as
// for the decode engine, with b and sb 3-D maps of the term arrays [rows, 4,
// K/2] and their scales [rows, 4, K/16], boxes of 3 terms x 64 rows.
cudaError_t launch_ffn_pf(int grid, const FfnMaps& maps, const FfnParams& p, cudaStream_t st);


#define MOE_DEFINE_FFN_LAUNCH(FMTV)                                                            \
  template <int NT>                                                                             \
  static cudaError_t launch_ffn_nt_##FMTV(int grid, const FfnMaps& m, const FfnParams& p,      \
                                          cudaStream_t st, bool pdl) {                          \
    constexpr int KS = (NT == 32) ? 1 : 2;                                                      \
    auto kern = ffn_kernel<FMTV, NT, KS>;                                                       \
    const int smem = StageGeom<FMTV, NT>::SMEM;                                                 \
    static std::atomic<unsigned long long> done{0};                                             \
    cudaError_t err = set_smem_once(kern, smem, done);                                          \
    if (err != cudaSuccess) return err;                                                         \
    cudaLaunchConfig_t cfg = {};                                                                \
    cfg.gridDim = dim3(grid);                                                                   \
    cfg.blockDim = dim3(ffn_threads<KS>());                                                     \
    cfg.dynamicSmemBytes = smem;                                                                \
    cfg.stream = st;                                                                            \
    cudaLaunchAttribute attr[1];                                                                \
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;                            \
    attr[0].val.programmaticStreamSerializationAllowed = 1;                                     \
    cfg.attrs = attr;                                                                           \
    cfg.numAttrs = pdl ? 1 : 0;                                                                 \
    return cudaLaunchKernelEx(&cfg, kern, m.a0, m.a1, m.s0, m.s1, m.b, p);                      \
  }                                                                                             \
  template <>                                                                                   \
  cudaError_t launch_ffn<FMTV>(int nt, int grid, const FfnMaps& m, const FfnParams& p,         \
                               cudaStream_t st, bool pdl) {                                     \
    switch (nt) {                                                                               \
      case 8:                                                                                   \
        return launch_ffn_nt_##FMTV<8>(grid, m, p, st, pdl);                                    \
      case 16:                                                                                  \
        return launch_ffn_nt_##FMTV<16>(grid, m, p, st, pdl);                                   \
      case 32:                                                                                  \
        return launch_ffn_nt_##FMTV<32>(grid, m, p, st, pdl);                                   \
      default:                                                                                  \
        return cudaErrorInvalidValue;                                                           \
    }                                                                                           \
  }                                                                                             \
  template <>                                                                                   \
  int ffn_smem_bytes<FMTV>(int nt) {                                                            \
    return nt == 8 ? StageGeom<FMTV, 8>::SMEM                                                   \
                   : (nt == 16 ? StageGeom<FMTV, 16>::SMEM : StageGeom<FMTV, 32>::SMEM);        \
  }

#define MOE_DEFINE_SWIGLU_LAUNCH(FMTV)                                                         \
  template <>                                                                                   \
  cudaError_t launch_swiglu<FMTV>(int rows, int sms, const FfnParams& p, bool perm,            \
                                  cudaStream_t st) {                                            \
    int blocks = rows;                                                                          \
    if (blocks > 8 * sms) blocks = 8 * sms;                                                     \
    if (blocks < 1) blocks = 1;                                                                 \
    return launch_pdl(swiglu_kernel<FMTV>, dim3(blocks), dim3(256), 0, st, p, rows,            \
                      perm ? 1 : 0);                                                            \
  }

}  // namespace moe
