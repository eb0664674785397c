// Router, top-k, permutation and small elementwise kernels of the MoE decode
// layer.
//
// route_kernel (grid = [ceil(E/4) expert blocks, ceil(T/8) token chunks]):
//   every CTA stages 8 token rows of x in shared memory and computes the fp32
//   logits of 4 experts (two warps per expert row of the router, one half of
//   H each, float4 loads, shuffle reduction).  The CTA that arrives last at a chunk's ticket does
//   the softmax/top-k of those 8 tokens (one warp per token, k rounds of a
//   warp arg-max with ties to the lower index); in the fused layer the CTA
//   that completes the last chunk builds the token->expert permutation and
//   the work plan of the expert kernels.  Tickets are atomic counters reset
//   by their last user; nothing waits on another CTA.
#pragma once

#include "common.cuh"

namespace moe {

constexpr int kMaxK = 32;

// Activation forms the expert engines read.
constexpr int kActF16 = 0;      // f16 rows (power-of-two scaled), natural order
constexpr int kActF16Perm = 1;  // f16 rows in the warp-MMA NVFP4 unit order
constexpr int kActTerms = 2;    // four NVFP4 terms per row (block-scaled engine)

struct RouteParams {
  const __nv_bfloat16* x;
  const float* wr;
  const float* bias;
  int T, H, E, k, renorm, prenorm, fmt, fused, nt;
  int act;  // activation form for the expert kernels (kAct*)
  float* logits;  // [T, E]
  int* ids;       // [T, k]
  float* gates;   // [T, k]
  int* ids2;      // optional copies
  float* gates2;
  unsigned* chunk_cnt;
  unsigned* done_cnt;
  // fused layer only
  __half* x16;
  uint8_t* xq;   // NVFP4 terms of x (kActTerms)
  uint8_t* xsf;
  float* xinv;
  float4* zero_a;
  size_t zero_a_n4;
  float4* zero_b;
  size_t zero_b_n4;
  int* counts;
  int* offsets;
  int* sorted;
  int* inv;
  int* active;
  int* cprefix;
  uint32_t* status;
};

struct PrepParams {
  const __nv_bfloat16* x;
  int T, H, E, k, fmt, nt;
  int act;
  __half* x16;
  uint8_t* xq;
  uint8_t* xsf;
  float* xinv;
  const int* offsets;  // [E+1] from the permutation
  const int* active;   // [E+1]
  int* counts;         // [E] (derived here)
  int* cprefix;        // [E+1]
  float4* zero_a;
  size_t zero_a_n4;
  float4* zero_b;
  size_t zero_b_n4;
};

struct CombineParams {
  const float* y_perm;
  const float* topk_w;
  const int* inv;
  int T, k, H;
  const __nv_bfloat16* residual;
  __nv_bfloat16* out;
};

cudaError_t launch_route(const RouteParams& p, cudaStream_t st);
cudaError_t launch_permute_standalone(const int* ids, int T, int k, int E, int* counts,
                                      int* offsets, int* sorted, int* inv, int* active,
                                      cudaStream_t st);
cudaError_t launch_prep(const PrepParams& p, cudaStream_t st);
cudaError_t launch_combine(const CombineParams& p, cudaStream_t st);
size_t route_smem_bytes(int H, int E);

}  // namespace moe
