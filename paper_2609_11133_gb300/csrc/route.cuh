// Router, top-k, permutation and small elementwise kernels of the MoE decode
// layer.
//
// route_kernel (grid = [ceil(E/epb) expert blocks, ceil(T/8) token chunks]):
//   every CTA stages 8 token rows of x in shared memory and computes the fp32
//   logits of epb experts (each warp covers one eighth of H for all of them,
//   float4 loads, shuffle reduction).  The CTA that arrives last at
//   a chunk's ticket does the softmax/top-k of those 8 tokens (one warp per
//   token, k rounds of a warp arg-max with ties to the lower index); in the
//   fused layer it also appends each assignment to its expert's list (an
//   atomic counter per expert), from which the expert kernels build their
//   work plan.  Tickets and counters are reset by their last user; nothing
//   waits on another CTA.
#pragma once

#include "common.cuh"

namespace moe {

constexpr int kMaxK = 32;


struct RouteParams {
  const __nv_bfloat16* x;
  const float* wr;
  const float* bias;
  int T, H, E, k, renorm, prenorm, fmt, fused;
  int epb;  // experts per CTA (1 to 4)
  int act;  // activation form for the expert kernels (kAct*)
  float* logits;  // [T, E]
  int* ids;       // [T, k]
  float* gates;   // [T, k]
  int* ids2;      // optional copies
  float* gates2;
  unsigned* chunk_cnt;
  // fused layer only
  __half* x16;
  uint8_t* xq;   // terms of x (kActTerms, kActE4M3)
  uint8_t* xsf;
  float* xinv;
  float4* zero_a;
  size_t zero_a_n4;
  float4* zero_b;
  size_t zero_b_n4;
  unsigned* acnt;  // [E] assignments per expert, zero on entry
  int* alist;      // [E, T] expert e's assignments t*k + j at alist[e*T + 0..]
};

struct PrepParams {
  const __nv_bfloat16* x;
  int T, H, E, k, fmt;
  int act;
  __half* x16;
  uint8_t* xq;
  uint8_t* xsf;
  float* xinv;
  const int* offsets;  // [E+1] from the permutation
  int* counts;         // [E] (derived here)
  float4* zero_a;
  size_t zero_a_n4;
  float4* zero_b;
  size_t zero_b_n4;
};

// Copy each assignment's activation-term rows (and NVFP4 scale rows) from
// token order into compact-row order (expert by expert, list order inside an
// expert), so that the gate/up kernel reads a chunk's B tile with one box.
struct GatherParams {
  const uint8_t* q;   // [T*terms, qrow] terms of x
  const uint8_t* sf;  // [T*terms, sfrow] their UE4M3 scales, or null
  uint8_t* gq;        // [T*k*terms, qrow]
  uint8_t* gsf;       // [T*k*terms, sfrow] (when sf)
  const unsigned* acnt;
  const int* alist;   // [E, T]
  int* inv;           // [T*k] compact row of each assignment, or null
  int T, k, E, terms, qrow, sfrow;
};

struct CombineParams {
  const float* y_perm;
  const float* topk_w;
  const int* inv;  // row of y_perm of each assignment, or null: row a = assignment a
  int T, k, H;
  const __nv_bfloat16* residual;
  __nv_bfloat16* out;
  unsigned* acnt_reset;  // the fused layer's per-expert counters, zeroed here (or null)
  int E;
};

cudaError_t launch_route(const RouteParams& p, cudaStream_t st);
cudaError_t launch_permute_standalone(const int* ids, int T, int k, int E, int* counts,
                                      int* offsets, int* sorted, int* inv, int* active,
                                      cudaStream_t st);
cudaError_t launch_prep(const PrepParams& p, cudaStream_t st);
cudaError_t launch_combine(const CombineParams& p, cudaStream_t st);
cudaError_t launch_gather(const GatherParams& p, cudaStream_t st);
size_t route_smem_bytes(int H, int E);

}  // namespace moe
