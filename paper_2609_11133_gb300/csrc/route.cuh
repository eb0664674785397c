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
//   waits on another CTA.  Batches routed on the tensor cores (route_tc.cu)
//   run the same grid after the GEMM: each CTA adds the GEMM's partial logits
//   of its experts in slice order instead of the GEMV.
#pragma once

#include "common.cuh"

namespace moe {

constexpr int kMaxK = 32;


// bf16(x / sqrt(mean(x^2) + eps)) of one row by one warp (unit weight, eps
// 1e-6); `out` may be `in`.  The router kernel and the tensor-core router's
// prep kernel both normalise with it, so their rows have the same bits.
__device__ __forceinline__ void rms_norm_row_bf16(const __nv_bfloat16* in, __nv_bfloat16* out,
                                                  int H, int lane) {
  float ss = 0.f;
  for (int h = lane; h < H; h += 32) {
    const float v = __bfloat162float(in[h]);
    ss = fmaf(v, v, ss);
  }
  ss = warp_sum(ss);
  const float r = 1.f / sqrtf(ss / (float)H + 1e-6f);
  __syncwarp();
  for (int h = lane; h < H; h += 32) out[h] = __float2bfloat16_rn(__bfloat162float(in[h]) * r);
}

struct RouteParams {
  const __nv_bfloat16* x;
  const float* wr;
  const float* bias;
  int T, H, E, k, renorm, prenorm, fmt, fused;
  int epb;  // experts per CTA (1, 4 or 8; any count with plog)
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
  // logits from the tensor-core router: partial sums [nsplit, T, ep] added in
  // slice order (no GEMV here); null: the GEMV here
  const float* plog;
  int nsplit, ep;
  // 1: the activation terms of x were written by router_prep_kernel (no rows
  // are staged here)
  int terms_done;
};

// The tensor-core router's two kernels (route_tc.cu): router_prep_kernel
// splits the fp32 router rows into three bf16 parts and, a warp per token,
// writes the RMS-normalised row (prenorm) and the row's activation terms;
// route_tc_kernel multiplies.
struct RouteTcParams {
  const float* wr;          // [E, H]
  const __nv_bfloat16* x;   // [T, H]
  __nv_bfloat16* xn;        // [T, H] normalised rows (prenorm), else unused
  // activation terms of the (normalised) rows for the expert kernels, when
  // act is kActTerms or kActE4M3 (as route_kernel writes them otherwise)
  int act;
  uint8_t* xq;
  uint8_t* xsf;
  float* xinv;
  __nv_bfloat16* w3;        // [3, Ep, H]: wr = w3[0] + w3[1] + w3[2]; rows >= E zero
  float* plog;              // [kRouteTcSplit, T, Ep]
  int T, H, E, Ep, prenorm;
  uint32_t* status;
  uint64_t wait_ns;
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
  uint32_t* status;   // device status word (an expired copy wait)
  uint64_t wait_ns;
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
cudaError_t launch_router_prep(const RouteTcParams& p, cudaStream_t st);
// tmA: rows of x (or xn), tmB: rows of w3; both bf16 boxes of 64 x rows, 128B swizzle
cudaError_t launch_route_tc(const CUtensorMap& tmA, const CUtensorMap& tmB,
                            const RouteTcParams& p, cudaStream_t st);

}  // namespace moe
