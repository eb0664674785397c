// Tensor-core router for large batches: logits[t, e] = sum_h x[t, h] * wr[e, h]
// (the fp32 router GEMV of the decode layer, step a1) as a bf16 GEMM on the
// tcgen05 tensor cores.
//
// Exactness.  x is bf16.  Each fp32 router weight w is written as the sum of
// three bf16 values, w0 = bf16(w), w1 = bf16(w - w0), w2 = bf16(w - w0 - w1):
// the first residual keeps at most 16 significant bits and the second at most
// 8, so w2 takes the rest exactly and w0 + w1 + w2 == w (for |w| >= 2^-110,
// where no residual falls below bf16's subnormals).  Every product of a bf16 x
// with a bf16 part is exact in fp32, so the GEMM x . (w0 + w1 + w2) differs
// from the fp32 GEMV only in the order of its fp32 additions.
//
// Work.  A CTA takes 128 tokens (the MMA's M) against every expert (N = E
// rounded up to 16, at most 256) over one of kRouteTcSplit slices of the K
// range, where K runs over (K-block of 64, part): per stage one TMA box of x
// (128 rows x 64) and one of the part's rows (Ep x 64), four MMAs of K = 16
// into one tensor-memory accumulator.  The epilogue writes the slice's fp32
// partial logits; the router kernel adds the slices in order, then does the
// softmax, top-k and the rest of the routing.
#include "act_terms.cuh"
#include "route.cuh"

namespace moe {
namespace {

constexpr int kTcThreads = 192;  // warp 0 TMA producer, warp 1 MMA issuer, warps 2-5 epilogue
constexpr int kTcM = 128;        // tokens per tile (MMA M)
constexpr int kTcK = 64;         // K elements per stage: one 128-byte swizzled row of bf16
constexpr int kTcMaxStages = 8;
constexpr uint32_t kTcABytes = kTcM * kTcK * 2;
constexpr uint32_t kTcRingBytes = 200u * 1024u;
constexpr uint32_t kTcTmemCols = 256;

// Instruction descriptor of kind::f16: f32 D, bf16 A and B, both K-major.
__host__ __device__ constexpr uint32_t tc_idesc_bf16(int M, int N) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(N >> 3) << 17) |
         ((uint32_t)(M >> 4) << 24);
}

__device__ __forceinline__ void tc_mma_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                            uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.u32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

__host__ __device__ inline uint32_t tc_stage_bytes(int Ep) {
  return (kTcABytes + (uint32_t)Ep * kTcK * 2 + 1023u) & ~1023u;
}
__host__ __device__ inline int tc_stages(int Ep) {
  const int s = (int)(kTcRingBytes / tc_stage_bytes(Ep));
  return s > kTcMaxStages ? kTcMaxStages : s;
}

// One fp32 router weight as three bf16 parts whose sum is the weight.
__device__ __forceinline__ void split3(float w, __nv_bfloat16& a, __nv_bfloat16& b,
                                       __nv_bfloat16& c) {
  a = __float2bfloat16_rn(w);
  const float r1 = w - __bfloat162float(a);
  b = __float2bfloat16_rn(r1);
  c = __float2bfloat16_rn(r1 - __bfloat162float(b));
}

// Blocks [0, nsplit): the router rows as three bf16 parts (rows E..Ep-1 zero).
// Blocks after them, a warp per token row: the RMS-normalised row (prenorm)
// and the row's activation terms (the same codes route_kernel writes).
__global__ void __launch_bounds__(256) router_prep_kernel(const RouteTcParams p, int nsplit) {
  pdl_launch_dependents();
  if ((int)blockIdx.x < nsplit) {
    const size_t n4 = (size_t)p.Ep * p.H / 4;
    const size_t part = (size_t)p.Ep * p.H;
    for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < n4;
         i += (size_t)nsplit * blockDim.x) {
      const size_t e = i * 4 / p.H;
      const size_t h = i * 4 - e * p.H;
      float4 w = make_float4(0.f, 0.f, 0.f, 0.f);
      if ((int)e < p.E) w = __ldg(reinterpret_cast<const float4*>(p.wr + e * p.H + h));
      __nv_bfloat16 q[3][4];
      split3(w.x, q[0][0], q[1][0], q[2][0]);
      split3(w.y, q[0][1], q[1][1], q[2][1]);
      split3(w.z, q[0][2], q[1][2], q[2][2]);
      split3(w.w, q[0][3], q[1][3], q[2][3]);
#pragma unroll
      for (int j = 0; j < 3; ++j)
        *reinterpret_cast<uint2*>(p.w3 + j * part + e * p.H + h) =
            *reinterpret_cast<const uint2*>(q[j]);
    }
    return;
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int t = ((int)blockIdx.x - nsplit) * 8 + warp;
  if (t >= p.T) return;
  const __nv_bfloat16* row = p.x + (size_t)t * p.H;
  if (p.prenorm) {
    rms_norm_row_bf16(row, p.xn + (size_t)t * p.H, p.H, lane);
    row = p.xn + (size_t)t * p.H;
    __syncwarp();  // the warp's own stores of the row are read back below
  }
  if (p.act == kActTerms)
    convert_row_terms(row, p.H, t, p.xq, p.xsf, p.xinv + t, lane);
  else if (p.act == kActE4M3)
    convert_row_e4m3(row, p.H, t, p.xq, p.xinv + t, lane);
}

__global__ void __launch_bounds__(kTcThreads, 1)
    route_tc_kernel(const __grid_constant__ CUtensorMap tmA,
                    const __grid_constant__ CUtensorMap tmB, const RouteTcParams p) {
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  __shared__ __align__(8) uint64_t full_bar[kTcMaxStages];
  __shared__ __align__(8) uint64_t empty_bar[kTcMaxStages];
  __shared__ __align__(8) uint64_t done_bar;
  __shared__ uint32_t s_tmem;
  __shared__ volatile int s_abort;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int Ep = p.Ep;
  const uint32_t stage_bytes = tc_stage_bytes(Ep);
  const int S = tc_stages(Ep);
  const int m0 = blockIdx.x * kTcM;
  const int split = blockIdx.y;
  const int Q = 3 * (p.H / kTcK);  // stages of the whole K range: (K-block, part)
  const int q_begin = (int)((long long)Q * split / kRouteTcSplit);
  const int nq = (int)((long long)Q * (split + 1) / kRouteTcSplit) - q_begin;

  if (threadIdx.x == 0) {
    s_abort = 0;
    for (int i = 0; i < S; ++i) {
      mbar_init(&full_bar[i], 1);
      mbar_init(&empty_bar[i], 1);
    }
    mbar_init(&done_bar, 1);
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(&s_tmem, kTcTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s_tmem;
  pdl_wait();  // the router parts (and the normalised rows) come from the prep kernel
  pdl_launch_dependents();

  // ================================================================ producer
  if (warp == 0) {
    if (lane == 0) {
      tma_prefetch_desc(&tmA);
      tma_prefetch_desc(&tmB);
      const uint64_t pol = policy_evict_last();  // each tile is read by several CTAs
      int issued = 0;
      for (int i = 0; i < nq; ++i) {
        const int slot = i % S;
        const uint32_t par = (uint32_t)(i / S) & 1u;
        if (!mbar_wait_bounded(&empty_bar[slot], par ^ 1u, p.wait_ns, &s_abort)) {
          set_status(p.status, kStatusTimeoutRoute);
          s_abort = 1;
          break;
        }
        const int q = q_begin + i, kb = q / 3, part = q - 3 * kb;
        unsigned char* st = smem + (size_t)slot * stage_bytes;
        mbar_arrive_expect_tx(&full_bar[slot], kTcABytes + (uint32_t)Ep * kTcK * 2);
        tma_load_2d(st, &tmA, &full_bar[slot], kb * kTcK, m0, pol);
        tma_load_2d(st + kTcABytes, &tmB, &full_bar[slot], kb * kTcK, part * Ep, pol);
        ++issued;
      }
      // every copy lands before the CTA exits
      for (int j = issued > S ? issued - S : 0; j < issued; ++j)
        mbar_wait_bounded(&full_bar[j % S], (uint32_t)(j / S) & 1u, p.wait_ns, nullptr);
    }
    return;
  }

  // ================================================================ MMA issuer
  if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = tc_idesc_bf16(kTcM, Ep);
      bool ok = true;
      for (int i = 0; i < nq; ++i) {
        const int slot = i % S;
        if (!mbar_wait_bounded(&full_bar[slot], (uint32_t)(i / S) & 1u, p.wait_ns, &s_abort)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t st = smem_u32(smem + (size_t)slot * stage_bytes);
#pragma unroll
        for (int kk = 0; kk < kTcK / 16; ++kk)
          tc_mma_bf16(tmem, tc_desc_sw128(st + 32 * kk), tc_desc_sw128(st + kTcABytes + 32 * kk),
                      idesc, (i > 0 || kk > 0) ? 1u : 0u);
        tc_commit(&empty_bar[slot]);
      }
      if (!ok) {
        set_status(p.status, kStatusTimeoutRoute);
        s_abort = 1;
      }
      // arrives when every MMA issued above has completed
      tc_commit(&done_bar);
      mbar_wait_bounded(&done_bar, 0, p.wait_ns, nullptr);
    }
    __syncwarp();
    asm volatile("bar.sync 1, 160;" ::: "memory");  // warps 1-5: the epilogue has read TMEM
    tc_fence_after();
    tmem_dealloc(tmem, kTcTmemCols);
    return;
  }

  // ================================================================ epilogue
  // Warp w reads TMEM lanes 32*(w%4)..+31: token rows m0 + 32*(w%4) + lane.
  {
    const int quad = warp & 3;
    const int row = m0 + quad * 32 + lane;
    int ok = 0;
    if (lane == 0) ok = mbar_wait_bounded(&done_bar, 0, p.wait_ns, &s_abort) && !s_abort;
    ok = __shfl_sync(0xffffffffu, ok, 0);
    __syncwarp();
    tc_fence_after();
    if (ok) {
      const uint32_t taddr = tmem + ((uint32_t)(quad * 32) << 16);
      float* dst = p.plog + ((size_t)split * p.T + (row < p.T ? row : 0)) * Ep;
      for (int c0 = 0; c0 < Ep; c0 += 16) {
        uint32_t v[16];
        tmem_ld16(taddr + (uint32_t)c0, v);
        tmem_ld_wait();
        if (row < p.T) {
#pragma unroll
          for (int i = 0; i < 4; ++i)
            *reinterpret_cast<float4*>(dst + c0 + 4 * i) =
                make_float4(__uint_as_float(v[4 * i]), __uint_as_float(v[4 * i + 1]),
                            __uint_as_float(v[4 * i + 2]), __uint_as_float(v[4 * i + 3]));
        }
      }
    }
    tc_fence_before();
    asm volatile("bar.sync 1, 160;" ::: "memory");
  }
}

}  // namespace

cudaError_t launch_router_prep(const RouteTcParams& p, cudaStream_t st) {
  const size_t n4 = (size_t)p.Ep * p.H / 4;
  int nsplit = (int)((n4 + 4 * 256 - 1) / (4 * 256));  // four float4 per thread
  if (nsplit < 1) nsplit = 1;
  const bool rows = p.prenorm || p.act == kActTerms || p.act == kActE4M3;
  const int nnorm = rows ? (p.T + 7) / 8 : 0;
  router_prep_kernel<<<nsplit + nnorm, 256, 0, st>>>(p, nsplit);
  return cudaGetLastError();
}

cudaError_t launch_route_tc(const CUtensorMap& tmA, const CUtensorMap& tmB,
                            const RouteTcParams& p, cudaStream_t st) {
  static std::atomic<unsigned long long> done{0};
  const int smax = (int)(kTcRingBytes + 1024u);
  cudaError_t err = set_smem_once(route_tc_kernel, smax, done);
  if (err != cudaSuccess) return err;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)((p.T + kTcM - 1) / kTcM), (unsigned)kRouteTcSplit);
  cfg.blockDim = dim3(kTcThreads);
  cfg.dynamicSmemBytes = (size_t)tc_stages(p.Ep) * tc_stage_bytes(p.Ep) + 1024;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, route_tc_kernel, tmA, tmB, p);
}

}  // namespace moe
