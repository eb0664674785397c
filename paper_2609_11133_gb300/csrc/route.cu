// Router GEMV + top-k, permutation / work plan, and the small elementwise
// kernels (activation conversion, combine) of the MoE decode layer.
#include "act_terms.cuh"
#include "ffn.cuh"
#include "route.cuh"

namespace moe {

// ------------------------------------------------------------------ helpers

// Scale one token row to f16 (power-of-two factor, exact for bf16 input) in
// the unit order the expert kernels read (act_pos), and store 1/factor.
template <int FMT>
__device__ void convert_row_x16(const __nv_bfloat16* row, int H, __half* dst, float* inv,
                                int lane, bool perm) {
  float amax = 0.f;
  for (int h = lane * 8; h < H; h += 256) {
    const uint4 v = *reinterpret_cast<const uint4*>(row + h);
    const __nv_bfloat162* b = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 f = __bfloat1622float2(b[i]);
      amax = fmaxf(amax, fmaxf(fabsf(f.x), fabsf(f.y)));
    }
  }
  amax = warp_max(amax);
  const float sc = pow2_scale_for(amax);
  constexpr int UPB = FmtTraits<FMT>::KEL / 8;  // 16-byte units per stage block
  for (int h = lane * 8; h < H; h += 256) {
    const uint4 v = *reinterpret_cast<const uint4*>(row + h);
    const __nv_bfloat162* b = reinterpret_cast<const __nv_bfloat162*>(&v);
    uint4 o;
    __half2* oh = reinterpret_cast<__half2*>(&o);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 f = __bfloat1622float2(b[i]);
      oh[i] = __floats2half2_rn(f.x * sc, f.y * sc);
    }
    const int U = h >> 3;
    const int phys = perm ? (U / UPB) * UPB + act_unit<FMT>(U % UPB) : U;
    *reinterpret_cast<uint4*>(dst + (size_t)phys * 8) = o;
  }
  if (lane == 0) *inv = 1.f / sc;
}

// perm: store the 16-byte units in the order of the warp-MMA NVFP4 engine
// (ffn.cuh); FP8 reads rows in natural order.
__device__ __forceinline__ void convert_row_dispatch(int fmt, const __nv_bfloat16* row, int H,
                                                     __half* dst, float* inv, int lane,
                                                     bool perm) {
  if (fmt == 2)
    convert_row_x16<2>(row, H, dst, inv, lane, perm);
  else
    convert_row_x16<1>(row, H, dst, inv, lane, perm);
}

// The NVFP4 terms of a chunk of token rows staged in shared memory (xs, nt
// rows of H bf16): every CTA of the chunk encodes an equal share of the
// 16-element blocks (`part` of `nparts`); every CTA derives the rows' scale.
__device__ void convert_chunk_terms(const __nv_bfloat16* xs, int nt, int H, int t0, int part,
                                    int nparts, uint8_t* xq, uint8_t* xsf, float* xinv) {
  __shared__ float s_sc[kRouteTok];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (warp < nt) {
    float amax = 0.f;
    for (int h = lane * 8; h < H; h += 256) {
      const uint4 v = *reinterpret_cast<const uint4*>(xs + (size_t)warp * H + h);
      const __nv_bfloat162* b = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float2 f = __bfloat1622float2(b[i]);
        amax = fmaxf(amax, fmaxf(fabsf(f.x), fabsf(f.y)));
      }
    }
    amax = warp_max(amax);
    const float sc = pow2_scale_terms(amax);
    if (lane == 0) {
      s_sc[warp] = sc;
      if (part == 0) xinv[t0 + warp] = 1.f / sc;
    }
  }
  __syncthreads();
  // a quad of lanes per 16-element block, four elements each; every warp runs
  // the same number of rounds (the quads' shuffles need all its lanes)
  const int nb = H / 16, total = nt * nb;
  const int nq = blockDim.x >> 2, lq = threadIdx.x & 3;
  for (int base = part * nq; base < total; base += nparts * nq) {
    const int idx = base + (threadIdx.x >> 2);
    const bool valid = idx < total;
    const int j = valid ? idx / nb : 0, b = valid ? idx - j * nb : 0;
    float r[4] = {0.f, 0.f, 0.f, 0.f};
    if (valid) {
      const uint2 v = *reinterpret_cast<const uint2*>(xs + (size_t)j * H + 16 * b + 4 * lq);
      const float2 a = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&v.x));
      const float2 c = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&v.y));
      r[0] = a.x * s_sc[j];
      r[1] = a.y * s_sc[j];
      r[2] = c.x * s_sc[j];
      r[3] = c.y * s_sc[j];
    }
    uint32_t pt[kTerms], sf[kTerms];
    encode_terms16_quad(r, pt, sf);
    store_terms16_quad(pt, sf, valid, xq, xsf, (size_t)(t0 + j) * kTerms, H, b);
  }
}

// The two E4M3 terms of a chunk of token rows staged in shared memory, every
// CTA of the chunk an equal share of the 8-element groups.
__device__ void convert_chunk_e4m3(const __nv_bfloat16* xs, int nt, int H, int t0, int part,
                                   int nparts, uint8_t* xq, float* xinv) {
  __shared__ float s_sc[kRouteTok];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (warp < nt) {
    float amax = 0.f;
    for (int h = lane * 8; h < H; h += 256) {
      const uint4 v = *reinterpret_cast<const uint4*>(xs + (size_t)warp * H + h);
      const __nv_bfloat162* b = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float2 f = __bfloat1622float2(b[i]);
        amax = fmaxf(amax, fmaxf(fabsf(f.x), fabsf(f.y)));
      }
    }
    amax = warp_max(amax);
    const float sc = pow2_scale_e4m3(amax);
    if (lane == 0) {
      s_sc[warp] = sc;
      if (part == 0) xinv[t0 + warp] = 1.f / sc;
    }
  }
  __syncthreads();
  const int n8 = H / 8;
  for (int idx = part * blockDim.x + threadIdx.x; idx < nt * n8; idx += nparts * blockDim.x) {
    const int j = idx / n8, c = idx - j * n8;
    const uint4 v = *reinterpret_cast<const uint4*>(xs + (size_t)j * H + 8 * c);
    const __nv_bfloat162* b = reinterpret_cast<const __nv_bfloat162*>(&v);
    float f[8];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 t = __bfloat1622float2(b[i]);
      f[2 * i] = t.x * s_sc[j];
      f[2 * i + 1] = t.y * s_sc[j];
    }
    uint2 hi, lo;
    encode_e4m3x2_8(f, hi, lo);
    store_e4m3x2_8(hi, lo, xq, (size_t)(t0 + j) * kF8Terms, H, c);
  }
}

// Order-preserving unsigned key of a finite float (larger value, larger key;
// -0 maps like +0), and its inverse.  Keys of finite values are never 0.
__device__ __forceinline__ unsigned logit_key(float v) {
  const unsigned b = __float_as_uint(v == 0.f ? 0.f : v);
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}
__device__ __forceinline__ float key_logit(unsigned k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7fffffffu) : ~k);
}

__device__ __forceinline__ unsigned lanemask_lt() {
  unsigned m;
  asm("mov.u32 %0, %%lanemask_lt;" : "=r"(m));
  return m;
}

// Token -> expert permutation (moe_permute), by one CTA of 256 threads.
// Assignments are ranked within eight contiguous segments (one warp each,
// match_any per 32), the per-segment counts are prefix-summed per expert, and
// every assignment is placed at offsets[e] + its stable rank.
// cw: shared scratch of 8*E + 2*(E+1) ints.
__device__ void permute_plan(const int* ids, int T, int k, int E, int* counts, int* offsets,
                             int* sorted, int* inv, int* active, int* cw) {
  const int A = T * k;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int seg = (A + 7) / 8;
  int* s_off = cw + 8 * E;
  int* s_bad = s_off + E + 1;
  for (int i = threadIdx.x; i < 8 * E; i += blockDim.x) cw[i] = 0;
  if (threadIdx.x == 0) *s_bad = 0;
  __syncthreads();
  {
    const int a_lo = warp * seg, a_hi = min(A, (warp + 1) * seg);
    for (int base = a_lo; base < a_hi; base += 32) {
      const int a = base + lane;
      int e = -1;
      if (a < a_hi) {
        e = __ldcg(ids + a);
        if (e < 0 || e >= E) {
          e = -1;
          *s_bad = 1;
        }
      }
      const int key = (e >= 0) ? e : -(lane + 2);
      const unsigned peers = __match_any_sync(0xffffffffu, key);
      int c = 0;
      if (e >= 0) c = cw[warp * E + e];
      __syncwarp();
      if (e >= 0 && lane == __ffs(peers) - 1) cw[warp * E + e] = c + __popc(peers);
      __syncwarp();
      if (e >= 0) inv[a] = c + __popc(peers & lanemask_lt());
    }
  }
  __syncthreads();
  for (int e = threadIdx.x; e < E; e += blockDim.x) {
    int run = 0;
    for (int w = 0; w < 8; ++w) {
      const int c = cw[w * E + e];
      cw[w * E + e] = run;
      run += c;
    }
    counts[e] = run;
    s_off[e] = run;  // counts for now
  }
  __syncthreads();
  if (warp == 0) {
    const int per = (E + 31) / 32;
    const int e0 = lane * per, e1 = min(E, e0 + per);
    int sc = 0, sa = 0;
    for (int e = e0; e < e1; ++e) {
      const int c = s_off[e];
      sc += c;
      sa += (c > 0);
    }
    int xc = sc, xa = sa;  // inclusive scans
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int yc = __shfl_up_sync(0xffffffffu, xc, o);
      const int ya = __shfl_up_sync(0xffffffffu, xa, o);
      if (lane >= o) {
        xc += yc;
        xa += ya;
      }
    }
    int rc = xc - sc, ra = xa - sa;  // exclusive
    for (int e = e0; e < e1; ++e) {
      const int c = s_off[e];
      s_off[e] = rc;
      offsets[e] = rc;
      if (c > 0) active[1 + ra++] = e;
      rc += c;
    }
    if (lane == 31) {
      offsets[E] = xc;
      s_off[E] = xc;
      active[0] = *s_bad ? -1 : xa;
    }
  }
  __syncthreads();
  for (int a = threadIdx.x; a < A; a += blockDim.x) {
    const int e = __ldcg(ids + a);
    if (e < 0 || e >= E) continue;
    const int w = a / seg;
    const int pos = s_off[e] + cw[w * E + e] + inv[a];
    sorted[pos] = a;
    inv[a] = pos;
  }
}

// Top-k of token t's logits by one warp, lane l holding logits l, l+32, ...
// (PER of them, E <= 32 * PER): the ids and gates, and - in the fused layer -
// the token's entries in the per-expert assignment lists.
template <int PER>
__device__ __forceinline__ void chunk_topk(const RouteParams& p, int t, int warp, int lane,
                                           int (*s_sel)[kMaxK], float (*s_selv)[kMaxK]) {
  const int E = p.E;
  float v[PER];
#pragma unroll
  for (int i = 0; i < PER; ++i) {
    const int ee = lane + 32 * i;
    v[i] = (ee < E) ? __ldcg(p.logits + (size_t)t * E + ee) : -INFINITY;
  }
  // Each lane keeps the best of its own untaken logits; a round takes the
  // warp's best by two warp reductions - the largest order-preserving key,
  // then the lowest expert index holding it (ties go to the lower index;
  // -0 and +0 share a key) - and only the winning lane rescans.
  unsigned key[PER];
#pragma unroll
  for (int i = 0; i < PER; ++i) key[i] = logit_key(v[i]);
  unsigned taken = 0u;
  unsigned lbk;  // best untaken key of this lane (0: none left)
  unsigned lbi;
  auto local_best = [&]() {
    lbk = 0u;
    lbi = 0xffffffffu;
#pragma unroll
    for (int i = 0; i < PER; ++i) {
      const int ee = lane + 32 * i;
      if (ee < E && !((taken >> i) & 1u) && key[i] > lbk) {
        lbk = key[i];  // a later (higher) index never wins a tie within a lane
        lbi = (unsigned)ee;
      }
    }
  };
  local_best();
  for (int j = 0; j < p.k; ++j) {
    const unsigned m = __reduce_max_sync(0xffffffffu, lbk);
    const unsigned bi = __reduce_min_sync(0xffffffffu, lbk == m ? lbi : 0xffffffffu);
    if ((int)(bi & 31u) == lane) {
      taken |= 1u << (bi >> 5);
      local_best();
    }
    if (lane == 0) {
      s_sel[warp][j] = (int)bi;
      s_selv[warp][j] = key_logit(m);
    }
  }
  __syncwarp();
  const float lmax = s_selv[warp][0];
  float den = 0.f;
  if (p.renorm) {
    for (int j = 0; j < p.k; ++j) den += expf(s_selv[warp][j] - lmax);
  } else {
    float part = 0.f;
#pragma unroll
    for (int i = 0; i < PER; ++i)
      if (lane + 32 * i < E) part += expf(v[i] - lmax);
    den = warp_sum(part);
  }
  for (int j = lane; j < p.k; j += 32) {
    const int id = s_sel[warp][j];
    const float gw = expf(s_selv[warp][j] - lmax) / den;
    p.ids[(size_t)t * p.k + j] = id;
    p.gates[(size_t)t * p.k + j] = gw;
    if (p.ids2) p.ids2[(size_t)t * p.k + j] = id;
    if (p.gates2) p.gates2[(size_t)t * p.k + j] = gw;
    if (p.fused) {
      // append to expert id's list (order within a list is arbitrary)
      const unsigned pos = atomicAdd(p.acnt + id, 1u);
      p.alist[(size_t)id * p.T + pos] = t * p.k + j;
    }
  }
}

// ------------------------------------------------------------------ route kernel
__global__ void __launch_bounds__(256) route_kernel(const RouteParams p) {
  extern __shared__ __align__(16) unsigned char route_smem[];
  __nv_bfloat16* xs = reinterpret_cast<__nv_bfloat16*>(route_smem);
  __shared__ int s_flag;
  __shared__ int s_sel[kRouteWarps][kMaxK];  // top-k of the chunk's tokens, by warp
  __shared__ float s_selv[kRouteWarps][kMaxK];

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int chunk = blockIdx.y, eb = blockIdx.x;
  if (p.plog) pdl_wait();  // the GEMM's partial logits (and xn) are complete
  pdl_launch_dependents();  // the expert kernel may start its prologue now
  const int t0 = chunk * kRouteTok;
  const int nt = min(kRouteTok, p.T - t0);
  const int H = p.H, E = p.E;

  // stage this chunk's token rows: every thread issues all of its 16-byte
  // loads before storing any of them (one memory latency, not one per load)
  if (!p.terms_done) {
    const uint4* src = reinterpret_cast<const uint4*>(p.x + (size_t)t0 * H);
    uint4* dst = reinterpret_cast<uint4*>(xs);
    const int n16 = nt * H / 8;
    constexpr int BATCH = 16;
    for (int base = 0; base < n16; base += BATCH * 256) {
      uint4 v[BATCH];
#pragma unroll
      for (int q = 0; q < BATCH; ++q) {
        const int i = base + q * 256 + threadIdx.x;
        if (i < n16) v[q] = __ldg(src + i);
      }
#pragma unroll
      for (int q = 0; q < BATCH; ++q) {
        const int i = base + q * 256 + threadIdx.x;
        if (i < n16) dst[i] = v[q];
      }
    }
  }
  __syncthreads();
  if (p.prenorm && warp < nt) {
    __nv_bfloat16* row = xs + (size_t)warp * H;
    rms_norm_row_bf16(row, row, H, lane);
  }
  __syncthreads();
  if (p.fused && !p.terms_done) {
    if (p.act == kActTerms) {
      convert_chunk_terms(xs, nt, H, t0, eb, gridDim.x, p.xq, p.xsf, p.xinv);
    } else if (p.act == kActE4M3) {
      convert_chunk_e4m3(xs, nt, H, t0, eb, gridDim.x, p.xq, p.xinv);
    } else if (eb == 0 && warp < nt) {
      const int t = t0 + warp;
      convert_row_dispatch(p.fmt, xs + (size_t)warp * H, H, p.x16 + (size_t)t * H, p.xinv + t,
                           lane, p.act == kActF16Perm);
    }
  }

  // router GEMV, in rounds of up to four of the CTA's experts: warp w covers
  // one eighth of H for the round's experts (each staged x value is read once
  // per warp and round), lanes -> 4 consecutive h per 128.  The 4 x 8 partial
  // sums of a lane meet across the warp in a butterfly (lane l ends with sum
  // l = expert slot l/8, token l%8), then across the warps in shared memory
  // in warp order.
  __shared__ float s_part[kRouteWarps][32];
  const int nexp = min(p.epb, E - eb * p.epb);  // experts of this CTA
  if (p.plog) {
    // the tensor-core router's partial logits of this chunk and these
    // experts, added in slice order
    const size_t slice = (size_t)p.T * p.ep;
    for (int i = threadIdx.x; i < nt * nexp; i += blockDim.x) {
      const int t = i / nexp, e = eb * p.epb + (i - t * nexp);
      const float* q = p.plog + (size_t)(t0 + t) * p.ep + e;
      float sum = __ldcg(q);
      for (int j = 1; j < p.nsplit; ++j) sum += __ldcg(q + j * slice);
      const float b = p.bias ? __ldg(p.bias + e) : 0.f;
      p.logits[(size_t)(t0 + t) * E + e] = sum + b;
    }
  }
  for (int q0 = 0; q0 < (p.plog ? 0 : nexp); q0 += 4) {
    constexpr int MAXEPB = 4;
    const int e0 = eb * p.epb + q0;
    const int nq = min(MAXEPB, nexp - q0);  // experts of this round
    {
      const int hpart = H / kRouteWarps;
      const int hbeg = warp * hpart;
      float acc[MAXEPB][kRouteTok];
#pragma unroll
      for (int x = 0; x < MAXEPB; ++x)
#pragma unroll
        for (int t = 0; t < kRouteTok; ++t) acc[x][t] = 0.f;
      constexpr int DEPTH = 4;  // 128-element steps whose router loads are in flight together
      for (int h0 = hbeg + lane * 4; h0 < hbeg + hpart; h0 += 128 * DEPTH) {
        float4 w[DEPTH][MAXEPB];
#pragma unroll
        for (int q = 0; q < DEPTH; ++q)
#pragma unroll
          for (int x = 0; x < MAXEPB; ++x)
            w[q][x] = (x < nq && h0 + 128 * q < hbeg + hpart)
                          ? __ldg(reinterpret_cast<const float4*>(p.wr + (size_t)(e0 + x) * H +
                                                                  h0 + 128 * q))
                          : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int q = 0; q < DEPTH; ++q) {
          const int h = h0 + 128 * q;
          if (h >= hbeg + hpart) break;
#pragma unroll
          for (int t = 0; t < kRouteTok; ++t) {
            if (t < nt) {
              const uint2 xv = *reinterpret_cast<const uint2*>(xs + (size_t)t * H + h);
              const float2 a =
                  __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&xv.x));
              const float2 b =
                  __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&xv.y));
#pragma unroll
              for (int x = 0; x < MAXEPB; ++x) {
                float sacc = acc[x][t];
                sacc = fmaf(a.x, w[q][x].x, sacc);
                sacc = fmaf(a.y, w[q][x].y, sacc);
                sacc = fmaf(b.x, w[q][x].z, sacc);
                sacc = fmaf(b.y, w[q][x].w, sacc);
                acc[x][t] = sacc;
              }
            }
          }
        }
      }
      float v[32];
#pragma unroll
      for (int i = 0; i < 32; ++i) v[i] = acc[i / kRouteTok][i % kRouteTok];
#pragma unroll
      for (int sft = 16; sft >= 1; sft >>= 1) {
        const bool upper = (lane & sft) != 0;
#pragma unroll
        for (int i = 0; i < sft; ++i) {
          const float send = upper ? v[i] : v[i + sft];
          const float keep = upper ? v[i + sft] : v[i];
          v[i] = keep + __shfl_xor_sync(0xffffffffu, send, sft);
        }
      }
      s_part[warp][lane] = v[0];
    }
    __syncthreads();
    if (threadIdx.x < 32) {
      const int x = threadIdx.x / kRouteTok, t = threadIdx.x % kRouteTok;
      const int e = e0 + x;
      if (x < nq && t < nt) {
        float sum = s_part[0][threadIdx.x];
#pragma unroll
        for (int w = 1; w < kRouteWarps; ++w) sum += s_part[w][threadIdx.x];
        const float b = p.bias ? __ldg(p.bias + e) : 0.f;
        p.logits[(size_t)(t0 + t) * E + e] = sum + b;
      }
    }
    __syncthreads();  // s_part is reused by the next round
  }

  // accumulators and counters of the later kernels start from zero
  if (p.fused) {
    const size_t nthr = (size_t)gridDim.x * gridDim.y * blockDim.x;
    const size_t tid = ((size_t)blockIdx.y * gridDim.x + blockIdx.x) * blockDim.x + threadIdx.x;
    const float4 z = make_float4(0.f, 0.f, 0.f, 0.f);
    for (size_t i = tid; i < p.zero_a_n4; i += nthr) p.zero_a[i] = z;
    for (size_t i = tid; i < p.zero_b_n4; i += nthr) p.zero_b[i] = z;
  }

  // chunk ticket: the last of this chunk's expert blocks does the top-k.  The
  // barrier orders every thread's writes before thread 0's fence and ticket
  // (release); the winner's fence after the ticket and the second barrier
  // order its reads of the other blocks' logits after it (acquire).
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    const unsigned old = atomicAdd(p.chunk_cnt + chunk, 1u);
    s_flag = (old == gridDim.x - 1);
    if (s_flag) {
      p.chunk_cnt[chunk] = 0u;
      __threadfence();
    }
  }
  __syncthreads();
  if (!s_flag) return;

  if (warp < nt) {
    const int per = (E + 31) / 32;  // logits held by each lane
    if (per <= 4)
      chunk_topk<4>(p, t0 + warp, warp, lane, s_sel, s_selv);
    else if (per <= 8)
      chunk_topk<8>(p, t0 + warp, warp, lane, s_sel, s_selv);
    else
      chunk_topk<kMaxE / 32>(p, t0 + warp, warp, lane, s_sel, s_selv);
  }
}

__global__ void __launch_bounds__(256) permute_kernel(const int* ids, int T, int k, int E,
                                                      int* counts, int* offsets, int* sorted,
                                                      int* inv, int* active) {
  extern __shared__ __align__(16) unsigned char route_smem[];
  permute_plan(ids, T, k, E, counts, offsets, sorted, inv, active,
               reinterpret_cast<int*>(route_smem));
}

// Activation conversion, zeroing and per-expert counts for the unfused
// expert FFN (the expert kernels build their plan from the counts).
__global__ void __launch_bounds__(256) prep_kernel(const PrepParams p) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  pdl_launch_dependents();
  {
    const size_t nthr = (size_t)gridDim.x * blockDim.x;
    const size_t tid = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
    const float4 z = make_float4(0.f, 0.f, 0.f, 0.f);
    for (size_t i = tid; i < p.zero_a_n4; i += nthr) p.zero_a[i] = z;
    for (size_t i = tid; i < p.zero_b_n4; i += nthr) p.zero_b[i] = z;
  }
  const int t = blockIdx.x * 8 + warp;
  if (t < p.T) {
    if (p.act == kActTerms)
      convert_row_terms(p.x + (size_t)t * p.H, p.H, t, p.xq, p.xsf, p.xinv + t, lane);
    else if (p.act == kActE4M3)
      convert_row_e4m3(p.x + (size_t)t * p.H, p.H, t, p.xq, p.xinv + t, lane);
    else
      convert_row_dispatch(p.fmt, p.x + (size_t)t * p.H, p.H, p.x16 + (size_t)t * p.H,
                           p.xinv + t, lane, p.act == kActF16Perm);
  }
  if (blockIdx.x == 0)
    for (int e = threadIdx.x; e < p.E; e += blockDim.x)
      p.counts[e] = __ldg(p.offsets + e + 1) - __ldg(p.offsets + e);
}

// grid ceil(T*k / 8): CTA b copies compact rows 8b..8b+7.  Compact row r is
// position r - pre[e] of expert e's list, pre the exclusive prefix of the
// per-expert counts (every CTA scans the counts; E <= 512).  A row's term rows
// (and their scales) are one contiguous block in both arrays, so one thread
// moves them with bulk copies: every block into shared memory under one
// mbarrier, then every block out.
constexpr int kGatherRows = 8;

__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void* src, uint32_t bytes,
                                         uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::
          "r"(dst),
      "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void bulk_s2g(void* dst, uint32_t src, uint32_t bytes) {
  asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(
                   reinterpret_cast<uint64_t>(dst)),
               "r"(src), "r"(bytes)
               : "memory");
}

__global__ void __launch_bounds__(128) gather_kernel(const GatherParams p) {
  extern __shared__ __align__(128) unsigned char g_rows[];
  __shared__ int s_pre[kMaxE + 1];
  __shared__ int s_tok[kGatherRows], s_row[kGatherRows];
  __shared__ __align__(8) uint64_t s_bar;
  pdl_wait();  // the routing that wrote the lists is complete
  pdl_launch_dependents();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 32) {
    mbar_init(&s_bar, 1);
    fence_mbar_init();
  }
  if (warp == 0) {
    constexpr int PER = kMaxE / 32;  // counts per lane
    int c[PER], run = 0;
#pragma unroll
    for (int i = 0; i < PER; ++i) {
      const int e = lane * PER + i;
      c[i] = e < p.E ? (int)__ldcg(p.acnt + e) : 0;
      run += c[i];
    }
    int inc = run;  // inclusive scan of the lanes' sums
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, inc, o);
      if (lane >= o) inc += y;
    }
    int pre = inc - run;
#pragma unroll
    for (int i = 0; i < PER; ++i) {
      s_pre[lane * PER + i] = pre;
      pre += c[i];
    }
    if (lane == 31) s_pre[kMaxE] = pre;
  }
  __syncthreads();
  const int total = s_pre[kMaxE];
  const int r0 = blockIdx.x * kGatherRows;
  const int nj = min(kGatherRows, total - r0);
  if (nj <= 0) return;
  if (threadIdx.x < nj) {
    const int r = r0 + threadIdx.x;
    int lo = 0, hi = p.E - 1;  // the last expert whose list starts at or before r
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (s_pre[mid] <= r) lo = mid; else hi = mid - 1;
    }
    const int a = __ldcg(p.alist + (size_t)lo * p.T + (r - s_pre[lo]));
    s_tok[threadIdx.x] = a / p.k;
    s_row[threadIdx.x] = r;
    // its compact row (prefill engine: the combine kernel reads each
    // assignment's down row there)
    if (p.inv) p.inv[a] = r;
  }
  __syncthreads();
  if (threadIdx.x != 0) return;
  const uint32_t rb = (uint32_t)(p.terms * p.qrow);              // term rows of a token
  const uint32_t sb = p.sf ? (uint32_t)(p.terms * p.sfrow) : 0u;  // their scales
  const uint32_t base = smem_u32(g_rows);
  mbar_arrive_expect_tx(&s_bar, (uint32_t)nj * (rb + sb));
  for (int j = 0; j < nj; ++j) {
    bulk_g2s(base + j * rb, p.q + (size_t)s_tok[j] * rb, rb, &s_bar);
    if (sb) bulk_g2s(base + kGatherRows * rb + j * sb, p.sf + (size_t)s_tok[j] * sb, sb, &s_bar);
  }
  if (!mbar_wait_bounded(&s_bar, 0, p.wait_ns, nullptr)) {
    set_status(p.status, kStatusTimeoutRoute);
    return;  // copies that never landed leave nothing to store
  }
  for (int j = 0; j < nj; ++j) {
    bulk_s2g(p.gq + (size_t)s_row[j] * rb, base + j * rb, rb);
    if (sb) bulk_s2g(p.gsf + (size_t)s_row[j] * sb, base + kGatherRows * rb + j * sb, sb);
  }
  asm volatile("cp.async.bulk.commit_group;" ::: "memory");
  // the shared memory is read out before the CTA exits
  asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}

__global__ void __launch_bounds__(256) combine_kernel(const CombineParams p) {
  pdl_wait();
  // the per-expert assignment counters start the next layer call from zero
  if (p.acnt_reset && blockIdx.x == 0)
    for (int e = threadIdx.x; e < p.E; e += blockDim.x) p.acnt_reset[e] = 0u;
  const size_t n4 = (size_t)p.T * p.H / 4;
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < n4;
       i += (size_t)gridDim.x * blockDim.x) {
    const size_t t = i * 4 / p.H;
    const int h = (int)(i * 4 - t * p.H);
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int j = 0; j < p.k; ++j) {
      const size_t a = t * p.k + j;
      const float w = __ldcg(p.topk_w + a);
      const int row = p.inv ? __ldcg(p.inv + a) : (int)a;  // no inv: rows by assignment
      const float4 y = __ldcg(reinterpret_cast<const float4*>(p.y_perm + (size_t)row * p.H + h));
      acc.x = fmaf(w, y.x, acc.x);
      acc.y = fmaf(w, y.y, acc.y);
      acc.z = fmaf(w, y.z, acc.z);
      acc.w = fmaf(w, y.w, acc.w);
    }
    if (p.residual) {
      const uint2 r = *reinterpret_cast<const uint2*>(p.residual + t * p.H + h);
      const float2 a = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&r.x));
      const float2 b = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&r.y));
      acc.x += a.x;
      acc.y += a.y;
      acc.z += b.x;
      acc.w += b.y;
    }
    __nv_bfloat162 o0 = __floats2bfloat162_rn(acc.x, acc.y);
    __nv_bfloat162 o1 = __floats2bfloat162_rn(acc.z, acc.w);
    uint2 o;
    o.x = *reinterpret_cast<uint32_t*>(&o0);
    o.y = *reinterpret_cast<uint32_t*>(&o1);
    *reinterpret_cast<uint2*>(p.out + t * p.H + h) = o;
  }
}

// ------------------------------------------------------------------ launchers
size_t route_smem_bytes(int H, int E) {
  (void)E;
  return (size_t)kRouteTok * H * 2;  // the chunk's token rows
}

cudaError_t launch_route(const RouteParams& p, cudaStream_t st) {
  // the largest dynamic size any call can ask for (H <= 8192, E <= 512)
  static std::atomic<unsigned long long> done{0};
  const size_t smem = route_smem_bytes(p.H, p.E);
  cudaError_t err = set_smem_once(route_kernel, (int)route_smem_bytes(8192, kMaxE), done);
  if (err != cudaSuccess) return err;
  if (p.plog) {
    // after the tensor-core router's GEMM, launched as a programmatic
    // dependent (it waits for the GEMM before it reads)
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)((p.E + p.epb - 1) / p.epb),
                       (unsigned)((p.T + kRouteTok - 1) / kRouteTok));
    cfg.blockDim = dim3(256);
    cfg.dynamicSmemBytes = p.terms_done ? 0 : smem;  // no rows staged
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, route_kernel, p);
  }
  dim3 grid((p.E + p.epb - 1) / p.epb, (p.T + kRouteTok - 1) / kRouteTok);
  route_kernel<<<grid, 256, smem, st>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_gather(const GatherParams& p, cudaStream_t st) {
  // shared memory for the rows of the largest shape (H = 8192)
  static std::atomic<unsigned long long> done{0};
  const int smax = kGatherRows * (4 * 4096 + 4 * 512);
  cudaError_t err = set_smem_once(gather_kernel, smax, done);
  if (err != cudaSuccess) return err;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(((size_t)p.T * p.k + kGatherRows - 1) / kGatherRows));
  cfg.blockDim = dim3(128);
  cfg.dynamicSmemBytes =
      (size_t)kGatherRows * (p.terms * p.qrow + (p.sf ? p.terms * p.sfrow : 0));
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, gather_kernel, p);
}

cudaError_t launch_permute_standalone(const int* ids, int T, int k, int E, int* counts,
                                      int* offsets, int* sorted, int* inv, int* active,
                                      cudaStream_t st) {
  static std::atomic<unsigned long long> done{0};
  const size_t smem = sizeof(int) * (size_t)(8 * E + 3 * (E + 1));
  cudaError_t err =
      set_smem_once(permute_kernel, (int)(sizeof(int) * (size_t)(8 * kMaxE + 3 * (kMaxE + 1))), done);
  if (err != cudaSuccess) return err;
  permute_kernel<<<1, 256, smem, st>>>(ids, T, k, E, counts, offsets, sorted, inv, active);
  return cudaGetLastError();
}

cudaError_t launch_prep(const PrepParams& p, cudaStream_t st) {
  const int grid = (p.T + 7) / 8 > 0 ? (p.T + 7) / 8 : 1;
  prep_kernel<<<grid < 64 ? 64 : grid, 256, 0, st>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_combine(const CombineParams& p, cudaStream_t st) {
  const size_t n4 = (size_t)p.T * p.H / 4;
  size_t blocks = (n4 + 255) / 256;
  if (blocks > 4096) blocks = 4096;
  if (blocks == 0) blocks = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)blocks);
  cfg.blockDim = dim3(256);
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, combine_kernel, p);
}

}  // namespace moe
