// Activations as sums of low-precision terms, the B operand of the
// tensor-core engines: four NVFP4 terms per row for the block-scaled engine
// (ffn_bs.cuh, below), two E4M3 terms per row for the FP8 engine (ffn_f8.cuh,
// at the end of this file).
//
// The tcgen05 kind::mxf4nvf4 MMA multiplies E2M1 codes with one UE4M3 scale
// per 16 K elements on BOTH operands.  The weights are stored that way; the
// activations (bf16 x, fp32 h) are not, and one E2M1 code keeps only two
// significant bits.  So every activation row v is written as
//
//     v * 2^p = sum_{t<4} s_t[b] * q_t[i],   i in block b of 16 elements,
//
// with 2^p a per-row power of two, s_t[b] UE4M3 and q_t[i] E2M1: term 0 codes
// v, term t codes what terms 0..t-1 left over.  Each scale is the smallest
// UE4M3 value >= max|residual| / 6, so |q| <= 6 never saturates, and the
// largest residual of a block shrinks by about 6x per term: after four terms
// it is below 2^-9.5 of the block maximum (finer than the bf16 input itself),
// and the layer output stays within ~1e-4 of the exact result.  Each term is
// one "token row" of the MMA's B operand, so a token costs 4 rows of N; the
// four partial products are summed in the epilogue.  The residual update
// r -= s*q is exact in fp32 (s*q has at most 6 significant bits).
#pragma once

#include "common.cuh"

namespace moe {

constexpr int kTerms = 4;

// Power-of-two factor that maps max|v| into [2^10, 2^11): the first term's
// scales stay below 2^11/6 < 448 (the UE4M3 maximum) and the fourth term's
// above the UE4M3 subnormal range for every block within 2^-8 of the row max.
__device__ __forceinline__ float pow2_scale_terms(float amax) {
  if (!(amax > 0.f) || !isfinite(amax)) return 1.f;
  int e;
  frexpf(amax, &e);  // amax = m * 2^e, 0.5 <= m < 1
  return ldexpf(1.f, min(11 - e, 126));
}

// Smallest UE4M3 value >= v (v >= 0), as its code byte; *val gets the value.
__device__ __forceinline__ uint32_t ue4m3_ceil(float v, float* val) {
  uint16_t two;  // both bytes hold e4m3(v), whichever source lands in which byte
  asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %1;" : "=h"(two) : "f"(v));
  uint32_t code = two & 0xffu;
  float f = __half2float(__ushort_as_half((uint16_t)(e4m3x2_to_f16x2(code) & 0xffffu)));
  if (f < v && code < 0x7eu) {
    ++code;  // the next larger magnitude
    f = __half2float(__ushort_as_half((uint16_t)(e4m3x2_to_f16x2(code) & 0xffffu)));
  }
  *val = f;
  return code;
}

// Eight floats to eight E2M1 codes, round to nearest even, saturating at 6;
// element 2i in the low nibble of byte i (the weights' packing).
__device__ __forceinline__ uint32_t e2m1x8_from_f32(const float* q) {
  uint32_t w;
  asm("{\n .reg .b8 b0, b1, b2, b3;\n"
      " cvt.rn.satfinite.e2m1x2.f32 b0, %2, %1;\n"
      " cvt.rn.satfinite.e2m1x2.f32 b1, %4, %3;\n"
      " cvt.rn.satfinite.e2m1x2.f32 b2, %6, %5;\n"
      " cvt.rn.satfinite.e2m1x2.f32 b3, %8, %7;\n"
      " mov.b32 %0, {b0, b1, b2, b3};\n}\n"
      : "=r"(w)
      : "f"(q[0]), "f"(q[1]), "f"(q[2]), "f"(q[3]), "f"(q[4]), "f"(q[5]), "f"(q[6]), "f"(q[7]));
  return w;
}

// Encode one 16-element block r (already scaled by the row's power of two)
// into its first NTERM terms (of kTerms): codes[t] (16 E2M1 codes, 8 bytes)
// and sf[t] (UE4M3).  r is consumed (it ends as the residual).
template <int NTERM = kTerms>
__device__ __forceinline__ void encode_terms16(float (&r)[16], uint2 (&codes)[kTerms],
                                               uint32_t (&sf)[kTerms]) {
#pragma unroll
  for (int t = 0; t < NTERM; ++t) {
    float m = 0.f;
#pragma unroll
    for (int i = 0; i < 16; ++i) m = fmaxf(m, fabsf(r[i]));
    float s = 0.f;
    const uint32_t c = ue4m3_ceil(m * (1.f / 6.f), &s);
    sf[t] = (m > 0.f) ? c : 0u;
    if (!(m > 0.f)) {
      codes[t] = make_uint2(0u, 0u);
      continue;
    }
    const float inv = 1.f / s;
    float q[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) q[i] = r[i] * inv;
    const uint32_t w0 = e2m1x8_from_f32(q), w1 = e2m1x8_from_f32(q + 8);
    codes[t] = make_uint2(w0, w1);
    // subtract the coded values (exact)
    uint32_t d0[4], d1[4];
    e2m1x8_to_f16x8(w0, d0);
    e2m1x8_to_f16x8(w1, d1);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const uint32_t di = (i < 4) ? d0[i] : d1[i - 4];
      const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&di));
      r[2 * i] = fmaf(-f.x, s, r[2 * i]);
      r[2 * i + 1] = fmaf(-f.y, s, r[2 * i + 1]);
    }
  }
}

// encode_terms16 spread over the four lanes of a quad (lanes 4j..4j+3 of a
// warp): lane q of the quad holds elements 4q..4q+3 of the block (already
// scaled by the row's power of two) in r.  Every step is the serial one's,
// element by element, so the codes are the same; the block maximum takes two
// shuffles.  All 32 lanes of the warp call it together (lanes whose quad has
// no block pass zeros).  part[t] gets this lane's 16 bits of term t's codes
// (elements 4q..4q+3, element 4q in the low nibble), sf[t] the term's scale.
__device__ __forceinline__ void encode_terms16_quad(float (&r)[4], uint32_t (&part)[kTerms],
                                                    uint32_t (&sf)[kTerms]) {
#pragma unroll
  for (int t = 0; t < kTerms; ++t) {
    float m = fmaxf(fmaxf(fabsf(r[0]), fabsf(r[1])), fmaxf(fabsf(r[2]), fabsf(r[3])));
    m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, 1));
    m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, 2));
    float s = 0.f;
    const uint32_t c = ue4m3_ceil(m * (1.f / 6.f), &s);
    sf[t] = (m > 0.f) ? c : 0u;
    part[t] = 0u;
    if (m > 0.f) {
      const float inv = 1.f / s;
      uint32_t w;
      asm("{\n .reg .b8 b0, b1;\n"
          " cvt.rn.satfinite.e2m1x2.f32 b0, %2, %1;\n"
          " cvt.rn.satfinite.e2m1x2.f32 b1, %4, %3;\n"
          " mov.b32 %0, {b0, b1, b0, b1};\n}\n"
          : "=r"(w)
          : "f"(r[0] * inv), "f"(r[1] * inv), "f"(r[2] * inv), "f"(r[3] * inv));
      part[t] = w & 0xffffu;
      uint32_t d[4];
      e2m1x8_to_f16x8(part[t], d);  // d[0], d[1]: elements 0-1, 2-3
#pragma unroll
      for (int i = 0; i < 2; ++i) {
        const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&d[i]));
        r[2 * i] = fmaf(-f.x, s, r[2 * i]);  // exact
        r[2 * i + 1] = fmaf(-f.y, s, r[2 * i + 1]);
      }
    }
  }
}

// Store the quad's block b: lanes q = 0 and 2 write the two 32-bit halves of
// each term's codes, lane 0 the scale bytes.  All lanes of the warp call it;
// `valid` is false on lanes whose quad has no block.
__device__ __forceinline__ void store_terms16_quad(const uint32_t (&part)[kTerms],
                                                   const uint32_t (&sf)[kTerms], bool valid,
                                                   uint8_t* q, uint8_t* sfp, size_t row4, int K,
                                                   int b) {
  const int lq = threadIdx.x & 3;
#pragma unroll
  for (int t = 0; t < kTerms; ++t) {
    uint32_t w = part[t] << (16 * (lq & 1));
    w |= __shfl_xor_sync(0xffffffffu, w, 1);  // lanes 0,1: elements 0-7; 2,3: 8-15
    if (valid && (lq & 1) == 0)
      *reinterpret_cast<uint32_t*>(q + (row4 + t) * (size_t)(K / 2) + 8 * b + 2 * lq) = w;
    if (valid && lq == 0) sfp[(row4 + t) * (size_t)(K / 16) + b] = (uint8_t)sf[t];
  }
}

// Write block b of a row's terms: row r of the term arrays is token/assignment
// `row4 / kTerms`, term `row4 % kTerms`; q rows are K/2 bytes, sf rows K/16.
template <int NTERM = kTerms>
__device__ __forceinline__ void store_terms16(const uint2 (&codes)[kTerms],
                                              const uint32_t (&sf)[kTerms], uint8_t* q,
                                              uint8_t* sfp, size_t row4, int K, int b) {
#pragma unroll
  for (int t = 0; t < NTERM; ++t) {
    *reinterpret_cast<uint2*>(q + (row4 + t) * (size_t)(K / 2) + 8 * b) = codes[t];
    sfp[(row4 + t) * (size_t)(K / 16) + b] = (uint8_t)sf[t];
  }
}

// Sixteen consecutive bf16 values (32 bytes, 16-byte aligned) times `sc`.
__device__ __forceinline__ void load_bf16x16_scaled(const __nv_bfloat16* src, float sc,
                                                    float (&r)[16]) {
  const uint4 a = *reinterpret_cast<const uint4*>(src);
  const uint4 b = *reinterpret_cast<const uint4*>(src + 8);
  const uint32_t w[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w[i]));
    r[2 * i] = f.x * sc;
    r[2 * i + 1] = f.y * sc;
  }
}


// ------------------------------------------------------------------ E4M3 terms
// The FP8 tensor-core engine (ffn_f8.cuh) multiplies E4M3 weights with E4M3
// activations (kind::f8f6f4, no block scale).  An activation row v is written
// as v * 2^p = hi + lo with hi = e4m3(v * 2^p) and lo = e4m3(v * 2^p - hi):
// hi keeps four significant bits, lo the next four, so a bf16 input (eight
// bits) is kept whole unless it is more than ~2^14 below the row maximum.
// Two B rows per token; the epilogue adds the two columns.
constexpr int kF8Terms = 2;

// Power-of-two factor that maps max|v| into [2^7, 2^8) (E4M3 max 448).
__device__ __forceinline__ float pow2_scale_e4m3(float amax) {
  if (!(amax > 0.f) || !isfinite(amax)) return 1.f;
  int e;
  frexpf(amax, &e);
  return ldexpf(1.f, min(8 - e, 126));
}

// Two floats to two E4M3 codes (round to nearest even, saturating), the
// first in the low byte.
__device__ __forceinline__ uint32_t e4m3x2_from_f32(float v0, float v1) {
  uint16_t two;
  asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(two) : "f"(v1), "f"(v0));
  return two;
}

// Eight values (already scaled) to their hi and lo E4M3 codes (8 bytes each).
__device__ __forceinline__ void encode_e4m3x2_8(const float (&v)[8], uint2& hi, uint2& lo) {
  uint32_t h[4], l[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    h[i] = e4m3x2_from_f32(v[2 * i], v[2 * i + 1]);
    const uint32_t hd = e4m3x2_to_f16x2(h[i]);  // exact
    const float2 d = __half22float2(*reinterpret_cast<const __half2*>(&hd));
    l[i] = e4m3x2_from_f32(v[2 * i] - d.x, v[2 * i + 1] - d.y);
  }
  hi = make_uint2(h[0] | (h[1] << 16), h[2] | (h[3] << 16));
  lo = make_uint2(l[0] | (l[1] << 16), l[2] | (l[3] << 16));
}

// Store the two terms of 8 values at column c8*8 of row `row2` (= 2 * row):
// rows are K bytes.
__device__ __forceinline__ void store_e4m3x2_8(const uint2& hi, const uint2& lo, uint8_t* q,
                                               size_t row2, int K, int c8) {
  *reinterpret_cast<uint2*>(q + row2 * (size_t)K + 8 * c8) = hi;
  *reinterpret_cast<uint2*>(q + (row2 + 1) * (size_t)K + 8 * c8) = lo;
}

// The two E4M3 terms of one token row in global memory, by one warp.
__device__ __forceinline__ void convert_row_e4m3(const __nv_bfloat16* row, int H, int t,
                                                 uint8_t* xq, float* inv, int lane) {
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
  const float sc = pow2_scale_e4m3(amax);
  for (int c = lane; c < H / 8; c += 32) {
    const uint4 v = *reinterpret_cast<const uint4*>(row + 8 * c);
    const __nv_bfloat162* b = reinterpret_cast<const __nv_bfloat162*>(&v);
    float f[8];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 tt = __bfloat1622float2(b[i]);
      f[2 * i] = tt.x * sc;
      f[2 * i + 1] = tt.y * sc;
    }
    uint2 hi, lo;
    encode_e4m3x2_8(f, hi, lo);
    store_e4m3x2_8(hi, lo, xq, (size_t)t * kF8Terms, H, c);
  }
  if (lane == 0) *inv = 1.f / sc;
}

// The NVFP4 terms of one token row in global memory, by one warp.
__device__ __forceinline__ void convert_row_terms(const __nv_bfloat16* row, int H, int t,
                                                  uint8_t* xq, uint8_t* xsf, float* inv,
                                                  int lane) {
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
  const float sc = pow2_scale_terms(amax);
  for (int b = lane; b < H / 16; b += 32) {
    float r[16];
    load_bf16x16_scaled(row + 16 * b, sc, r);
    uint2 codes[kTerms];
    uint32_t sf[kTerms];
    encode_terms16(r, codes, sf);
    store_terms16(codes, sf, xq, xsf, (size_t)t * kTerms, H, b);
  }
  if (lane == 0) *inv = 1.f / sc;
}

}  // namespace moe
