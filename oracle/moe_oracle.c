/*
 * Float64 CPU oracle for one decode step of a Mixture-of-Experts FFN layer.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path may call this file:
 * only the test-suite, the smoke check and the CPU-baseline leg of the
 * benchmark load it.  It shares no code, header, table or constant with the
 * CUDA path.
 *
 * What is computed (the plain definition, written out in float64):
 *   logits[t,e] = sum_h x[t,h] * Wr[e,h]  (+ bias[e])
 *   S_t         = the k experts of largest logit, ties to the lower index
 *   w_tj        = exp(l_j - lmax) / sum_{i in S_t} exp(l_i - lmax)     (renorm)
 *              or exp(l_j - lmax) / sum_{all e} exp(l_e - lmax)        (no renorm)
 *   g = x_t . Wg_e^T,  u = x_t . Wu_e^T,  h = g / (1 + exp(-g)) * u    (SwiGLU)
 *   y = h . Wd_e^T
 *   out_t = sum_j w_tj * y_{t,e_tj}  (+ residual_t)
 *
 * The decode step of the MoE layers named in the paper's setup table
 * (Qwen3-Coder-480B FP8, Qwen3-235B-A22B NVFP4; Section 4, "Setup") is what
 * this computes; the paper states that decode is dominated by weight reads
 * and is memory-bound (Section 2.1).  The paper fixes none of the numeric
 * details; the readings used here are:
 *   - top-k on the logits (not probabilities), ordered by (value desc,
 *     index asc); -0.0 == +0.0 is a tie;
 *   - SwiGLU with separate gate and up matrices, no biases;
 *   - FP8: OCP OFP8 E4M3 codes with one fp32 scale per 128x128 tile of the
 *     [N_out, K_in] matrix;
 *   - NVFP4: OCP E2M1 codes, two per byte (low nibble = even K index), one
 *     E4M3 scale per 16 consecutive K elements, one fp32 scale per expert
 *     and matrix;
 *   - activations used exactly as given (bf16), no rounding of h or y.
 * Parity status: the codecs, the top-k, the permutation and the layer are
 * pinned by the tests (exhaustive codec tables, brute force, closed forms and
 * invariants).  The paper itself prints no value of this computation.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define FMT_FP8 1
#define FMT_NVFP4 2

/* ---------------- codecs (OCP OFP8 / OCP MX E2M1 definitions) ---------------- */

/* E4M3: 1 sign, 4 exponent (bias 7), 3 mantissa bits.  No infinities; the two
 * codes with all exponent and mantissa bits set (0x7F, 0xFF) are NaN.
 * normal:    (-1)^s * 2^(e-7) * (1 + m/8)   for e > 0
 * subnormal: (-1)^s * 2^(-6) * (m/8)        for e = 0 */
double oracle_e4m3(uint8_t code) {
  int s = (code >> 7) & 1;
  int e = (code >> 3) & 15;
  int m = code & 7;
  double v;
  if (e == 15 && m == 7) return NAN;
  if (e == 0)
    v = ldexp((double)m / 8.0, -6);
  else
    v = ldexp(1.0 + (double)m / 8.0, e - 7);
  return s ? -v : v;
}

/* E2M1: 1 sign, 2 exponent (bias 1), 1 mantissa bit; 4-bit code.
 * normal:    (-1)^s * 2^(e-1) * (1 + m/2)   for e > 0
 * subnormal: (-1)^s * (m/2)                 for e = 0 */
double oracle_e2m1(uint8_t nibble) {
  int s = (nibble >> 3) & 1;
  int e = (nibble >> 1) & 3;
  int m = nibble & 1;
  double v;
  if (e == 0)
    v = (double)m / 2.0;
  else
    v = ldexp(1.0 + (double)m / 2.0, e - 1);
  return s ? -v : v;
}

/* bf16 bits -> value: the bf16 pattern is the top half of an IEEE binary32. */
double oracle_bf16(uint16_t bits) {
  uint32_t u = (uint32_t)bits << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return (double)f;
}

/* ---------------- dequantised weight element ---------------- */

typedef struct {
  int fmt;          /* FMT_FP8 or FMT_NVFP4 */
  int N, K;         /* one expert's matrix is [N, K], K contiguous */
  const uint8_t* codes;   /* FP8: [E, N, K]; NVFP4: [E, N, K/2] */
  const void* scales;     /* FP8: float [E, N/128, K/128]; NVFP4: e4m3 [E, N, K/16] */
  const float* tscale;    /* NVFP4: float [E]; unused for FP8 */
} oracle_mat_t;

/* W_e[n][k] as a float64 number. */
static double w_at(const oracle_mat_t* m, int e, int n, int k) {
  if (m->fmt == FMT_FP8) {
    const uint8_t* c = m->codes + ((size_t)e * m->N + n) * (size_t)m->K;
    const float* s = (const float*)m->scales;
    size_t nb = (size_t)(m->N / 128), kb = (size_t)(m->K / 128);
    double scale = (double)s[((size_t)e * nb + (size_t)(n / 128)) * kb + (size_t)(k / 128)];
    return oracle_e4m3(c[k]) * scale;
  } else {
    const uint8_t* c = m->codes + ((size_t)e * m->N + n) * (size_t)(m->K / 2);
    uint8_t byte = c[k / 2];
    uint8_t nib = (k % 2 == 0) ? (byte & 15) : (byte >> 4);
    const uint8_t* sf = (const uint8_t*)m->scales + ((size_t)e * m->N + n) * (size_t)(m->K / 16);
    return oracle_e2m1(nib) * oracle_e4m3(sf[k / 16]) * (double)m->tscale[e];
  }
}

/* Dequantise one whole expert matrix into dst[N*K] (row-major). */
void oracle_dequant(int fmt, int N, int K, const uint8_t* codes, const void* scales,
                    const float* tscale, int e, double* dst) {
  oracle_mat_t m = {fmt, N, K, codes, scales, tscale};
  for (int n = 0; n < N; ++n)
    for (int k = 0; k < K; ++k) dst[(size_t)n * K + k] = w_at(&m, e, n, k);
}

/* ---------------- router ---------------- */

/* logits[t,e] = sum_h x[t,h] * Wr[e,h] (+ bias[e]), float64 sum in h order. */
void oracle_router_logits(const uint16_t* x, const float* wr, const float* bias, int T, int H,
                          int E, double* logits) {
#pragma omp parallel for collapse(2) schedule(static)
  for (int t = 0; t < T; ++t)
    for (int e = 0; e < E; ++e) {
      double acc = 0.0;
      for (int h = 0; h < H; ++h)
        acc += oracle_bf16(x[(size_t)t * H + h]) * (double)wr[(size_t)e * H + h];
      if (bias) acc += (double)bias[e];
      logits[(size_t)t * E + e] = acc;
    }
}

/* Top-k by (value desc, index asc) and the gate weights.
 * renorm = 1: softmax restricted to the selected experts.
 * renorm = 0: the full-softmax probability of each selected expert. */
void oracle_topk(const double* logits, int T, int E, int k, int renorm, int32_t* ids,
                 double* gates) {
  for (int t = 0; t < T; ++t) {
    const double* l = logits + (size_t)t * E;
    int32_t* id = ids + (size_t)t * k;
    for (int j = 0; j < k; ++j) {
      int best = -1;
      for (int e = 0; e < E; ++e) {
        int taken = 0;
        for (int i = 0; i < j; ++i)
          if (id[i] == e) taken = 1;
        if (taken) continue;
        /* strictly greater keeps the lower index on equal values */
        if (best < 0 || l[e] > l[best]) best = e;
      }
      id[j] = best;
    }
    double lmax = l[id[0]];
    double den = 0.0;
    if (renorm) {
      for (int j = 0; j < k; ++j) den += exp(l[id[j]] - lmax);
    } else {
      for (int e = 0; e < E; ++e) den += exp(l[e] - lmax);
    }
    for (int j = 0; j < k; ++j) gates[(size_t)t * k + j] = exp(l[id[j]] - lmax) / den;
  }
}

/* Token -> expert permutation.  Assignment a = t*k + j goes to expert ids[a].
 * counts[e]    = number of assignments to e
 * offsets[e]   = sum_{e' < e} counts[e'],  offsets[E] = T*k
 * sorted[p]    = the assignments sorted stably by expert (then by a)
 * inv[a]       = position of a in sorted
 * active[0]    = number of experts with counts > 0; active[1..] = those ids, ascending */
void oracle_permute(const int32_t* ids, int T, int k, int E, int32_t* counts, int32_t* offsets,
                    int32_t* sorted, int32_t* inv, int32_t* active) {
  int A = T * k;
  for (int e = 0; e < E; ++e) counts[e] = 0;
  for (int a = 0; a < A; ++a) counts[ids[a]] += 1;
  offsets[0] = 0;
  for (int e = 0; e < E; ++e) offsets[e + 1] = offsets[e] + counts[e];
  int p = 0;
  for (int e = 0; e < E; ++e)
    for (int a = 0; a < A; ++a)
      if (ids[a] == e) {
        sorted[p] = a;
        inv[a] = p;
        ++p;
      }
  int n = 0;
  for (int e = 0; e < E; ++e)
    if (counts[e] > 0) active[1 + n++] = e;
  active[0] = n;
}

/* ---------------- one expert applied to one token ---------------- */

/* y[H] = W_d,e . (silu(W_g,e . x) * (W_u,e . x)), everything in float64. */
static void expert_ffn(const oracle_mat_t* mg, const oracle_mat_t* mu, const oracle_mat_t* md,
                       int e, int H, int I, const double* x, double* h, double* y) {
  for (int i = 0; i < I; ++i) {
    double g = 0.0, u = 0.0;
    for (int c = 0; c < H; ++c) {
      g += x[c] * w_at(mg, e, i, c);
      u += x[c] * w_at(mu, e, i, c);
    }
    h[i] = g / (1.0 + exp(-g)) * u;
  }
  for (int r = 0; r < H; ++r) {
    double acc = 0.0;
    for (int i = 0; i < I; ++i) acc += h[i] * w_at(md, e, r, i);
    y[r] = acc;
  }
}

/* The layer output for the tokens listed in `tokens` (n_tok of them), given the
 * routing (ids, gates) of every token.  x_rows: [T, H] bf16 bits.  out: [n_tok, H].
 * residual (nullable): [T, H] bf16 bits added to the output. */
void oracle_moe_tokens(int fmt, int E, int H, int I, const uint8_t* wg, const uint8_t* wu,
                       const uint8_t* wd, const void* sg, const void* su, const void* sd,
                       const float* tsg, const float* tsu, const float* tsd, const uint16_t* x,
                       const int32_t* ids, const double* gates, int T, int k,
                       const uint16_t* residual, const int32_t* tokens, int n_tok, double* out) {
  oracle_mat_t mg = {fmt, I, H, wg, sg, tsg};
  oracle_mat_t mu = {fmt, I, H, wu, su, tsu};
  oracle_mat_t md = {fmt, H, I, wd, sd, tsd};
  (void)E;
  (void)T;
  /* y of every (token, slot) pair first, then the gate-weighted sum in slot
   * order, so the result does not depend on the thread schedule. */
  double* ybuf = (double*)malloc(sizeof(double) * (size_t)n_tok * (size_t)k * (size_t)H);
#pragma omp parallel
  {
    double* xv = (double*)malloc(sizeof(double) * (size_t)H);
    double* hv = (double*)malloc(sizeof(double) * (size_t)I);
#pragma omp for collapse(2) schedule(dynamic, 1)
    for (int q = 0; q < n_tok; ++q)
      for (int j = 0; j < k; ++j) {
        int t = tokens[q];
        for (int c = 0; c < H; ++c) xv[c] = oracle_bf16(x[(size_t)t * H + c]);
        int e = ids[(size_t)t * k + j];
        expert_ffn(&mg, &mu, &md, e, H, I, xv, hv, ybuf + ((size_t)q * k + j) * H);
      }
    free(xv);
    free(hv);
  }
  for (int q = 0; q < n_tok; ++q) {
    int t = tokens[q];
    for (int r = 0; r < H; ++r) {
      double acc = 0.0;
      for (int j = 0; j < k; ++j)
        acc += gates[(size_t)t * k + j] * ybuf[((size_t)q * k + j) * H + r];
      if (residual) acc += oracle_bf16(residual[(size_t)t * H + r]);
      out[(size_t)q * H + r] = acc;
    }
  }
  free(ybuf);
}

/* One expert applied to one float64 input vector (used by the unfused-path
 * tests, which compare the per-assignment expert outputs y). */
void oracle_expert_vec(int fmt, int H, int I, const uint8_t* wg, const uint8_t* wu,
                       const uint8_t* wd, const void* sg, const void* su, const void* sd,
                       const float* tsg, const float* tsu, const float* tsd, int e,
                       const double* x, double* y) {
  oracle_mat_t mg = {fmt, I, H, wg, sg, tsg};
  oracle_mat_t mu = {fmt, I, H, wu, su, tsu};
  oracle_mat_t md = {fmt, H, I, wd, sd, tsd};
  double* hv = (double*)malloc(sizeof(double) * (size_t)I);
  expert_ffn(&mg, &mu, &md, e, H, I, x, hv, y);
  free(hv);
}

/* Round a finite double to the nearest bf16 value (ties to even) and return
 * its bit pattern.  bf16 keeps 8 significant bits and binary32's exponent
 * range; the values handled here are normal binary32 numbers. */
static uint16_t bf16_rne_bits(double v) {
  if (v == 0.0) return signbit(v) ? 0x8000u : 0u;
  int ex;
  double m = frexp(v, &ex);            /* v = m * 2^ex, 0.5 <= |m| < 1 */
  double r = nearbyint(ldexp(m, 8));   /* 8 significant bits, ties to even */
  float f = (float)ldexp(r, ex - 8);   /* exactly representable */
  uint32_t u;
  memcpy(&u, &f, sizeof u);
  return (uint16_t)(u >> 16);
}

/* RMSNorm with unit weight, rounded to bf16:
 * xn[t,h] = bf16( x[t,h] / sqrt(mean_h x[t,h]^2 + eps) ).  Returns bf16 bits. */
void oracle_rmsnorm_bf16(const uint16_t* x, int T, int H, double eps, uint16_t* xn) {
  for (int t = 0; t < T; ++t) {
    double ss = 0.0;
    for (int h = 0; h < H; ++h) {
      double v = oracle_bf16(x[(size_t)t * H + h]);
      ss += v * v;
    }
    double r = 1.0 / sqrt(ss / H + eps);
    for (int h = 0; h < H; ++h) xn[(size_t)t * H + h] = bf16_rne_bits(oracle_bf16(x[(size_t)t * H + h]) * r);
  }
}

/* Round doubles to bf16 bit patterns (used to state the bf16 output format). */
void oracle_to_bf16(const double* v, size_t n, uint16_t* bits) {
  for (size_t i = 0; i < n; ++i) bits[i] = bf16_rne_bits(v[i]);
}
