// Expert FFN kernels on the 5th-generation tensor cores (tcgen05).
//
// Same work decomposition as ffn.cuh (stream-K over (expert, token chunk,
// row tile) items, TMA-fed shared-memory ring, tickets for SwiGLU and the
// bf16 conversion), different engine:
//
// * Decoder warps 0-7 own one weight row each: warp w, lane l decodes row
//   32*(w%4)+l of box A0 (w < 4) or A1 (w >= 4), which is also its TMEM lane.
//   FP8/NVFP4 codes are converted exactly to f16 in registers and written to
//   a 3-deep ring of A operands in tensor memory (tcgen05.st), 128 K per unit.
// * Warp 13 (one thread) issues tcgen05.mma kind::f16, M=128, N=NT, K=16,
//   with A from TMEM, the token rows (B, K-major, 128B-swizzled shared
//   memory, put there by TMA) and an fp32 accumulator in TMEM.  Every stage
//   gets a fresh accumulator so that the FP8 128x128 block scale can be
//   applied to it.
// * Epilogue warps 8-11 read each stage's accumulator back (tcgen05.ld),
//   apply the scale, keep the item's sums in registers, and flush them with
//   red.global.add at the item's end, as ffn.cuh does.  Decoding never waits
//   for an accumulator read.
// * Warp 12 (one thread) is the TMA producer.
// Every mbarrier wait is bounded; TMEM is always released before exit.
#pragma once

#include "ffn.cuh"

namespace moe {

constexpr int kTcDecWarps = 8;                   // warps 0-7: decode weights into TMEM
constexpr int kTcEpiWarp0 = 8;                   // warps 8-11: read back accumulators
constexpr int kTcEpiWarps = 4;
constexpr int kTcProducerWarp = 12;              // warp 12: TMA producer
constexpr int kTcMmaWarp = 13;                   // warp 13: MMA issuer, owns TMEM
constexpr int kTcThreads = 14 * 32;
constexpr int kTcUK = 64;                        // K elements per A unit
constexpr int kTcUCols = kTcUK / 2;              // TMEM columns per box per unit
constexpr int kTcARing = 6;                      // A units in flight (both boxes each)
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kTmemA = 0;                   // A ring: 6 x (2 boxes x 32 columns)
constexpr uint32_t kTmemD = 384;                 // D ring: 2 x (2 boxes x NT columns)

template <int FMT, int NT>
struct TcGeom {
  static constexpr int KEL = FmtTraits<FMT>::KEL;
  static constexpr int UPS = KEL / kTcUK;  // A units per stage
  static constexpr int A0 = 0;
  static constexpr int A1 = kRowsHalf * kRowBytes;
  static constexpr int S0 = 2 * kRowsHalf * kRowBytes;
  static constexpr int S1 = S0 + kRowsHalf * FmtTraits<FMT>::SBYTES;
  static constexpr int B = S0 + 2 * kRowsHalf * FmtTraits<FMT>::SBYTES;  // 1024-aligned
  static constexpr int KATOMS = KEL / 64;          // 64-element (128-byte) K atoms
  static constexpr int BATOM = NT * 128;           // bytes of one K atom of the B tile
  static constexpr int RAW = B + KATOMS * BATOM;
  static constexpr int BYTES = (RAW + 1023) / 1024 * 1024;
  static constexpr int STAGES_RAW = (224 * 1024) / BYTES;
  static constexpr int STAGES = STAGES_RAW > 8 ? 8 : STAGES_RAW;
  static constexpr int SMEM = STAGES * BYTES + 1024;
};

template <int FMT, int NT>
__global__ void __launch_bounds__(kTcThreads, 1)
    ffn_tc_kernel(const __grid_constant__ CUtensorMap tmA0,
                  const __grid_constant__ CUtensorMap tmA1,
                  const __grid_constant__ CUtensorMap tmS0,
                  const __grid_constant__ CUtensorMap tmS1,
                  const __grid_constant__ CUtensorMap tmB, const FfnParams p) {
  using G = TcGeom<FMT, NT>;
  constexpr int KEL = G::KEL;
  constexpr int UPS = G::UPS;
  constexpr int S = G::STAGES;
  static_assert(NT == 16 || NT == 32, "tcgen05 tile N must be 16 or 32 tokens");
  static_assert(kTmemD + 4 * NT <= kTmemCols, "TMEM budget");

  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);

  __shared__ __align__(8) uint64_t full_bar[S];
  __shared__ __align__(8) uint64_t empty_bar[S];
  __shared__ __align__(8) uint64_t afull_bar[kTcARing];
  __shared__ __align__(8) uint64_t aempty_bar[kTcARing];
  __shared__ __align__(8) uint64_t dfull_bar[2];
  __shared__ __align__(8) uint64_t dempty_bar[2];
  __shared__ __align__(8) uint64_t final_bar;
  __shared__ int s_cpre[kMaxE + 1];
  __shared__ int s_tok[NT];
  __shared__ uint32_t s_tmem;
  __shared__ volatile int s_abort;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    s_abort = 0;
    for (int i = 0; i < S; ++i) {
      mbar_init(&full_bar[i], 1);
      mbar_init(&empty_bar[i], 1);
    }
    for (int i = 0; i < kTcARing; ++i) {
      mbar_init(&afull_bar[i], kTcDecWarps);
      mbar_init(&aempty_bar[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&dfull_bar[i], 1);
      mbar_init(&dempty_bar[i], kTcEpiWarps);
    }
    mbar_init(&final_bar, 1);
    fence_mbar_init();
  }
  if (warp == kTcMmaWarp) {
    tmem_alloc(&s_tmem, kTmemCols);
    tmem_relinquish();
  }
  // Launched as a programmatic dependent: everything above overlapped the
  // previous kernel; from here on its outputs are read.
  pdl_wait();
  pdl_launch_dependents();
  const int nA = __ldg(p.active);
  for (int i = threadIdx.x; i <= nA; i += blockDim.x) s_cpre[i] = __ldg(p.cprefix + i);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s_tmem;

  const int N = (p.phase == 1) ? p.I : p.H;
  const int K = (p.phase == 1) ? p.H : p.I;
  const int rtiles = (p.phase == 1) ? p.I / kRowsHalf : p.H / (2 * kRowsHalf);
  const int KB = K / KEL;
  const long long items = (long long)s_cpre[nA] * rtiles;
  const long long total = items * KB;
  const long long s_begin = total * blockIdx.x / gridDim.x;
  const long long s_end = total * (blockIdx.x + 1) / gridDim.x;
  const long long nst = s_end - s_begin;
  const uint32_t timeout_bit = (p.phase == 1) ? kStatusTimeoutGateUp : kStatusTimeoutDown;
  constexpr int kTeardown = (kTcDecWarps + kTcEpiWarps + 1) * 32;

  // ================================================================ producer
  if (warp == kTcProducerWarp) {
    if (lane == 0 && nst > 0) {
      tma_prefetch_desc(&tmA0);
      tma_prefetch_desc(&tmA1);
      tma_prefetch_desc(&tmB);
      if (FMT == 2) {
        tma_prefetch_desc(&tmS0);
        tma_prefetch_desc(&tmS1);
      }
      const uint64_t pol_w = policy_evict_first();
      const uint64_t pol_a = policy_evict_last();
      long long cur_item = -1;
      ItemInfo inf{};
      long long issued = 0;
      for (long long s = s_begin; s < s_end; ++s, ++issued) {
        const long long it = s / KB;
        const int kb = (int)(s % KB);
        if (it != cur_item) {
          cur_item = it;
          inf = decode_item(it, rtiles, s_cpre, nA, p, NT);
          if (p.phase == 1)
            for (int j = 0; j < inf.nvalid; ++j) s_tok[j] = __ldg(p.sorted + inf.arow0 + j) / p.k;
        }
        const int slot = (int)(issued % S);
        const uint32_t round = (uint32_t)(issued / S);
        if (!mbar_wait_bounded(&empty_bar[slot], (round & 1u) ^ 1u, p.wait_ns, &s_abort)) {
          set_status(p.status, timeout_bit);
          s_abort = 1;
          break;
        }
        if (p.test_stall && issued == 0) continue;  // test hook: this stage never arrives
        unsigned char* st = smem + (size_t)slot * G::BYTES;
        const int npad8 = (inf.nvalid + 7) & ~7;
        uint32_t bytes = 2u * kRowsHalf * kRowBytes + 2u * kRowsHalf * FmtTraits<FMT>::SBYTES;
        bytes += (p.phase == 1) ? (uint32_t)(inf.nvalid * KEL * 2)
                                : (uint32_t)(G::KATOMS * npad8 * 128);
        mbar_arrive_expect_tx(&full_bar[slot], bytes);
        int rowA0, rowA1;
        if (p.phase == 1) {
          rowA0 = inf.e * N + inf.rt * kRowsHalf;
          rowA1 = rowA0;
        } else {
          rowA0 = inf.e * N + inf.rt * 2 * kRowsHalf;
          rowA1 = rowA0 + kRowsHalf;
        }
        tma_load_2d(st + G::A0, &tmA0, &full_bar[slot], kb * kRowBytes, rowA0, pol_w);
        tma_load_2d(st + G::A1, &tmA1, &full_bar[slot], kb * kRowBytes, rowA1, pol_w);
        if (FMT == 2) {
          tma_load_2d(st + G::S0, &tmS0, &full_bar[slot], kb * 16, rowA0, pol_w);
          tma_load_2d(st + G::S1, &tmS1, &full_bar[slot], kb * 16, rowA1, pol_w);
        }
        // token rows: K atom q of row j lands at B + q*NT*128 + j*128 (128B swizzle)
        if (p.phase == 1) {
          for (int j = 0; j < inf.nvalid; ++j)
#pragma unroll
            for (int q = 0; q < G::KATOMS; ++q)
              tma_load_2d(st + G::B + q * G::BATOM + j * 128, &tmB, &full_bar[slot],
                          kb * KEL + q * 64, s_tok[j], pol_a);
        } else {
          for (int r8 = 0; r8 < npad8; r8 += 8)
#pragma unroll
            for (int q = 0; q < G::KATOMS; ++q)
              tma_load_2d(st + G::B + q * G::BATOM + r8 * 128, &tmB, &full_bar[slot],
                          kb * KEL + q * 64, inf.arow0 + r8, pol_a);
        }
      }
      const long long first = issued > S ? issued - S : 0;
      for (long long j = first; j < issued; ++j) {
        if (p.test_stall && j == 0) continue;
        mbar_wait_bounded(&full_bar[j % S], (uint32_t)((j / S) & 1), p.wait_ns, nullptr);
      }
    }
    return;
  }

  // ================================================================ MMA issuer
  if (warp == kTcMmaWarp) {
    if (lane == 0) {
      constexpr uint32_t idesc = tc_idesc_f16(128, NT);
      long long uc = 0;
      bool ok = true;
      for (long long i = 0; i < nst && ok; ++i) {
        const int slot = (int)(i % S);
        const int db = (int)(i & 1);
        ok = mbar_wait_bounded(&full_bar[slot], (uint32_t)(i / S) & 1u, p.wait_ns, &s_abort) &&
             mbar_wait_bounded(&dempty_bar[db], ((uint32_t)(i >> 1) & 1u) ^ 1u, p.wait_ns,
                               &s_abort);
        const uint32_t bbase = smem_u32(smem + (size_t)slot * G::BYTES + G::B);
        for (int v = 0; v < UPS && ok; ++v, ++uc) {
          const int ab = (int)(uc % kTcARing);
          ok = mbar_wait_bounded(&afull_bar[ab], (uint32_t)(uc / kTcARing) & 1u, p.wait_ns,
                                 &s_abort);
          if (!ok) break;
          tc_fence_after();
#pragma unroll
          for (int kk = 0; kk < kTcUK / 16; ++kk) {
            const int kel = v * kTcUK + kk * 16;  // element offset in the stage
            const uint64_t bdesc =
                tc_desc_sw128(bbase + (kel >> 6) * G::BATOM + (kel & 63) * 2);
#pragma unroll
            for (int box = 0; box < 2; ++box) {
              const uint32_t a_t = tmem + kTmemA + ab * (2 * kTcUCols) + box * kTcUCols + kk * 8;
              const uint32_t d_t = tmem + kTmemD + db * 2 * NT + box * NT;
              tc_mma_f16_ts(d_t, a_t, bdesc, idesc, (v > 0 || kk > 0) ? 1u : 0u);
            }
          }
          tc_commit(&aempty_bar[ab]);
        }
        if (!ok) break;
        tc_commit(&empty_bar[slot]);
        tc_commit(&dfull_bar[db]);
      }
      if (!ok) {
        set_status(p.status, timeout_bit);
        s_abort = 1;
      }
      // every MMA this thread issued has completed before TMEM is released
      tc_commit(&final_bar);
      mbar_wait_bounded(&final_bar, 0, p.wait_ns, nullptr);
    }
    __syncwarp();
    asm volatile("bar.sync 2, %0;" ::"n"(kTeardown) : "memory");
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
    return;
  }

  // ================================================================ decoders
  if (warp < kTcDecWarps) {
    const int quad = warp & 3;
    const int box = warp >> 2;           // 0: rows of box A0, 1: rows of box A1
    const int row = quad * 32 + lane;    // row within the box == TMEM lane
    const uint32_t lane_addr = (uint32_t)(quad * 32) << 16;
    const uint32_t sw = (uint32_t)(row & 7);
    bool dead = false;
    long long uc = 0;         // A units stored so far
    bool pending = false;     // the last unit's stores are issued but not yet announced
    uint32_t scb[16];         // NVFP4: this row's 16 stage scales as f16 broadcast pairs
    uint32_t abox = 0;
    for (long long i = 0; i < nst && !dead; ++i) {
      const int slot = (int)(i % S);
      if (!mbar_wait_bounded(&full_bar[slot], (uint32_t)(i / S) & 1u, p.wait_ns, &s_abort)) {
        set_status(p.status, timeout_bit);
        s_abort = 1;
        dead = true;
        break;
      }
      const uint32_t st = smem_u32(smem + (size_t)slot * G::BYTES);
      abox = st + (box == 0 ? G::A0 : G::A1) + row * kRowBytes;
      if (FMT == 2) {
        const uint4 sv = lds128(st + (box == 0 ? G::S0 : G::S1) + row * 16);
        const uint32_t sw4[4] = {sv.x, sv.y, sv.z, sv.w};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          uint32_t lo, hi;
          e4m3x4_to_f16x4(sw4[q], lo, hi);
          scb[4 * q + 0] = __byte_perm(lo, 0, 0x1010);
          scb[4 * q + 1] = __byte_perm(lo, 0, 0x3232);
          scb[4 * q + 2] = __byte_perm(hi, 0, 0x1010);
          scb[4 * q + 3] = __byte_perm(hi, 0, 0x3232);
        }
      }
#pragma unroll
      for (int v = 0; v < UPS; ++v) {
        // decode kTcUK (=64) K of this row into 32 f16x2 columns
        uint32_t col[kTcUCols];
        if (FMT == 1) {
#pragma unroll
          for (int cc = 0; cc < 4; ++cc) {
            const int c = 4 * v + cc;  // 16-byte chunk = 16 codes
            const uint4 q4 = lds128(abox + ((c ^ sw) << 4));
            e4m3x4_to_f16x4(q4.x, col[8 * cc + 0], col[8 * cc + 1]);
            e4m3x4_to_f16x4(q4.y, col[8 * cc + 2], col[8 * cc + 3]);
            e4m3x4_to_f16x4(q4.z, col[8 * cc + 4], col[8 * cc + 5]);
            e4m3x4_to_f16x4(q4.w, col[8 * cc + 6], col[8 * cc + 7]);
          }
        } else {
#pragma unroll
          for (int cc = 0; cc < 2; ++cc) {
            const int c = 2 * v + cc;  // 16-byte chunk = 32 codes = blocks 2c, 2c+1
            const uint4 q4 = lds128(abox + ((c ^ sw) << 4));
            const uint32_t w4[4] = {q4.x, q4.y, q4.z, q4.w};
#pragma unroll
            for (int ww = 0; ww < 4; ++ww) {
              uint32_t d[4];
              e2m1x8_to_f16x8(w4[ww], d);
              const uint32_t sc = scb[2 * c + (ww >> 1)];
#pragma unroll
              for (int q = 0; q < 4; ++q) col[16 * cc + 4 * ww + q] = hmul2_u32(d[q], sc);
            }
          }
        }
        // announce the previous unit now that its stores have had a decode to drain
        if (pending) {
          tmem_st_wait();
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&afull_bar[(uc - 1) % kTcARing]);
          pending = false;
        }
        const int ab = (int)(uc % kTcARing);
        if (!mbar_wait_bounded(&aempty_bar[ab], ((uint32_t)(uc / kTcARing) & 1u) ^ 1u,
                               p.wait_ns, &s_abort)) {
          set_status(p.status, timeout_bit);
          s_abort = 1;
          dead = true;
          break;
        }
        tc_fence_after();
        const uint32_t a_t = tmem + lane_addr + kTmemA + ab * (2 * kTcUCols) + box * kTcUCols;
#pragma unroll
        for (int q = 0; q < kTcUCols / 16; ++q) {
          uint32_t part[16];
#pragma unroll
          for (int m = 0; m < 16; ++m) part[m] = col[16 * q + m];
          tmem_st16(a_t + 16 * q, part);
        }
        pending = true;
        ++uc;
      }
    }
    if (pending && !dead) {
      tmem_st_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&afull_bar[(uc - 1) % kTcARing]);
    }
    tc_fence_before();
    asm volatile("bar.sync 2, %0;" ::"n"(kTeardown) : "memory");
    return;
  }

  // ================================================================ epilogue warps
  // Warp 8+q reads TMEM lanes 32q..32q+31: row 32q+lane of both boxes.
  const int quad = warp - kTcEpiWarp0;
  const int row = quad * 32 + lane;
  const uint32_t lane_addr = (uint32_t)(quad * 32) << 16;
  const int et = threadIdx.x - kTcEpiWarp0 * 32;  // 0..127
  constexpr int kEpiThreads = kTcEpiWarps * 32;

  float acc0[NT], acc1[NT];
#pragma unroll
  for (int j = 0; j < NT; ++j) acc0[j] = acc1[j] = 0.f;
  bool dead = false;

  auto flush = [&](const ItemInfo& fi, bool is_dead) {
    float ts0 = 1.f, ts1 = 1.f;
    if (FMT == 2) {
      ts0 = __ldg(p.ts0 + fi.e);
      ts1 = __ldg(p.ts1 + fi.e);
    }
    if (!is_dead) {
#pragma unroll
      for (int j = 0; j < NT; ++j) {
        if (j >= fi.nvalid) continue;
        const int arow = fi.arow0 + j;
        const int a = __ldg(p.sorted + arow);
        if (p.phase == 1) {
          const float sc = __ldg(p.xinv + a / p.k);
          const int f = fi.rt * kRowsHalf + row;
          float* gr = p.gu + (size_t)arow * 2 * p.I + f;
          red_add_f32(gr, acc0[j] * sc * ts0);
          red_add_f32(gr + p.I, acc1[j] * sc * ts1);
        } else {
          const float sc = __ldcg(p.xinv + arow);
          const int hrow = fi.rt * 2 * kRowsHalf + row;
          if (p.fused) {
            const float gw = __ldg(p.gates + a) * sc;
            float* orow = p.oacc + (size_t)(a / p.k) * p.H + hrow;
            red_add_f32(orow, gw * acc0[j] * ts0);
            red_add_f32(orow + kRowsHalf, gw * acc1[j] * ts1);
          } else {
            float* yrow = p.y_perm + (size_t)arow * p.H + hrow;
            red_add_f32(yrow, acc0[j] * sc * ts0);
            red_add_f32(yrow + kRowsHalf, acc1[j] * sc * ts1);
          }
        }
      }
    }
#pragma unroll
    for (int j = 0; j < NT; ++j) acc0[j] = acc1[j] = 0.f;
  };

  long long cur_item = -1;
  ItemInfo inf{};
  for (long long i = 0; i < nst; ++i) {
    const long long s = s_begin + i;
    const long long it = s / KB;
    const int kb = (int)(s % KB);
    if (it != cur_item) {
      cur_item = it;
      inf = decode_item(it, rtiles, s_cpre, nA, p, NT);
    }
    float bs0 = 1.f, bs1 = 1.f;
    if (FMT == 1) {  // the FP8 block scales of this stage's two boxes
      const int KB128 = K / 128;
      if (p.phase == 1) {
        const size_t tile = ((size_t)inf.e * (N / 128) + inf.rt) * KB128 + kb;
        bs0 = __ldg(p.s0 + tile);
        bs1 = __ldg(p.s1 + tile);
      } else {
        const size_t tile = ((size_t)inf.e * (N / 128) + 2 * inf.rt) * KB128 + kb;
        bs0 = __ldg(p.s0 + tile);
        bs1 = __ldg(p.s0 + tile + KB128);
      }
    }
    const int db = (int)(i & 1);
    if (!dead &&
        !mbar_wait_bounded(&dfull_bar[db], (uint32_t)(i >> 1) & 1u, p.wait_ns, &s_abort)) {
      set_status(p.status, timeout_bit);
      s_abort = 1;
      dead = true;
    }
    if (!dead) {
      tc_fence_after();
      const uint32_t d_t = tmem + lane_addr + kTmemD + db * 2 * NT;
      uint32_t d0[NT], d1[NT];
#pragma unroll
      for (int c = 0; c < NT; c += 16) {
        uint32_t t0[16], t1[16];
        tmem_ld16(d_t + c, t0);
        tmem_ld16(d_t + NT + c, t1);
#pragma unroll
        for (int q = 0; q < 16; ++q) {
          d0[c + q] = t0[q];
          d1[c + q] = t1[q];
        }
      }
      tmem_ld_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&dempty_bar[db]);
#pragma unroll
      for (int j = 0; j < NT; ++j) {
        acc0[j] = fmaf(bs0, __uint_as_float(d0[j]), acc0[j]);
        acc1[j] = fmaf(bs1, __uint_as_float(d1[j]), acc1[j]);
      }
    }
    const bool closes = (i + 1 == nst) || ((s + 1) / KB != it);
    if (closes) flush(inf, dead);
  }
  tc_fence_before();
  asm volatile("bar.sync 2, %0;" ::"n"(kTeardown) : "memory");
}

}  // namespace moe
