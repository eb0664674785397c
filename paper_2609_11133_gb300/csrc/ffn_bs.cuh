// NVFP4 expert FFN on the tensor cores' block-scaled path:
// tcgen05.mma kind::mxf4nvf4 with one UE4M3 scale per 16 K on both operands.
//
// The weights go to the tensor core exactly as stored: TMA copies 128-row x
// 128-byte boxes of E2M1 codes (256 K) with the 128B swizzle into shared
// memory, and their E4M3 scales (128 rows x 16 bytes) next to them.  The
// activations arrive as four NVFP4 terms per token (act_terms.cuh), i.e. four
// rows of the B operand.  Nothing is decoded on the CUDA cores; the kernel is
// a TMA -> tensor-core stream.
//
// Work decomposition as in ffn.cuh: a persistent grid, stream-K over the
// K-stages of all (active expert, <=NT-token chunk, row tile) items.  Per
// stage and matrix (gate/up in phase 1, the two 128-row halves of down in
// phase 2) four MMAs of M=128, N=4*NT, K=64 accumulate into tensor memory.
//
// Roles (352 threads):
//   warps 0-3  scale writers: copy the stage's A scales from shared memory and
//              the B scales from global memory into tensor memory, in the
//              layout the MMA reads (below); warp w owns TMEM lanes 32w..32w+31
//   warps 4-7  epilogue: read an item's accumulators (tcgen05.ld), add the
//              four terms of each token, apply the tensor and activation
//              scales and add the partial sums to global memory (red.add)
//   warps 8,10 TMA producers (one thread each): warp 8 arms each stage's
//              barrier and copies box A0 and its scales, warp 10 box A1, its
//              scales and the activation rows (two issuing warps keep more
//              copies going than one)
//   warp 9     MMA issuer (one thread); allocates and frees tensor memory
//
// Scale-factor layout in tensor memory (scale_vec::4X, M = 128): the four
// scales of A row m for one MMA (K = 64) are the bytes of the 32-bit cell at
// lane m % 32 (of every lane quadrant), column c + m / 32, where c, the
// address the MMA is given, is a multiple of 4; B row n likewise.  So one MMA
// uses 4 columns per operand, written by four warps with the same values.
//
// Every wait is bounded (p.wait_ns); an expired wait sets the status word and
// the kernel winds down, freeing its tensor memory.
#pragma once

#include "act_terms.cuh"
#include "ffn.cuh"

namespace moe {

constexpr int kBsThreads = 11 * 32;
constexpr int kBsSfWarp0 = 0, kBsEpiWarp0 = 4, kBsProducerWarp = 8, kBsMmaWarp = 9;
constexpr int kBsProducerWarp2 = 10;
constexpr uint32_t kBsTmemCols = 512;
constexpr int kBsSfCols = 48;  // per stage: A scales 2 x 16 columns, B scales 16
constexpr int kSwigluThreads = 384;  // swiglu_terms_kernel: 96 quads of lanes
// above this many rows the 128-thread kernel (more rows in flight per SM) runs
constexpr int kSwigluQuadMaxRows = 512;

template <int NT>
struct BsGeom {
  static constexpr int BN = kTerms * NT;  // B rows = MMA N
  static constexpr int A0 = 0;
  static constexpr int A1 = kRowsHalf * kRowBytes;             // 16 KB
  static constexpr int S0 = 2 * kRowsHalf * kRowBytes;         // 32 KB
  static constexpr int S1 = S0 + kRowsHalf * 16;
  static constexpr int B = S0 + 2 * kRowsHalf * 16;            // 36 KB, 1024-aligned
  static constexpr int RAW = B + BN * kRowBytes;
  static constexpr int BYTES = (RAW + 1023) / 1024 * 1024;
  static constexpr int STAGES_RAW = (212 * 1024) / BYTES;  // + ~10 KB static
  static constexpr int STAGES = STAGES_RAW > 8 ? 8 : STAGES_RAW;
  static constexpr int SMEM = STAGES * BYTES + 1024;
  // tensor memory: accumulators D[db][mat] (BN columns each; ND items in
  // flight between the MMA and the epilogue), then per-stage scales
  static constexpr int ND = (NT == 8) ? 3 : 2;
  static constexpr uint32_t D_COLS = 2 * ND * BN;
  static_assert(D_COLS + STAGES * kBsSfCols <= kBsTmemCols, "tensor memory budget");
  static_assert(B % 1024 == 0, "B tile must start a swizzle atom");
};

// Instruction descriptor of kind::mxf4nvf4: A and B E2M1 (format 1), UE4M3
// scales (bit 23 clear), both operands K-major, f32 accumulator.
__host__ __device__ constexpr uint32_t tc_idesc_mxf4nvf4(int M, int N) {
  return (1u << 7) | (1u << 10) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

__device__ __forceinline__ void tc_mma_mxf4nvf4(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                                uint32_t idesc, uint32_t sfa_tmem,
                                                uint32_t sfb_tmem, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.u32 p, %6, 0;\n"
      " tcgen05.mma.cta_group::1.kind::mxf4nvf4.block_scale.scale_vec::4X"
      " [%0], %1, %2, %3, [%4], [%5], p;\n}\n" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(sfa_tmem), "r"(sfb_tmem), "r"(accumulate)
      : "memory");
}

__device__ __forceinline__ uint4 ldg_nc_v4(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

template <int NT, int PHASE, bool DET>
__global__ void __launch_bounds__(kBsThreads, 1)
    ffn_bs_kernel(const __grid_constant__ CUtensorMap tmA0,
                  const __grid_constant__ CUtensorMap tmA1,
                  const __grid_constant__ CUtensorMap tmS0,
                  const __grid_constant__ CUtensorMap tmS1,
                  const __grid_constant__ CUtensorMap tmB, const FfnParams p) {
  using G = BsGeom<NT>;
  constexpr int BN = G::BN;
  constexpr int S = G::STAGES;
  constexpr int KEL = 256;  // K per stage

  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);

  __shared__ __align__(8) uint64_t full_bar[S];
  __shared__ __align__(8) uint64_t empty_bar[S];
  __shared__ __align__(8) uint64_t sf_bar[S];
  __shared__ __align__(8) uint64_t dfull_bar[G::ND];
  __shared__ __align__(8) uint64_t dempty_bar[G::ND];
  __shared__ __align__(8) uint64_t final_bar;
  __shared__ PlanSmem pl;
  __shared__ int s_tok[NT];
  __shared__ uint32_t s_tmem;
  __shared__ volatile int s_abort;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    s_abort = 0;
    for (int i = 0; i < S; ++i) {
      mbar_init(&full_bar[i], 1);
      mbar_init(&empty_bar[i], 1);
      mbar_init(&sf_bar[i], 4);
    }
    for (int i = 0; i < G::ND; ++i) {
      mbar_init(&dfull_bar[i], 1);
      mbar_init(&dempty_bar[i], 4);
    }
    mbar_init(&final_bar, 1);
    fence_mbar_init();
  }
  if (warp == kBsMmaWarp) {
    tmem_alloc(&s_tmem, kBsTmemCols);
    tmem_relinquish();
  }
  // Launched as a programmatic dependent: everything above overlapped the
  // previous kernel.  The gate/up step waits for it here.  The down step's
  // plan and weights do not depend on it (the counts were written by a kernel
  // that completed before the gate/up step started), so its first weight
  // copies start at once and only the roles that read the SwiGLU output wait
  // (griddepcontrol.wait) before their first read of it.
  constexpr bool early = (PHASE == 2);
  if (!early) pdl_wait();
  pdl_launch_dependents();
  if (warp == 0) build_plan(p.counts, p.E, NT, pl, lane);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s_tmem;

  const int N = (PHASE == 1) ? p.I : p.H;  // rows of one expert matrix
  const int K = (PHASE == 1) ? p.H : p.I;  // contraction length
  const int rtiles = (PHASE == 1) ? p.I / kRowsHalf : p.H / (2 * kRowsHalf);
  const int KB = K / KEL;
  // this CTA's share of the stages of all items (< 2^31 for every supported
  // shape), divided by cost (items of many tokens cost more per stage when
  // their rows come token by token)
  const int cost_a = stage_cost_base((PHASE == 1) && !p.b_compact);
  int s_begin = cost_split_stage(pl, rtiles, KB, NT, cost_a, kTokenCost, blockIdx.x, gridDim.x);
  int s_end = cost_split_stage(pl, rtiles, KB, NT, cost_a, kTokenCost, blockIdx.x + 1, gridDim.x);
  if (DET) {
    s_begin = (int)item_boundary(s_begin, KB);
    s_end = (int)item_boundary(s_end, KB);
  }
  const int nst = s_end - s_begin;
  const uint32_t timeout_bit = (PHASE == 1) ? kStatusTimeoutGateUp : kStatusTimeoutDown;
  // B rows: per token (phase 1, tokens scattered) or one box per chunk
  const bool btok = (PHASE == 1) && !p.b_compact;
  constexpr int kTeardown = 9 * 32;  // scale writers, epilogue and MMA warps

  // ================================================================ producer
  if (warp == kBsProducerWarp || warp == kBsProducerWarp2) {
    const bool lead = (warp == kBsProducerWarp);
    if (!lead && early) pdl_wait();  // the activation rows are the SwiGLU output
    if (lane == 0 && nst > 0) {
      tma_prefetch_desc(&tmA0);
      tma_prefetch_desc(&tmA1);
      tma_prefetch_desc(&tmS0);
      tma_prefetch_desc(&tmS1);
      tma_prefetch_desc(&tmB);
      // weights stream through L2 once (evict first), except the tile of an
      // item whose expert has tokens in a later chunk: that chunk's item,
      // next in the order, reads the same tile again (evict last)
      const uint64_t pol_w = policy_evict_first();
      const uint64_t pol_keep = policy_evict_last();
      uint64_t pol_item = pol_w;
      const uint64_t pol_a = policy_evict_last();
      int cur_item = -1;
      ItemInfo inf{};
      int issued = 0;
      for (StageCursor<S> c(s_begin, KB); issued < nst; ++issued, c.next()) {
        const int it = c.it;
        const int kb = c.kb;
        if (it != cur_item) {
          cur_item = it;
          inf = decode_item(it, rtiles, pl, p, NT);
          pol_item = (inf.arow0 + NT < pl.aoff[inf.slot] + pl.acnt[inf.slot]) ? pol_keep : pol_w;
          if (!lead && btok)
            for (int j = 0; j < inf.nvalid; ++j) s_tok[j] = __ldg(p.sorted + inf.lrow0 + j) / p.k;
        }
        const int slot = c.slot;
        if (!mbar_wait_bounded(&empty_bar[slot], c.par ^ 1u, p.wait_ns, &s_abort)) {
          set_status(p.status, timeout_bit);
          s_abort = 1;
          break;
        }
        if (p.test_stall && issued == 0) continue;  // test hook: this stage never arrives
        unsigned char* st = smem + (size_t)slot * G::BYTES;
        uint32_t bytes = 2u * kRowsHalf * kRowBytes + 2u * kRowsHalf * 16u;
        bytes += btok ? (uint32_t)inf.nvalid * kTerms * kRowBytes
                                : (uint32_t)BN * kRowBytes;
        // the second producer's copies may land before this arms the barrier:
        // the transaction count then dips below zero, and the phase still
        // cannot complete before the arrival below
        if (lead) mbar_arrive_expect_tx(&full_bar[slot], bytes);
        int rowA0, rowA1;
        if (PHASE == 1) {
          rowA0 = inf.e * N + inf.rt * kRowsHalf;
          rowA1 = rowA0;
        } else {
          rowA0 = inf.e * N + inf.rt * 2 * kRowsHalf;
          rowA1 = rowA0 + kRowsHalf;
        }
        // Box A0 (and its scales) always come from the lead producer, box A1
        // from the second one - except for the down step's first ring of
        // stages, whose weights the lead copies before the SwiGLU kernel ends.
        const bool a1_lead = early && issued < S;
        if (lead) {
          tma_load_2d(st + G::A0, &tmA0, &full_bar[slot], kb * kRowBytes, rowA0, pol_item);
          tma_load_2d(st + G::S0, &tmS0, &full_bar[slot], kb * 16, rowA0, pol_item);
          if (a1_lead) {
            tma_load_2d(st + G::A1, &tmA1, &full_bar[slot], kb * kRowBytes, rowA1, pol_item);
            tma_load_2d(st + G::S1, &tmS1, &full_bar[slot], kb * 16, rowA1, pol_item);
          }
          continue;
        }
        if (!a1_lead) {
          tma_load_2d(st + G::A1, &tmA1, &full_bar[slot], kb * kRowBytes, rowA1, pol_item);
          tma_load_2d(st + G::S1, &tmS1, &full_bar[slot], kb * 16, rowA1, pol_item);
        }
        // activation terms: token j's four rows land at B rows 4j..4j+3
        if (btok) {
          for (int j = 0; j < inf.nvalid; ++j)
            tma_load_2d(st + G::B + j * kTerms * kRowBytes, &tmB, &full_bar[slot],
                        kb * kRowBytes, s_tok[j] * kTerms, pol_a);
        } else {
          tma_load_2d(st + G::B, &tmB, &full_bar[slot], kb * kRowBytes, inf.arow0 * kTerms,
                      pol_a);
        }
      }
      // Let every copy this CTA issued land before the CTA exits (the
      // barriers complete only when both producers' copies have landed).
      if (!lead) return;
      const int first = issued > S ? issued - S : 0;
      for (int j = first; j < issued; ++j) {
        if (p.test_stall && j == 0) continue;
        mbar_wait_bounded(&full_bar[j % S], (uint32_t)((j / S) & 1), p.wait_ns, nullptr);
      }
    }
    return;
  }

  // ================================================================ MMA issuer
  if (warp == kBsMmaWarp) {
    if (lane == 0) {
      constexpr uint32_t idesc = tc_idesc_mxf4nvf4(128, BN);
      int nitem = 0;
      bool ok = true;
      StageCursor<S> c(s_begin, KB);
      for (int i = 0; i < nst && ok; ++i, c.next()) {
        const int kb = c.kb;
        const bool first = (i == 0) || (kb == 0);
        const bool last = (i + 1 == nst) || (kb + 1 == KB);
        const int slot = c.slot;
        const int db = nitem % G::ND;
        if (first)
          ok = mbar_wait_bounded(&dempty_bar[db], ((uint32_t)(nitem / G::ND) & 1u) ^ 1u,
                                 p.wait_ns, &s_abort);
        ok = ok && mbar_wait_bounded(&full_bar[slot], c.par, p.wait_ns, &s_abort) &&
             mbar_wait_bounded(&sf_bar[slot], c.par, p.wait_ns, &s_abort);
        if (!ok) break;
        tc_fence_after();
        const uint32_t st = smem_u32(smem + (size_t)slot * G::BYTES);
        const uint32_t sfc = tmem + G::D_COLS + (uint32_t)slot * kBsSfCols;
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {
          const uint64_t bdesc = tc_desc_sw128(st + G::B + 32 * kk);
          const uint32_t acc = (first && kk == 0) ? 0u : 1u;
          tc_mma_mxf4nvf4(tmem + (uint32_t)(2 * db) * BN, tc_desc_sw128(st + G::A0 + 32 * kk),
                          bdesc, idesc, sfc + 4 * kk, sfc + 32 + 4 * kk, acc);
          tc_mma_mxf4nvf4(tmem + (uint32_t)(2 * db + 1) * BN,
                          tc_desc_sw128(st + G::A1 + 32 * kk), bdesc, idesc, sfc + 16 + 4 * kk,
                          sfc + 32 + 4 * kk, acc);
        }
        tc_commit(&empty_bar[slot]);
        if (last) {
          tc_commit(&dfull_bar[db]);
          ++nitem;
        }
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
    tmem_dealloc(tmem, kBsTmemCols);
    return;
  }

  // ================================================================ scale writers
  if (warp < kBsEpiWarp0) {
    if (early) pdl_wait();  // the B scales are the SwiGLU output
    const int quad = warp - kBsSfWarp0;
    const uint32_t lane_addr = (uint32_t)(quad * 32) << 16;
    const int bstride = K / 16;  // bytes per B-scale row
    int cur_item = -1;
    ItemInfo inf{};
    int grow[2] = {-1, -1};  // global B-scale rows of B rows lane and lane + 32
    // B scales (16 bytes per row: 4 MMAs x 4 blocks) are loaded one stage
    // ahead, by a second cursor
    StageCursor<S> cn(s_begin, KB);
    auto load_bsf = [&](uint4 (&out)[2]) {
      if (cn.it != cur_item) {
        cur_item = cn.it;
        inf = decode_item(cn.it, rtiles, pl, p, NT);
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int n = lane + 32 * h;
          const int j = n / kTerms;
          grow[h] = -1;
          if (n < BN && j < inf.nvalid) {
            const int base = btok ? __ldg(p.sorted + inf.lrow0 + j) / p.k : inf.arow0 + j;
            grow[h] = base * kTerms + n % kTerms;
          }
        }
      }
#pragma unroll
      for (int h = 0; h < 2; ++h)
        out[h] = (grow[h] >= 0) ? ldg_nc_v4(p.bsf + (size_t)grow[h] * bstride + 16 * cn.kb)
                                : make_uint4(0u, 0u, 0u, 0u);
      cn.next();
    };
    uint4 bsf[2], bnext[2];
    if (nst > 0) load_bsf(bsf);
    StageCursor<S> c(s_begin, KB);
    for (int i = 0; i < nst; ++i, c.next()) {
      if (i + 1 < nst) load_bsf(bnext);
      const int slot = c.slot;
      // the MMAs that read this slot's scales last round are done, and this
      // round's A scales have landed
      if (!mbar_wait_bounded(&empty_bar[slot], c.par ^ 1u, p.wait_ns, &s_abort) ||
          !mbar_wait_bounded(&full_bar[slot], c.par, p.wait_ns, &s_abort)) {
        set_status(p.status, timeout_bit);
        s_abort = 1;
        break;
      }
      tc_fence_after();
      const uint32_t st = smem_u32(smem + (size_t)slot * G::BYTES);
      const uint32_t sfc = tmem + lane_addr + G::D_COLS + (uint32_t)slot * kBsSfCols;
#pragma unroll
      for (int mat = 0; mat < 2; ++mat) {
        // rows lane + 32*r1 of this matrix's 128-row scale box
        uint4 v[4];
#pragma unroll
        for (int r1 = 0; r1 < 4; ++r1)
          v[r1] = lds128(st + (mat == 0 ? G::S0 : G::S1) + (lane + 32 * r1) * 16);
        uint32_t c[16];
#pragma unroll
        for (int r1 = 0; r1 < 4; ++r1) {
          c[0 + r1] = v[r1].x;   // MMA 0 (K 0-63 of the stage)
          c[4 + r1] = v[r1].y;   // MMA 1
          c[8 + r1] = v[r1].z;   // MMA 2
          c[12 + r1] = v[r1].w;  // MMA 3
        }
        tmem_st16(sfc + 16 * mat, c);
      }
      {
        uint32_t c[16];
        const uint32_t b0[4] = {bsf[0].x, bsf[0].y, bsf[0].z, bsf[0].w};
        const uint32_t b1[4] = {bsf[1].x, bsf[1].y, bsf[1].z, bsf[1].w};
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {
          c[4 * kk + 0] = b0[kk];
          c[4 * kk + 1] = (BN > 32) ? b1[kk] : 0u;
          c[4 * kk + 2] = 0u;
          c[4 * kk + 3] = 0u;
        }
        tmem_st16(sfc + 32, c);
      }
      tmem_st_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sf_bar[slot]);
      bsf[0] = bnext[0];
      bsf[1] = bnext[1];
    }
    tc_fence_before();
    asm volatile("bar.sync 2, %0;" ::"n"(kTeardown) : "memory");
    return;
  }

  // ================================================================ epilogue
  // Warp 4+q reads TMEM lanes 32q..32q+31: row 32q+lane of both matrices.
  {
    if (early) pdl_wait();  // the row scales are the SwiGLU output
    const int quad = warp - kBsEpiWarp0;
    const int row = quad * 32 + lane;
    const uint32_t lane_addr = (uint32_t)(quad * 32) << 16;
    bool dead = false;
    int nitem = 0;
    if (nst > 0) {
      const int it0 = s_begin / KB, it1 = (s_end - 1) / KB;
      for (int it = it0; it <= it1 && !dead; ++it, ++nitem) {
        const ItemInfo inf = decode_item(it, rtiles, pl, p, NT);
        const int db = nitem % G::ND;
        if (!mbar_wait_bounded(&dfull_bar[db], (uint32_t)(nitem / G::ND) & 1u, p.wait_ns,
                               &s_abort)) {
          set_status(p.status, timeout_bit);
          s_abort = 1;
          dead = true;
          break;
        }
        tc_fence_after();
        // the four terms of token j are accumulator columns 4j..4j+3
        float acc[2][NT];
#pragma unroll
        for (int mat = 0; mat < 2; ++mat) {
          const uint32_t d_t = tmem + lane_addr + (uint32_t)(2 * db + mat) * BN;
#pragma unroll
          for (int c0 = 0; c0 < BN; c0 += 16) {
            uint32_t v[16];
            tmem_ld16(d_t + c0, v);
            tmem_ld_wait();
#pragma unroll
            for (int q = 0; q < 4; ++q)
              acc[mat][c0 / 4 + q] = (__uint_as_float(v[4 * q]) + __uint_as_float(v[4 * q + 1])) +
                                     (__uint_as_float(v[4 * q + 2]) + __uint_as_float(v[4 * q + 3]));
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&dempty_bar[db]);
        const float ts0 = __ldg(p.ts0 + inf.e), ts1 = __ldg(p.ts1 + inf.e);
#pragma unroll
        for (int j = 0; j < NT; ++j) {
          if (j >= inf.nvalid) continue;
          const int arow = inf.arow0 + j;
          const int a = __ldg(p.sorted + inf.lrow0 + j);
          if (PHASE == 1) {
            const float sc = __ldg(p.xinv + a / p.k);
            const int f = inf.rt * kRowsHalf + row;
            float* gr = p.gu + (size_t)arow * 2 * p.I + f;
            put_f32(gr, acc[0][j] * sc * ts0, DET);
            put_f32(gr + p.I, acc[1][j] * sc * ts1, DET);
          } else {
            const float sc = __ldcg(p.xinv + arow);  // hinv, written by the previous kernel
            const int hrow = inf.rt * 2 * kRowsHalf + row;
            if (p.fused) {
              const float gw = __ldg(p.gates + a) * sc;
              float* orow = p.oacc + (size_t)(a / p.k) * p.H + hrow;
              red_add_f32(orow, gw * acc[0][j] * ts0);
              red_add_f32(orow + kRowsHalf, gw * acc[1][j] * ts1);
            } else {
              float* yrow = p.y_perm + (size_t)(DET ? a : arow) * p.H + hrow;
              put_f32(yrow, acc[0][j] * sc * ts0, DET);
              put_f32(yrow + kRowsHalf, acc[1][j] * sc * ts1, DET);
            }
          }
        }
      }
    }
    tc_fence_before();
    asm volatile("bar.sync 2, %0;" ::"n"(kTeardown) : "memory");
  }
}

// SwiGLU of every assignment row into four NVFP4 terms (the B operand of the
// down step): h = silu(g) * u from the fp32 gate|up accumulators, a per-row
// power of two, then the terms of each 16-column block by a quad of lanes
// (four columns each).  One CTA per row, one pass over the row when I <= 1536
// (96 blocks); every load of the row is issued before the first is used.
static __global__ void __launch_bounds__(kSwigluThreads, 2) swiglu_terms_kernel(const FfnParams p, int rows) {
  constexpr int BPP = kSwigluThreads / 4;          // blocks per pass
  constexpr int PMAX = (8192 / 16 + BPP - 1) / BPP;  // passes for I <= 8192
  __shared__ float s_max[kSwigluThreads / 32];
  // the down step may launch now: what it does before its own wait (plan,
  // weight copies) does not read this kernel's output
  pdl_launch_dependents();
  pdl_wait();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int lq = threadIdx.x & 3, quad = threadIdx.x >> 2;
  const int nb = p.I / 16;
  const int np = (nb + BPP - 1) / BPP;
  for (int row = blockIdx.x; row < rows; row += gridDim.x) {
    const float* g = p.gu + (size_t)row * 2 * p.I;
    const float* u = g + p.I;
    float h[PMAX][4];
    float amax = 0.f;
    float4 gv[PMAX], uv[PMAX];
#pragma unroll
    for (int ps = 0; ps < PMAX; ++ps) {
      const int b = quad + BPP * ps;
      gv[ps] = uv[ps] = make_float4(0.f, 0.f, 0.f, 0.f);
      if (ps < np && b < nb) {
        gv[ps] = __ldcg(reinterpret_cast<const float4*>(g + 16 * b + 4 * lq));
        uv[ps] = __ldcg(reinterpret_cast<const float4*>(u + 16 * b + 4 * lq));
      }
    }
#pragma unroll
    for (int ps = 0; ps < PMAX; ++ps) {
      if (ps < np) {  // the same on every thread
        h[ps][0] = gv[ps].x / (1.f + expf(-gv[ps].x)) * uv[ps].x;
        h[ps][1] = gv[ps].y / (1.f + expf(-gv[ps].y)) * uv[ps].y;
        h[ps][2] = gv[ps].z / (1.f + expf(-gv[ps].z)) * uv[ps].z;
        h[ps][3] = gv[ps].w / (1.f + expf(-gv[ps].w)) * uv[ps].w;
#pragma unroll
        for (int i = 0; i < 4; ++i) amax = fmaxf(amax, fabsf(h[ps][i]));
      }
    }
    amax = warp_max(amax);
    if (lane == 0) s_max[warp] = amax;
    __syncthreads();
    amax = s_max[0];
#pragma unroll
    for (int i = 1; i < kSwigluThreads / 32; ++i) amax = fmaxf(amax, s_max[i]);
    const float sc = pow2_scale_terms(amax);
#pragma unroll
    for (int ps = 0; ps < PMAX; ++ps) {
      if (ps < np) {  // the same on every thread
        const int b = quad + BPP * ps;
        float r[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) r[i] = h[ps][i] * sc;
        uint32_t part[kTerms], sf[kTerms];
        encode_terms16_quad(r, part, sf);
        store_terms16_quad(part, sf, b < nb, p.hq, p.hsf, (size_t)row * kTerms, p.I, b);
      }
    }
    if (threadIdx.x == 0) p.hinv[row] = 1.f / sc;
    __syncthreads();  // s_max is reused by the next row
  }
}

// The same SwiGLU with one thread per 16-column block (encode_terms16 run
// serially by that thread) in 128-thread CTAs, G blocks per thread (I <= 2048
// G), for batches with many rows.  With one block per thread the next row's
// gate|up values load while this row is encoded (with more, the registers
// that would take cost more CTAs per SM than the overlap gains).  The row
// maximum meets in a double-buffered shared array, one barrier per row.  The
// first NTERM terms are written (the prefill engine reads three); the codes
// are the quad kernel's.
template <int G, int NTERM>
static __global__ void __launch_bounds__(128) swiglu_terms_rows_kernel(const FfnParams p, int rows) {
  __shared__ float s_max[2][4];
  // the down step may launch now: what it does before its own wait (plan,
  // weight copies) does not read this kernel's output
  pdl_launch_dependents();
  pdl_wait();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int nb = p.I / 16;
  constexpr bool kAhead = (G == 1);
  float4 ng[4], nu[4];  // kAhead: the next row's gate and up values of this thread's block
  auto load_ahead = [&](int row) {
    const float* g = p.gu + (size_t)row * 2 * p.I + 16 * threadIdx.x;
    if (row < rows && (int)threadIdx.x < nb) {
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        ng[i] = __ldcg(reinterpret_cast<const float4*>(g + 4 * i));
        nu[i] = __ldcg(reinterpret_cast<const float4*>(g + p.I + 4 * i));
      }
    }
  };
  auto silu4 = [](float4 gv, float4 uv, float* h) {
    h[0] = gv.x / (1.f + expf(-gv.x)) * uv.x;
    h[1] = gv.y / (1.f + expf(-gv.y)) * uv.y;
    h[2] = gv.z / (1.f + expf(-gv.z)) * uv.z;
    h[3] = gv.w / (1.f + expf(-gv.w)) * uv.w;
  };
  if (kAhead) load_ahead(blockIdx.x);
  int par = 0;
  for (int row = blockIdx.x; row < rows; row += gridDim.x, par ^= 1) {
    const float* g = p.gu + (size_t)row * 2 * p.I;
    float h[G][16];
    float amax = 0.f;
#pragma unroll
    for (int q = 0; q < G; ++q) {
      const int b = threadIdx.x + 128 * q;
      if (b < nb) {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          if (kAhead) {
            silu4(ng[i], nu[i], &h[q][4 * i]);
          } else {
            silu4(__ldcg(reinterpret_cast<const float4*>(g + 16 * b + 4 * i)),
                  __ldcg(reinterpret_cast<const float4*>(g + p.I + 16 * b + 4 * i)), &h[q][4 * i]);
          }
        }
#pragma unroll
        for (int i = 0; i < 16; ++i) amax = fmaxf(amax, fabsf(h[q][i]));
      }
    }
    if (kAhead) load_ahead(row + gridDim.x);
    amax = warp_max(amax);
    if (lane == 0) s_max[par][warp] = amax;
    __syncthreads();  // a warp reaches the next row's barrier only after this row's reads
    amax = fmaxf(fmaxf(s_max[par][0], s_max[par][1]), fmaxf(s_max[par][2], s_max[par][3]));
    const float sc = pow2_scale_terms(amax);
#pragma unroll
    for (int q = 0; q < G; ++q) {
      const int b = threadIdx.x + 128 * q;
      if (b < nb) {
#pragma unroll
        for (int i = 0; i < 16; ++i) h[q][i] *= sc;
        uint2 codes[kTerms];
        uint32_t sf[kTerms];
        encode_terms16<NTERM>(h[q], codes, sf);
        store_terms16<NTERM>(codes, sf, p.hq, p.hsf, (size_t)row * kTerms, p.I, b);
      }
    }
    if (threadIdx.x == 0) p.hinv[row] = 1.f / sc;
  }
}

}  // namespace moe
