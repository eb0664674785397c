// FP8 expert FFN on the tensor cores: tcgen05.mma kind::f8f6f4, E4M3 weights
// as stored times E4M3 activation terms, fp32 accumulation in tensor memory.
//
// Work decomposition as in ffn.cuh / ffn_bs.cuh: a persistent grid, stream-K
// over the K-stages of all (active expert, <=NT-token chunk, row tile) items;
// with 32-token chunks, the stages of an expert with several chunks in slab
// order (SlabCursor).
// A stage is 128 K, which is exactly one column of the weights' 128x128 fp32
// block scales.  The MMA has no block scaling for this format pair, so every
// stage accumulates into its own slot of a ring of tensor-memory accumulators
// and the epilogue warps multiply it by the stage's two block scales while
// adding it into registers; an item's sums are flushed with red.add at its
// last stage in this CTA, or at the end of its run in a slab.  The activations arrive as two E4M3 terms per
// token (act_terms.cuh): B rows 2j, 2j+1 of token j; the epilogue adds the
// two columns.
//
// Roles (224 threads; 352 in the down step with 32-token chunks):
//   warps 0-3  epilogue: warp w reads TMEM lanes 32w..32w+31 (rows of the tile)
//   warps 4,6  TMA producers (one thread each): warp 4 arms each stage's
//              barrier and copies box A0, warp 6 box A1 and the activation rows
//   warp 5     MMA issuer (one thread); allocates and frees tensor memory
//   warps 7-10 (down step, 32-token chunks) a second epilogue group: warp w
//              reads lanes 32(w%4).. like warp w%4, for the chunk's tokens
//              16-31, warps 0-3 then taking tokens 0-15
// Every wait is bounded (p.wait_ns); an expired wait sets the status word and
// the kernel winds down, freeing its tensor memory.
#pragma once

#include <type_traits>

#include "act_terms.cuh"
#include "ffn.cuh"

namespace moe {

constexpr int kF8ProducerWarp = 4, kF8MmaWarp = 5, kF8ProducerWarp2 = 6;

template <int NT, int PHASE>
struct F8Geom {
  // epilogue warps: one per TMEM lane quadrant, or two in the down step with
  // 32-token chunks, each adding half of the chunk's token columns.  Measured
  // on the 480B-shaped layer with Zipf routing: the down step at T = 256
  // 400 -> 380 us, at T = 128 267 -> 253 us; the gate/up step was no faster
  // (696 -> 708 us at T = 256), so it keeps four.  (64-token chunks with
  // eight warps of 32 tokens each and a 2-deep accumulator ring were slower
  // in both steps.)
  static constexpr int EPI = (NT >= 32 && PHASE == 2) ? 8 : 4;
  static constexpr int NTH = NT * 4 / EPI;  // tokens per epilogue thread
  static constexpr int THREADS = (EPI + 3) * 32;
  static constexpr int BN = kF8Terms * NT;  // B rows = MMA N
  static constexpr int A0 = 0;
  static constexpr int A1 = kRowsHalf * kRowBytes;      // 16 KB
  static constexpr int B = 2 * kRowsHalf * kRowBytes;   // 32 KB, 1024-aligned
  static constexpr int RAW = B + BN * kRowBytes;
  static constexpr int BYTES = (RAW + 1023) / 1024 * 1024;
  static constexpr int STAGES_RAW = (212 * 1024) / BYTES;  // + ~9 KB static
  static constexpr int STAGES = STAGES_RAW > 8 ? 8 : STAGES_RAW;
  static constexpr int SMEM = STAGES * BYTES + 1024;
  static constexpr int DR = 4;  // accumulator ring (stages)
  static constexpr uint32_t TMEM_COLS = (DR * 2 * BN <= 256) ? 256u : 512u;
  static_assert(DR * 2 * BN <= (int)TMEM_COLS, "tensor memory budget");
  static_assert(BN % 16 == 0 && BN <= 256, "MMA N");
};

// Instruction descriptor of kind::f8f6f4: f32 D, E4M3 A and B, K-major.
__host__ __device__ constexpr uint32_t tc_idesc_e4m3(int M, int N) {
  return (1u << 4) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

__device__ __forceinline__ void tc_mma_f8(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                          uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.u32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

template <int NT, int PHASE, bool DET>
__global__ void __launch_bounds__(F8Geom<NT, PHASE>::THREADS, 1)
    ffn_f8_kernel(const __grid_constant__ CUtensorMap tmA0,
                  const __grid_constant__ CUtensorMap tmA1,
                  const __grid_constant__ CUtensorMap tmB, const FfnParams p) {
  using G = F8Geom<NT, PHASE>;
  constexpr int BN = G::BN;
  constexpr int S = G::STAGES;
  constexpr int DR = G::DR;
  constexpr int KEL = 128;  // K per stage

  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);

  __shared__ __align__(8) uint64_t full_bar[S];
  __shared__ __align__(8) uint64_t empty_bar[S];
  __shared__ __align__(8) uint64_t dfull_bar[DR];
  __shared__ __align__(8) uint64_t dempty_bar[DR];
  __shared__ __align__(8) uint64_t final_bar;
  __shared__ PlanSmem pl;
  __shared__ int s_tok[NT];
  __shared__ uint32_t s_tmem;
  __shared__ volatile int s_abort;
  __shared__ __align__(8) UnitRing s_units;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    s_abort = 0;
    for (int i = 0; i < S; ++i) {
      mbar_init(&full_bar[i], 1);
      mbar_init(&empty_bar[i], 1);
    }
    for (int i = 0; i < DR; ++i) {
      mbar_init(&dfull_bar[i], 1);
      mbar_init(&dempty_bar[i], G::EPI);
    }
    mbar_init(&final_bar, 1);
    // readers of each unit: second producer, MMA issuer, the epilogue warps
    for (int i = 0; i < kUnitRing; ++i) {
      mbar_init(&s_units.full[i], 1);
      mbar_init(&s_units.empty[i], 2 + G::EPI);
    }
    fence_mbar_init();
  }
  if (warp == kF8MmaWarp) {
    tmem_alloc(&s_tmem, G::TMEM_COLS);
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
  // Stages of all items (< 2^31 for every supported shape), divided between
  // the CTAs by cost (items of many tokens cost more per stage when their rows
  // come token by token).  With 8-token chunks and enough stages per CTA for
  // the units to be small, the CTAs divide only the first kStaticNum /
  // kStaticDen of the cost and the stages from s_dyn on are the shared tail
  // (measured: it evens out the CTAs' finishing times on the 480B-shaped layer
  // at 64 tokens; with wider chunks or little work per CTA the static split
  // alone is faster).
  const int total = pl.cpre[pl.nA] * rtiles * KB;
  const bool tail = (NT == 8) && total >= kTailMinStages * (int)gridDim.x;
  const int snum = tail ? kStaticNum : 1, sden = tail ? kStaticDen : 1;
  const int cost_a = stage_cost_base((PHASE == 1) && !p.b_compact);
  const long long den = (long long)gridDim.x * sden;
  int s_begin = cost_split_stage(pl, rtiles, KB, NT, cost_a, kTokenCost,
                                 (long long)blockIdx.x * snum, den);
  int s_end = cost_split_stage(pl, rtiles, KB, NT, cost_a, kTokenCost,
                               (long long)(blockIdx.x + 1) * snum, den);
  if (DET) {
    s_begin = (int)item_boundary(s_begin, KB);
    s_end = (int)item_boundary(s_end, KB);
  }
  int s_dyn = tail ? cost_split_stage(pl, rtiles, KB, NT, cost_a, kTokenCost, snum, sden)
                   : total;
  if (DET) s_dyn = (int)item_boundary(s_dyn, KB);  // the last CTA's share ends here too
  const int us = DET ? KB : kUnitStages;  // stages per unit of the tail
  // Slab order for experts of several 32-token chunks; whole items in the
  // deterministic mode (every item summed by one CTA in K order) and with
  // narrower chunks: with 8-token chunks slabs gained nothing (Zipf routing
  // at T = 32: 486.5 -> 484.9 us) and the slab cursor cost the uniform
  // 480B-shaped layer at T = 64 1.4% of its gate/up time (703 -> 713 us).
  const int slab = DET ? 0 : p.slab;
  uint32_t* units = p.units + 2 * (PHASE - 1);
  const uint32_t timeout_bit = (PHASE == 1) ? kStatusTimeoutGateUp : kStatusTimeoutDown;
  // B rows: per token (phase 1, tokens scattered) or one box per chunk
  const bool btok = (PHASE == 1) && !p.b_compact;
  constexpr int kTeardown = (G::EPI + 1) * 32;  // epilogue and MMA warps

  // ================================================================ producers
  if (warp == kF8ProducerWarp || warp == kF8ProducerWarp2) {
    const bool lead = (warp == kF8ProducerWarp);
    if (!lead && early) pdl_wait();  // the activation rows are the SwiGLU output
    if (lane == 0) {
      tma_prefetch_desc(&tmA0);
      tma_prefetch_desc(&tmA1);
      if (!lead) tma_prefetch_desc(&tmB);
      // weights stream through L2 once (evict first), except the boxes of an
      // item whose expert has tokens in a later chunk: that chunk reads the
      // same boxes again (evict last), within the slab in slab order
      const uint64_t pol_w = policy_evict_first();
      const uint64_t pol_keep = policy_evict_last();
      uint64_t pol_item = pol_w;
      const uint64_t pol_a = policy_evict_last();
      int cur_item = -1;
      ItemInfo inf{};
      int issued = 0, uj = 0;
      bool ok = true;
      std::conditional_t<(NT >= 32), SlabCursor<S>, ItemCursor<S>> c(pl, rtiles, KB, slab,
                                                                      s_begin);
      // segments: this CTA's own share, then units of the shared tail (the
      // lead takes them and publishes them; the second producer reads them)
      for (int a = s_begin, b = s_end; ok;) {
        for (int s = a; s < b; ++s, ++issued, c.next()) {
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
            ok = false;
            break;
          }
          if (p.test_stall && issued == 0) continue;  // test hook: this stage never arrives
          unsigned char* st = smem + (size_t)slot * G::BYTES;
          int rowA0, rowA1;
          if (PHASE == 1) {
            rowA0 = inf.e * N + inf.rt * kRowsHalf;
            rowA1 = rowA0;
          } else {
            rowA0 = inf.e * N + inf.rt * 2 * kRowsHalf;
            rowA1 = rowA0 + kRowsHalf;
          }
          if (lead) {
            // the second producer's copies may land before this arms the
            // barrier: the transaction count then dips below zero, and the
            // phase still cannot complete before this arrival
            uint32_t bytes = 2u * kRowsHalf * kRowBytes;
            bytes += btok ? (uint32_t)inf.nvalid * kF8Terms * kRowBytes
                                    : (uint32_t)BN * kRowBytes;
            mbar_arrive_expect_tx(&full_bar[slot], bytes);
            // box A0 always; box A1 too for the down step's first ring of
            // stages, copied before the SwiGLU kernel ends
            tma_load_2d(st + G::A0, &tmA0, &full_bar[slot], kb * kRowBytes, rowA0, pol_item);
            if (early && issued < S)
              tma_load_2d(st + G::A1, &tmA1, &full_bar[slot], kb * kRowBytes, rowA1, pol_item);
            continue;
          }
          if (!(early && issued < S))
            tma_load_2d(st + G::A1, &tmA1, &full_bar[slot], kb * kRowBytes, rowA1, pol_item);
          // activation terms: token j's two rows land at B rows 2j, 2j+1
          if (btok) {
            for (int j = 0; j < inf.nvalid; ++j)
              tma_load_2d(st + G::B + j * kF8Terms * kRowBytes, &tmB, &full_bar[slot],
                          kb * kRowBytes, s_tok[j] * kF8Terms, pol_a);
          } else {
            tma_load_2d(st + G::B, &tmB, &full_bar[slot], kb * kRowBytes, inf.arow0 * kF8Terms,
                        pol_a);
          }
        }
        if (!ok || !tail) break;
        if (lead) {
          const int next = unit_take(units, s_dyn, total, us);
          if (!unit_push(s_units, uj++, next, p.wait_ns, &s_abort)) {
            ok = false;
            break;
          }
          if (next < 0) break;
          a = next;
          b = min(next + us, total);
        } else if (!unit_next(s_units, uj, total, us, a, b, false, p.wait_ns, &s_abort, &ok)) {
          break;
        }
        c.seek(a);
      }
      if (!ok) {
        set_status(p.status, timeout_bit);
        s_abort = 1;
      }
      if (lead) {
        if (tail) {
          if (!ok) unit_push(s_units, uj, -1, p.wait_ns, &s_abort);  // best effort
          unit_done(units);
        }
        // Let every copy land before the CTA exits (the barriers complete
        // only when both producers' copies have landed).
        const int first = issued > S ? issued - S : 0;
        for (int j = first; j < issued; ++j) {
          if (p.test_stall && j == 0) continue;
          mbar_wait_bounded(&full_bar[j % S], (uint32_t)((j / S) & 1), p.wait_ns, nullptr);
        }
      }
    }
    return;
  }

  // ================================================================ MMA issuer
  if (warp == kF8MmaWarp) {
    if (lane == 0) {
      constexpr uint32_t idesc = tc_idesc_e4m3(128, BN);
      bool ok = true;
      int uj = 0;
      StageCursor<S> c(s_begin, KB);
      StageCursor<DR> d(0, 1);  // accumulator ring position
      // every stage has its own accumulator: only the number of stages of
      // each segment matters here
      for (int a = s_begin, b = s_end; ok;) {
        for (int i = a; i < b && ok; ++i, c.next(), d.next()) {
          const int slot = c.slot;
          const int db = d.slot;
          ok = mbar_wait_bounded(&dempty_bar[db], d.par ^ 1u, p.wait_ns, &s_abort) &&
               mbar_wait_bounded(&full_bar[slot], c.par, p.wait_ns, &s_abort);
          if (!ok) break;
          tc_fence_after();
          const uint32_t st = smem_u32(smem + (size_t)slot * G::BYTES);
#pragma unroll
          for (int kk = 0; kk < 4; ++kk) {  // K = 32 per MMA
            const uint64_t bdesc = tc_desc_sw128(st + G::B + 32 * kk);
            tc_mma_f8(tmem + (uint32_t)(2 * db) * BN, tc_desc_sw128(st + G::A0 + 32 * kk), bdesc,
                      idesc, kk > 0 ? 1u : 0u);
            tc_mma_f8(tmem + (uint32_t)(2 * db + 1) * BN, tc_desc_sw128(st + G::A1 + 32 * kk),
                      bdesc, idesc, kk > 0 ? 1u : 0u);
          }
          tc_commit(&empty_bar[slot]);
          tc_commit(&dfull_bar[db]);
        }
        if (!ok || !tail || !unit_next(s_units, uj, total, us, a, b, false, p.wait_ns, &s_abort, &ok))
          break;
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
    tmem_dealloc(tmem, G::TMEM_COLS);
    return;
  }

  // ================================================================ epilogue
  // Warp w reads TMEM lanes 32q..32q+31, q = w % 4: row 32q+lane of both
  // boxes, for the chunk's tokens j0 .. j0 + NTH - 1.
  {
    if (early) pdl_wait();  // the row scales are the SwiGLU output
    constexpr int NTH = G::NTH;
    const int quad = warp & 3;
    const int j0 = (G::EPI > 4 && warp > kF8ProducerWarp2) ? NTH : 0;
    const int row = quad * 32 + lane;
    const uint32_t lane_addr = (uint32_t)(quad * 32) << 16;
    const int KB128 = K / 128;
    float acc0[NTH], acc1[NTH];
#pragma unroll
    for (int j = 0; j < NTH; ++j) acc0[j] = acc1[j] = 0.f;
    bool dead = false;
    ItemInfo inf{};
    // the block scales of a stage's two boxes
    auto scales = [&](const ItemInfo& f, int kb, float& b0, float& b1) {
      if (PHASE == 1) {
        const size_t tile = ((size_t)f.e * (N / 128) + f.rt) * KB128 + kb;
        b0 = __ldg(p.s0 + tile);
        b1 = __ldg(p.s1 + tile);
      } else {
        const size_t tile = ((size_t)f.e * (N / 128) + 2 * f.rt) * KB128 + kb;
        b0 = __ldg(p.s0 + tile);
        b1 = __ldg(p.s0 + tile + KB128);
      }
    };
    float bs0 = 0.f, bs1 = 0.f;
    // c: this stage (it, kb) and its accumulator ring slot; the stage after
    // it is found first (its block scales load while this stage's
    // accumulator is awaited), reading the shared-tail units as they come
    using Cursor = std::conditional_t<(NT >= 32), SlabCursor<DR>, ItemCursor<DR>>;
    Cursor c(pl, rtiles, KB, slab, s_begin);
    int cs = s_begin, cend = s_end, uj = 0;
    bool ok = true;
    bool have = cs < cend;
    if (!have && tail && unit_next(s_units, uj, total, us, cs, cend, true, p.wait_ns, &s_abort, &ok)) {
      c.seek(cs);
      have = true;
    }
    if (have) {
      inf = decode_item(c.it, rtiles, pl, p, NT);
      scales(inf, c.kb, bs0, bs1);
    }
    while (have && !dead) {
      // the next stage: the following one in this segment, or the first of
      // the next unit (a new accumulation even within the same item)
      int ns = cs + 1, nend = cend;
      Cursor nc = c;  // its accumulator slot is the next one in any case
      nc.next();
      bool have_next = ns < nend, jump = false;
      if (!have_next && tail) {
        have_next = unit_next(s_units, uj, total, us, ns, nend, true, p.wait_ns, &s_abort, &ok);
        jump = true;
        if (have_next) nc.seek(ns);
      }
      float nb0 = 0.f, nb1 = 0.f;
      ItemInfo ninf = inf;
      const bool closes = !have_next || jump || c.ends_run();
      if (have_next) {
        if (nc.it != c.it) ninf = decode_item(nc.it, rtiles, pl, p, NT);
        scales(ninf, nc.kb, nb0, nb1);
      }
      const int db = c.slot;
      if (!mbar_wait_bounded(&dfull_bar[db], c.par, p.wait_ns, &s_abort)) {
        set_status(p.status, timeout_bit);
        s_abort = 1;
        dead = true;
        break;
      }
      tc_fence_after();
      // token j's two terms are accumulator columns 2j and 2j+1; each box's
      // columns are read with all loads in flight before one wait
#pragma unroll
      for (int mat = 0; mat < 2; ++mat) {
        const uint32_t d_t = tmem + lane_addr + (uint32_t)((2 * db + mat) * BN + 2 * j0);
        const float bsc = mat == 0 ? bs0 : bs1;
        uint32_t v[2 * NTH];
#pragma unroll
        for (int c0 = 0; c0 < 2 * NTH; c0 += 16)
          tmem_ld16(d_t + c0, *reinterpret_cast<uint32_t(*)[16]>(v + c0));
        tmem_ld_wait();
#pragma unroll
        for (int j = 0; j < NTH; ++j) {
          const float t2 = __uint_as_float(v[2 * j]) + __uint_as_float(v[2 * j + 1]);
          if (mat == 0)
            acc0[j] = fmaf(bsc, t2, acc0[j]);
          else
            acc1[j] = fmaf(bsc, t2, acc1[j]);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&dempty_bar[db]);
      if (closes) {
#pragma unroll
        for (int jj = 0; jj < NTH; ++jj) {
          const int j = j0 + jj;
          if (j < inf.nvalid) {
            const int arow = inf.arow0 + j;
            const int a = __ldg(p.sorted + inf.lrow0 + j);
            if (PHASE == 1) {
              const float sc = __ldg(p.xinv + a / p.k);
              const int f = inf.rt * kRowsHalf + row;
              float* gr = p.gu + (size_t)arow * 2 * p.I + f;
              put_f32(gr, acc0[jj] * sc, DET);
              put_f32(gr + p.I, acc1[jj] * sc, DET);
            } else {
              const float sc = __ldcg(p.xinv + arow);  // hinv, written by the previous kernel
              const int hrow = inf.rt * 2 * kRowsHalf + row;
              if (p.fused) {
                const float gw = __ldg(p.gates + a) * sc;
                float* orow = p.oacc + (size_t)(a / p.k) * p.H + hrow;
                red_add_f32(orow, gw * acc0[jj]);
                red_add_f32(orow + kRowsHalf, gw * acc1[jj]);
              } else {
                float* yrow = p.y_perm + (size_t)(DET ? a : arow) * p.H + hrow;
                put_f32(yrow, acc0[jj] * sc, DET);
                put_f32(yrow + kRowsHalf, acc1[jj] * sc, DET);
              }
            }
          }
          acc0[jj] = acc1[jj] = 0.f;
        }
      }
      inf = ninf;
      bs0 = nb0;
      bs1 = nb1;
      c = nc;
      cs = ns;
      cend = nend;
      have = have_next;
    }
    if (!ok) {
      set_status(p.status, timeout_bit);
      s_abort = 1;
    }
    tc_fence_before();
    asm volatile("bar.sync 2, %0;" ::"n"(kTeardown) : "memory");
  }
}

// SwiGLU of every assignment row into two E4M3 terms (the B operand of the
// FP8 engine's down step): h = silu(g) * u from the fp32 gate|up
// accumulators, a per-row power of two, then hi/lo per 8 columns.  One CTA
// per row; each thread owns up to 8 groups of 8 columns (I <= 8192).
__global__ void __launch_bounds__(128) swiglu_e4m3_kernel(const FfnParams p, int rows) {
  constexpr int G = 8;
  __shared__ float s_max[4];
  // the down step may launch now: what it does before its own wait (plan,
  // weight copies) does not read this kernel's output
  pdl_launch_dependents();
  pdl_wait();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int n8 = p.I / 8;
  for (int row = blockIdx.x; row < rows; row += gridDim.x) {
    const float* g = p.gu + (size_t)row * 2 * p.I;
    const float* u = g + p.I;
    float h[G][8];
    float amax = 0.f;
#pragma unroll
    for (int q = 0; q < G; ++q) {
      const int c = threadIdx.x + 128 * q;
      if (c < n8) {
#pragma unroll
        for (int i = 0; i < 8; i += 4) {
          const float4 gv = __ldcg(reinterpret_cast<const float4*>(g + 8 * c + i));
          const float4 uv = __ldcg(reinterpret_cast<const float4*>(u + 8 * c + i));
          h[q][i + 0] = gv.x / (1.f + expf(-gv.x)) * uv.x;
          h[q][i + 1] = gv.y / (1.f + expf(-gv.y)) * uv.y;
          h[q][i + 2] = gv.z / (1.f + expf(-gv.z)) * uv.z;
          h[q][i + 3] = gv.w / (1.f + expf(-gv.w)) * uv.w;
        }
#pragma unroll
        for (int i = 0; i < 8; ++i) amax = fmaxf(amax, fabsf(h[q][i]));
      }
    }
    amax = warp_max(amax);
    if (lane == 0) s_max[warp] = amax;
    __syncthreads();
    amax = fmaxf(fmaxf(s_max[0], s_max[1]), fmaxf(s_max[2], s_max[3]));
    const float sc = pow2_scale_e4m3(amax);
#pragma unroll
    for (int q = 0; q < G; ++q) {
      const int c = threadIdx.x + 128 * q;
      if (c < n8) {
#pragma unroll
        for (int i = 0; i < 8; ++i) h[q][i] *= sc;
        uint2 hi, lo;
        encode_e4m3x2_8(h[q], hi, lo);
        store_e4m3x2_8(hi, lo, p.hq, (size_t)row * kF8Terms, p.I, c);
      }
    }
    if (threadIdx.x == 0) p.hinv[row] = 1.f / sc;
    __syncthreads();  // s_max is reused by the next row
  }
}

}  // namespace moe
