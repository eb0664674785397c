// NVFP4 expert FFN for prefill-shaped batches (many tokens per expert) on the
// tensor cores' block-scaled path, tcgen05.mma kind::mxf4nvf4.
//
// The decode engine (ffn_bs.cuh) cuts an expert's tokens into chunks of 8-16
// and reads each weight tile once per chunk; with ~128 tokens per expert that
// re-stages every tile eight times and the kernel is bound by the traffic
// into each SM.  Here an item is two adjacent 128-row weight tiles against a
// group of up to kPfTok = 64 tokens, over the whole K range:
//
//   * N = 3 x 64 = 192: the first kPfTerms = 3 of the four NVFP4 terms that
//     encode each activation row (act_terms.cuh).  Three terms leave a block
//     residual below ~1/216 of its maximum; the layer output stays within
//     ~2e-3 of the exact result.  One 3-D TMA box copies terms 0-2 of the
//     group's 64 compact rows: B row 3j + t is term t of the group's token j.
//   * Two weight tiles per item, two MMAs per K step against the same
//     activation box: a stage brings 63 KB (two 16 KB weight boxes and their
//     scales, 24 KB of activation rows and theirs) for 256 x 192 outputs.
//     The engine is bound by the bytes each SM can take in (about 70 GB/s
//     with three or four stages in flight); one tile per item brought 45 KB
//     for half the outputs.
//   * Whole K per item: the partial sums are complete in the accumulators, so
//     the epilogue stores them (no atomics, no zeroing): phase 1 the gate or
//     up pre-activations, phase 2 each assignment's down row (y_perm, summed
//     over a token's experts by the combine kernel).
//   * Items (active expert, token group, matrix, tile pair), dealt
//     round-robin (CTA c takes items c, c + G, c + 2G, ...): at any moment
//     the grid works on ~G consecutive items, a few experts, so a group's
//     activation rows (read by every tile of its expert) and a tile (read by
//     both groups of its expert, evict-last until the last group) stay in L2.
//
// Roles (480 threads): warps 0-3 write the stage's scales into tensor memory
// (both weight tiles: 128 rows of 16 B each; the activation rows: 192 rows of
// 16 B; all from shared memory), warps 4-7 and 11-14 are the epilogues of the
// pair's two tiles (TMEM lane quadrant = warp % 4), warp 8 the lead producer
// (the two weight boxes and their scales), warp 9 the MMA issuer, warp 10 the
// second producer (the activation box and its scales: 3-D boxes of three
// terms of 64 rows).  Each epilogue reads its tile, frees it, then stores
// while the next item's MMAs run: with one epilogue for both tiles the MMAs
// waited for its stores (measured on the 235B-shaped layer at 2048 tokens:
// gate/up 406 us, 318 us with the stores left out).
//
// Tensor memory: the two accumulators (192 columns each, one item in flight:
// the MMA issuer waits for the epilogue to read them before an item starts;
// the epilogue loads its per-token scales before that wait), then two slots
// of 64 columns of scales, fewer than the three shared-memory stages: a scale
// slot has its own full and empty barriers.  B scale factors (scale_vec::4X):
// B row n's four scales of one MMA are the 32-bit cell at lane n % 32,
// column c + n / 32 (c a multiple of 4); 192 rows take six columns per MMA,
// eight reserved.
//
// Every wait is bounded (p.wait_ns); an expired wait sets the status word and
// the kernel winds down, freeing its tensor memory.
#pragma once

#include "ffn_bs.cuh"

namespace moe {

constexpr int kPfN = kPfTok * kPfTerms;   // MMA N (kPfTok tokens x kPfTerms terms, ffn.cuh)
// warps 0-10 as in ffn_bs.cuh (warps 4-7: the epilogue of the pair's first
// tile), warps 11-14 the epilogue of its second tile
constexpr int kPfEpi1Warp0 = 11;
constexpr int kPfThreads = 15 * 32;

struct PfGeom {
  static constexpr int A = 0;                                // 2 x 128 rows x 128 B of codes
  static constexpr int SA = 2 * kRowsHalf * kRowBytes;       // 2 x 128 rows x 16 B of scales
  static constexpr int B = SA + 2 * kRowsHalf * 16;          // 36 KB, 1024-aligned
  static constexpr int SB = B + kPfN * kRowBytes;            // + 24 KB of activation rows
  static constexpr int RAW = SB + kPfN * 16;                 // + their scales (16 B a row)
  static constexpr int BYTES = (RAW + 1023) / 1024 * 1024;
  static constexpr int STAGES = 3;
  static constexpr int SMEM = STAGES * BYTES + 1024;
  static constexpr int BYTES_USED = RAW;   // bytes the copies of one stage bring
  static constexpr uint32_t D1 = kPfN;     // tile 1's accumulator (tile 0's at column 0)
  static constexpr uint32_t D_COLS = 2 * kPfN;
  static constexpr int SF_SLOTS = 2;       // scale slots: A0 16, A1 16, B 32 columns
  static constexpr uint32_t SF_COLS = 64;
  static_assert(B % 1024 == 0, "B tile must start a swizzle atom");
  static_assert(D_COLS + SF_SLOTS * SF_COLS <= kBsTmemCols, "tensor memory budget");
  static_assert(kPfN % 16 == 0 && kPfN <= 256, "MMA N");
  static_assert(SMEM <= 227 * 1024 - 10 * 1024, "shared memory");
};

// 3-D tiled TMA load: x the innermost (contiguous) coordinate in elements.
__device__ __forceinline__ void tma_load_3d(void* dst, const CUtensorMap* map, uint64_t* bar,
                                            int x, int y, int z, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      ".L2::cache_hint [%0], [%1, {%3, %4, %5}], [%2], %6;" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_u32(bar)), "r"(x), "r"(y), "r"(z),
      "l"(policy)
      : "memory");
}

struct PfItem {
  int slot, e, mat, rt, arow0, lrow0, nvalid, last_group;  // rt: the pair's first tile
};

// Item `it` of a phase: per active slot, (group, matrix, tile pair) with the
// pair fastest; phase 1 has two matrices (gate, up) of I/256 pairs of 128-row
// tiles, phase 2 one matrix of H/256 pairs.  `rtiles` counts pairs.  The
// plan's chunk prefix counts groups of kPfTok tokens.
__device__ __forceinline__ PfItem pf_item(int it, int per, int rtiles, const PlanSmem& pl,
                                          const FfnParams& p) {
  PfItem r;
  int lo = 0, hi = pl.nA - 1;  // last slot with per * cpre[slot] <= it
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (per * pl.cpre[mid] <= it) lo = mid; else hi = mid - 1;
  }
  r.slot = lo;
  const int ng = pl.cpre[lo + 1] - pl.cpre[lo];
  const int local = it - per * pl.cpre[lo];
  const int g = local / per, q = local - g * per;
  r.rt = 2 * (q % rtiles);
  r.mat = q / rtiles;
  r.e = pl.act[lo];
  r.arow0 = pl.aoff[lo] + g * kPfTok;
  r.lrow0 = r.e * p.T + g * kPfTok;
  const int rem = pl.acnt[lo] - g * kPfTok;
  r.nvalid = rem < kPfTok ? rem : kPfTok;
  r.last_group = (g + 1 == ng);
  return r;
}

template <int PHASE>
__global__ void __launch_bounds__(kPfThreads, 1)
    ffn_pf_kernel(const __grid_constant__ CUtensorMap tmA0,  // gate (phase 2: down) codes
                  const __grid_constant__ CUtensorMap tmA1,  // up codes (phase 1)
                  const __grid_constant__ CUtensorMap tmS0,  // their UE4M3 scales
                  const __grid_constant__ CUtensorMap tmS1,
                  const __grid_constant__ CUtensorMap tmB,   // terms [rows, 4, K/2], 3-term box
                  const __grid_constant__ CUtensorMap tmSB,  // their scales [rows, 4, K/16]
                  const FfnParams p) {
  using G = PfGeom;
  constexpr int S = G::STAGES;
  constexpr int SFS = G::SF_SLOTS;

  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);

  __shared__ __align__(8) uint64_t full_bar[S];
  __shared__ __align__(8) uint64_t empty_bar[S];
  __shared__ __align__(8) uint64_t sf_full[SFS];
  __shared__ __align__(8) uint64_t sf_empty[SFS];
  __shared__ __align__(8) uint64_t dfull_bar;
  __shared__ __align__(8) uint64_t dempty_bar;
  __shared__ __align__(8) uint64_t final_bar;
  __shared__ PlanSmem pl;
  __shared__ float s_sc[2][kPfTok];  // epilogue: per-token scales of an item, by item parity
  __shared__ float s_ts[2];
  __shared__ uint32_t s_tmem;
  __shared__ volatile int s_abort;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    s_abort = 0;
    for (int i = 0; i < S; ++i) {
      mbar_init(&full_bar[i], 1);
      mbar_init(&empty_bar[i], 1);
    }
    for (int i = 0; i < SFS; ++i) {
      mbar_init(&sf_full[i], 4);
      mbar_init(&sf_empty[i], 1);
    }
    mbar_init(&dfull_bar, 1);
    mbar_init(&dempty_bar, 8);  // the eight epilogue warps
    mbar_init(&final_bar, 1);
    fence_mbar_init();
  }
  if (warp == kBsMmaWarp) {
    tmem_alloc(&s_tmem, kBsTmemCols);
    tmem_relinquish();
  }
  // Launched as a programmatic dependent.  Phase 1 waits for the routing and
  // the gathered activation rows here; phase 2's plan and weights do not
  // depend on the SwiGLU kernel before it, so only the roles that read its
  // output wait.
  constexpr bool early = (PHASE == 2);
  if (!early) pdl_wait();
  pdl_launch_dependents();
  if (warp == 0) build_plan(p.counts, p.E, kPfTok, pl, lane);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s_tmem;

  const int N = (PHASE == 1) ? p.I : p.H;  // rows of one expert matrix
  const int K = (PHASE == 1) ? p.H : p.I;  // contraction length
  const int rpairs = N / (2 * kRowsHalf);  // pairs of 128-row tiles
  const int per = (PHASE == 1) ? 2 * rpairs : rpairs;  // items per token group
  const int KB = K / 256;
  const int items = per * pl.cpre[pl.nA];
  // this CTA's items: blockIdx.x, + gridDim.x, ...
  const int my_items = (items > (int)blockIdx.x)
                           ? (items - 1 - (int)blockIdx.x) / (int)gridDim.x + 1 : 0;
  const int i_begin = blockIdx.x;
  const int nst = my_items * KB;
  const uint32_t timeout_bit = (PHASE == 1) ? kStatusTimeoutGateUp : kStatusTimeoutDown;
  constexpr int kTeardown = 13 * 32;  // scale writers, epilogues and MMA warps

  // ================================================================ producers
  if (warp == kBsProducerWarp || warp == kBsProducerWarp2) {
    const bool lead = (warp == kBsProducerWarp);
    if (!lead && early) pdl_wait();  // the activation rows are the SwiGLU output
    if (lane == 0 && nst > 0) {
      tma_prefetch_desc(lead ? &tmA0 : &tmB);
      if (!lead) tma_prefetch_desc(&tmSB);
      if (lead) {
        tma_prefetch_desc(&tmA1);
        tma_prefetch_desc(&tmS0);
        tma_prefetch_desc(&tmS1);
      }
      const uint64_t pol_first = policy_evict_first();
      const uint64_t pol_last = policy_evict_last();
      int it = i_begin, kb = 0, slot = 0, issued = 0;
      uint32_t par = 0u;
      PfItem inf = pf_item(it, per, rpairs, pl, p);
      for (; issued < nst; ++issued) {
        if (!mbar_wait_bounded(&empty_bar[slot], par ^ 1u, p.wait_ns, &s_abort)) {
          set_status(p.status, timeout_bit);
          s_abort = 1;
          break;
        }
        if (!(p.test_stall && issued == 0)) {  // test hook: the first stage never arrives
          unsigned char* st = smem + (size_t)slot * G::BYTES;
          if (lead) {
            mbar_arrive_expect_tx(&full_bar[slot], (uint32_t)(G::BYTES_USED));
            // the next group of the same expert reads these tiles again
            const uint64_t pol = inf.last_group ? pol_first : pol_last;
            const CUtensorMap* ma = inf.mat ? &tmA1 : &tmA0;
            const CUtensorMap* ms = inf.mat ? &tmS1 : &tmS0;
            const int row = inf.e * N + inf.rt * kRowsHalf;
#pragma unroll
            for (int t = 0; t < 2; ++t) {
              tma_load_2d(st + G::A + t * kRowsHalf * kRowBytes, ma, &full_bar[slot],
                          kb * kRowBytes, row + t * kRowsHalf, pol);
              tma_load_2d(st + G::SA + t * kRowsHalf * 16, ms, &full_bar[slot], kb * 16,
                          row + t * kRowsHalf, pol);
            }
          } else {
            tma_load_3d(st + G::B, &tmB, &full_bar[slot], kb * kRowBytes, 0, inf.arow0,
                        pol_last);
            tma_load_3d(st + G::SB, &tmSB, &full_bar[slot], kb * 16, 0, inf.arow0, pol_last);
          }
        }
        if (++slot == S) {
          slot = 0;
          par ^= 1u;
        }
        if (++kb == KB && issued + 1 < nst) {
          kb = 0;
          it += gridDim.x;
          inf = pf_item(it, per, rpairs, pl, p);
        }
      }
      // every copy this CTA issued lands before the CTA exits
      if (lead) {
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
  if (warp == kBsMmaWarp) {
    if (lane == 0) {
      constexpr uint32_t idesc = tc_idesc_mxf4nvf4(128, kPfN);
      bool ok = true;
      int slot = 0, fs = 0, kb = 0, nitem = 0;
      uint32_t par = 0u, fpar = 0u;
      for (int i = 0; i < nst && ok; ++i) {
        if (kb == 0)
          ok = mbar_wait_bounded(&dempty_bar, ((uint32_t)nitem & 1u) ^ 1u, p.wait_ns, &s_abort);
        ok = ok && mbar_wait_bounded(&full_bar[slot], par, p.wait_ns, &s_abort) &&
             mbar_wait_bounded(&sf_full[fs], fpar, p.wait_ns, &s_abort);
        if (!ok) break;
        tc_fence_after();
        const uint32_t st = smem_u32(smem + (size_t)slot * G::BYTES);
        const uint32_t sfc = tmem + G::D_COLS + (uint32_t)fs * G::SF_COLS;
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {
          const uint64_t bdesc = tc_desc_sw128(st + G::B + 32 * kk);
          const uint32_t acc = (kb == 0 && kk == 0) ? 0u : 1u;
          tc_mma_mxf4nvf4(tmem, tc_desc_sw128(st + G::A + 32 * kk), bdesc, idesc, sfc + 4 * kk,
                          sfc + 32 + 8 * kk, acc);
          tc_mma_mxf4nvf4(tmem + G::D1, tc_desc_sw128(st + G::A + kRowsHalf * kRowBytes + 32 * kk),
                          bdesc, idesc, sfc + 16 + 4 * kk, sfc + 32 + 8 * kk, acc);
        }
        tc_commit(&empty_bar[slot]);
        tc_commit(&sf_empty[fs]);
        if (++kb == KB) {
          kb = 0;
          tc_commit(&dfull_bar);
          ++nitem;
        }
        if (++slot == S) {
          slot = 0;
          par ^= 1u;
        }
        if (++fs == SFS) {
          fs = 0;
          fpar ^= 1u;
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
    constexpr int NH = kPfN / 32;  // B rows per lane: lane + 32 h
    int slot = 0, fs = 0;
    uint32_t par = 0u, fpar = 0u;
    for (int i = 0; i < nst; ++i) {
      // the stage's copies have landed, and the scale slot's previous MMAs are done
      if (!mbar_wait_bounded(&full_bar[slot], par, p.wait_ns, &s_abort) ||
          !mbar_wait_bounded(&sf_empty[fs], fpar ^ 1u, p.wait_ns, &s_abort)) {
        set_status(p.status, timeout_bit);
        s_abort = 1;
        break;
      }
      tc_fence_after();
      const uint32_t st = smem_u32(smem + (size_t)slot * G::BYTES);
      const uint32_t sfc = tmem + lane_addr + G::D_COLS + (uint32_t)fs * G::SF_COLS;
#pragma unroll
      for (int t = 0; t < 2; ++t) {  // the weight tiles' scales: columns 16t + 4kk + r
        uint4 v[4];
#pragma unroll
        for (int r1 = 0; r1 < 4; ++r1)
          v[r1] = lds128(st + G::SA + t * kRowsHalf * 16 + (lane + 32 * r1) * 16);
        uint32_t c[16];
#pragma unroll
        for (int r1 = 0; r1 < 4; ++r1) {
          c[0 + r1] = v[r1].x;   // MMA 0 (K 0-63 of the stage)
          c[4 + r1] = v[r1].y;
          c[8 + r1] = v[r1].z;
          c[12 + r1] = v[r1].w;
        }
        tmem_st16(sfc + 16 * t, c);
      }
      {
        // B row n = 3j + t: term t of the group's token j (rows past the
        // group's tokens hold other rows or the copy's zeros; their columns
        // are not stored)
        uint4 bsf[NH];
#pragma unroll
        for (int h = 0; h < NH; ++h) bsf[h] = lds128(st + G::SB + (lane + 32 * h) * 16);
#pragma unroll
        for (int half = 0; half < 2; ++half) {  // MMAs 2 half, 2 half + 1: 8 columns each
          uint32_t c[16];
#pragma unroll
          for (int m2 = 0; m2 < 2; ++m2) {
            const int kk = 2 * half + m2;
#pragma unroll
            for (int h = 0; h < 8; ++h) {
              uint32_t wv = 0u;
              if (h < NH) {
                const uint4 bb = bsf[h < NH ? h : 0];
                wv = kk == 0 ? bb.x : kk == 1 ? bb.y : kk == 2 ? bb.z : bb.w;
              }
              c[8 * m2 + h] = wv;
            }
          }
          tmem_st16(sfc + 32 + 16 * half, c);
        }
      }
      tmem_st_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sf_full[fs]);
      if (++slot == S) {
        slot = 0;
        par ^= 1u;
      }
      if (++fs == SFS) {
        fs = 0;
        fpar ^= 1u;
      }
    }
    tc_fence_before();
    asm volatile("bar.sync 2, %0;" ::"n"(kTeardown) : "memory");
    return;
  }

  // ================================================================ epilogues
  // Warp w reads TMEM lanes 32(w%4)..+31 of its tile's accumulator: row
  // 32(w%4) + lane of the tile.
  {
    if (early) pdl_wait();  // the row scales of h are the SwiGLU output
    const int tile = warp >= kPfEpi1Warp0 ? 1 : 0;
    const int quad = warp & 3;
    const int tid = tile ? 128 + (warp - kPfEpi1Warp0) * 32 + lane
                         : (warp - kBsEpiWarp0) * 32 + lane;  // 0..255
    const int row = quad * 32 + lane;
    const uint32_t lane_addr = (uint32_t)(quad * 32) << 16;
    // true in every epilogue thread when it is true in any (the waits are per
    // thread; the named barrier of the next item needs all 256 threads)
    auto any_dead = [&](bool v) -> bool {
      uint32_t rr;
      asm volatile(
          "{\n .reg .pred p, q;\n setp.ne.u32 p, %1, 0;\n"
          " bar.red.or.pred q, 3, 256, p;\n selp.u32 %0, 1, 0, q;\n}\n"
          : "=r"(rr)
          : "r"((uint32_t)v)
          : "memory");
      return rr != 0;
    };
    // per-token scales of item `it` (x's row scale in phase 1, h's in phase
    // 2) and its tensor scale, read by threads 0..kPfTok
    auto load_scales = [&](int it, float& v) {
      const PfItem inf = pf_item(it, per, rpairs, pl, p);
      v = 0.f;
      if (tid < inf.nvalid) {
        if (PHASE == 1)
          v = __ldg(p.xinv + __ldg(p.sorted + inf.lrow0 + tid) / p.k);
        else
          v = __ldg(p.xinv + inf.arow0 + tid);
      } else if (tid == kPfTok) {
        v = __ldg((inf.mat ? p.ts1 : p.ts0) + inf.e);
      }
    };
    float v_next = 0.f;
    if (my_items > 0) {
      load_scales(i_begin, v_next);
      if (tid < kPfTok) s_sc[0][tid] = v_next;
      if (tid == kPfTok) s_ts[0] = v_next;
    }
    for (int n = 0, it = i_begin; n < my_items; ++n, it += gridDim.x) {
      const PfItem inf = pf_item(it, per, rpairs, pl, p);
      const int b = n & 1;
      // the next item's scales are requested now and stored after this
      // item's accumulator is read: their latency overlaps the MMAs
      const bool has_next = n + 1 < my_items;
      if (has_next) load_scales(it + gridDim.x, v_next);
      asm volatile("bar.sync 3, 256;" ::: "memory");
      const bool ok = mbar_wait_bounded(&dfull_bar, (uint32_t)n & 1u, p.wait_ns, &s_abort);
      if (any_dead(!ok)) {
        set_status(p.status, timeout_bit);
        s_abort = 1;
        break;
      }
      tc_fence_after();
      // the three terms of token j are the tile's accumulator columns 3j..3j+2
      float acc[kPfTok];
#pragma unroll
      for (int c0 = 0; c0 < kPfN; c0 += 48) {
        uint32_t v[48];
        const uint32_t ta = tmem + lane_addr + (uint32_t)tile * G::D1 + (uint32_t)c0;
        tmem_ld16(ta, *reinterpret_cast<uint32_t(*)[16]>(v));
        tmem_ld16(ta + 16, *reinterpret_cast<uint32_t(*)[16]>(v + 16));
        tmem_ld16(ta + 32, *reinterpret_cast<uint32_t(*)[16]>(v + 32));
        tmem_ld_wait();
#pragma unroll
        for (int j = 0; j < 16; ++j)
          acc[c0 / 3 + j] = (__uint_as_float(v[3 * j]) + __uint_as_float(v[3 * j + 1])) +
                            __uint_as_float(v[3 * j + 2]);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&dempty_bar);  // this warp's part of the accumulators is read
      if (has_next) {  // every thread is past the previous item: its buffer is free
        if (tid < kPfTok) s_sc[b ^ 1][tid] = v_next;
        if (tid == kPfTok) s_ts[b ^ 1] = v_next;
      }
      const float ts = s_ts[b];
      const int col = (inf.rt + tile) * kRowsHalf + row;
#pragma unroll
      for (int j = 0; j < kPfTok; ++j) {
        if (j >= inf.nvalid) break;
        const float y = acc[j] * s_sc[b][j] * ts;
        if (PHASE == 1)
          p.gu[(size_t)(inf.arow0 + j) * 2 * p.I + inf.mat * p.I + col] = y;
        else
          p.y_perm[(size_t)(inf.arow0 + j) * p.H + col] = y;
      }
    }
    tc_fence_before();
    asm volatile("bar.sync 2, %0;" ::"n"(kTeardown) : "memory");
  }
}

}  // namespace moe
