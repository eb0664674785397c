// Expert FFN kernels of the MoE decode layer (gate/up + SwiGLU, and down +
// combine), for FP8 E4M3 with 128x128 fp32 block scales and NVFP4: what the
// three engines share (parameters, work plan, stage split and cursors, the
// FP8 engine's shared tail, SwiGLU and finalize kernels), and the warp-MMA
// engine itself (ffn_kernel).  The tensor-core engines are in ffn_bs.cuh
// (NVFP4) and ffn_f8.cuh (FP8).
//
// Shape of the work.  Per active expert e with n_e routed tokens, the
// gate/up step streams 2*I*H weights and the down step H*I weights, each
// used against only n_e <= a few dozen token columns: the steps are
// HBM-bound weight streams (the decode-lane regime of the paper's
// Section 2.1).  The kernels are built around keeping HBM busy:
//
// * Work list.  Items are (active expert, row tile, token chunk of <= NT
//   tokens); each item is a run of K-blocks ("stages").  The stages of all
//   items are laid end to end and every CTA of a persistent grid takes a
//   contiguous share of them (stream-K): an equal share in the warp-MMA
//   engine, a share of equal cost in the tensor-core engines
//   (cost_split_stage), where the FP8 engine also leaves a shared tail of
//   units to whichever CTA is free.  Partial sums of an item split between
//   CTAs meet in fp32 accumulators through red.global.add.
// * Pipeline.  Producer threads issue 2-D TMA tensor copies of each stage
//   (weight boxes of 128 rows x 128 bytes with 128B swizzle, the NVFP4 scale
//   boxes, and the stage's token rows) into a ring of shared-memory stages
//   guarded by mbarriers.  In the warp-MMA engine consumer warps (eight per
//   128-row box, or sixteen with each stage's K split in two) decode and
//   multiply.
// * Decode (warp-MMA engine).  E4M3 and E2M1*E4M3 values are exact in f16,
//   so weights are converted exactly in registers (cvt e4m3x2/e2m1x2 ->
//   f16x2; the NVFP4 per-16 scale multiplied in f16, still exact).
//   Activations are stored as f16 after a per-row power-of-two scaling
//   (exact for bf16 inputs).  mma m16n8k16 (fp32 accumulate) does the
//   multiply-adds with the tokens as the n=8 side; FP8 block scales and
//   NVFP4 tensor scales are applied to the fp32 accumulators.
// * Fusion.  The gate/up step adds fp32 pre-activations into [T*k, 2I]
//   accumulators; a SwiGLU kernel turns them into the down step's input.
//   The down step multiplies by the gate weight and adds straight into a
//   [T, H] fp32 accumulator (the scatter-combine); finalize_kernel writes
//   bf16 (+ residual).
#pragma once

#include "common.cuh"

namespace moe {

constexpr int kFfnMTiles = 8;  // 16-row MMA tiles per 128-row weight box
// Consumer warps = kFfnMTiles * KS: with KS = 2 the two halves of each stage's
// K range go to different warps, which doubles the warps that hide latency.
template <int KS>
constexpr int ffn_threads() { return (kFfnMTiles * KS + 1) * 32; }
constexpr int kRowsHalf = 128;  // rows of each of the two weight boxes of a stage
constexpr int kRowBytes = 128;  // weight bytes per row per stage
// Prefill engine (ffn_pf.cuh): tokens per item and activation terms used.
constexpr int kPfTok = 64;
constexpr int kPfTerms = 3;

template <int FMT>
struct FmtTraits;
template <>
struct FmtTraits<1> {           // FP8 E4M3, 128x128 block scales
  static constexpr int KEL = 128;  // K elements per stage
  static constexpr int NU = 2;     // 16-byte activation units per (thread, half)
  static constexpr int SBYTES = 0; // scale bytes per row per stage (in smem)
};
template <>
struct FmtTraits<2> {           // NVFP4
  static constexpr int KEL = 256;
  static constexpr int NU = 4;
  static constexpr int SBYTES = 16;
};

// Physical position of 16-byte unit U of an activation row block of one
// stage.  NVFP4 rows swap units so that the four threads of an MMA quad hit
// four different bank groups; FP8 rows are stored in order.
template <int FMT>
__host__ __device__ __forceinline__ int act_unit(int U) {
  if (FMT == 2) return U ^ ((U >> 2) & 2);
  return U;
}

// Element index within a row of x16 / h16 where logical column `col` lives.
template <int FMT>
__host__ __device__ __forceinline__ int act_pos(int col) {
  constexpr int KEL = FmtTraits<FMT>::KEL;
  const int kb = col / KEL, q = col % KEL;
  return kb * KEL + act_unit<FMT>(q >> 3) * 8 + (q & 7);
}

template <int FMT, int NT>
struct StageGeom {
  static constexpr int KEL = FmtTraits<FMT>::KEL;
  static constexpr int A0 = 0;
  static constexpr int A1 = kRowsHalf * kRowBytes;                   // 16 KB
  static constexpr int S0 = 2 * kRowsHalf * kRowBytes;               // 32 KB
  static constexpr int S1 = S0 + kRowsHalf * FmtTraits<FMT>::SBYTES;
  static constexpr int B = S0 + 2 * kRowsHalf * FmtTraits<FMT>::SBYTES;
  static constexpr int BROW = KEL * 2;                               // bytes per token row
  static constexpr int RAW = B + NT * BROW;
  static constexpr int BYTES = (RAW + 1023) / 1024 * 1024;
  static constexpr int STAGES_RAW = (212 * 1024) / BYTES;  // + ~10 KB static
  static constexpr int STAGES = STAGES_RAW > 8 ? 8 : STAGES_RAW;
  static constexpr int SMEM = STAGES * BYTES + 1024;  // + alignment slack
};

struct FfnParams {
  int T, k, E, H, I, phase;  // phase 1 = gate/up, 2 = down
  int fused;                 // phase 2: 1 = scatter into oacc + bf16 out, 0 = y_perm
  // 1 = deterministic mode: every CTA's share of the stages starts and ends
  // on an item boundary (the units of the FP8 engine's shared tail are whole
  // items), and the unfused phase 2 writes row
  // a (the assignment t*k + j) of y_perm instead of the compact row.  The
  // tensor-core engines then store each output element once (gu and y_perm
  // need no zeroing); the warp-MMA engine still adds the partial sums of its
  // two K-halves (two adds onto zero give the same bits in either order).
  // The tensor-core engines take it as a template parameter: runtime branches
  // on it in the epilogue's unrolled loops made the default NVFP4 down
  // kernel 13% slower (16-token chunks, 82 -> 93 us a launch).
  int det;
  // FP8 tensor-core engine with 32-token chunks: K-blocks per slab of an
  // expert with several chunks (SlabCursor); 0 or >= K/128 keeps each
  // chunk's item whole
  int slab;
  // routing: tokens per expert, and each expert's assignments (t*k + j).
  // list_T = 1: expert e's list starts at sorted[e*T] (the fused layer's
  // per-expert lists); 0: at sorted[offsets[e]] (one array sorted by expert).
  const int* counts;   // [E]
  const int* sorted;
  int list_T;
  // phase 1 of the tensor-core engines: 1 = the activation terms were
  // gathered into compact-row order (one B box per chunk), 0 = per token
  int b_compact;
  const float* gates;  // [T*k] by assignment (fused only)
  uint32_t* acnt_reset;  // finalize_kernel zeroes these E counters (fused only)
  // scales
  const float* s0;     // FP8 block scales of the matrix behind box A0/A1
  const float* s1;
  const float* ts0;    // NVFP4 tensor scales [E]
  const float* ts1;
  // activations / accumulators
  const float* xinv;   // phase 1: [T]; phase 2: hinv [T*k]
  float* gu;           // phase 1 out / phase 2 (unused)
  __half* h16;         // SwiGLU output (warp-MMA engine)
  float* hinv;         // SwiGLU output row scales
  float* oacc;         // phase 2 fused accumulator [T, H]
  float* y_perm;       // phase 2 unfused output [T*k, H]
  __nv_bfloat16* out;  // phase 2 fused output
  const __nv_bfloat16* residual;
  // block-scaled engine (ffn_bs.cuh): scales of the activation terms of this
  // phase's B operand, and the SwiGLU output as terms
  const uint8_t* bsf;  // [rows * 4, K/16] UE4M3
  uint8_t* hq;         // [T*k*4, I/2] E2M1 codes
  uint8_t* hsf;        // [T*k*4, I/16] UE4M3
  uint32_t* status;
  // tensor-core engines: {next unit, CTAs done} of this phase's shared tail;
  // the last CTA to finish puts both back to zero
  uint32_t* units;
  uint64_t wait_ns;
  int test_stall;      // test hook: producer withholds its first stage
};

// ------------------------------------------------------------------ work plan
// The expert kernels build their work plan from the per-expert token counts
// in shared memory: the active experts in increasing id order, their first
// row in the compact [T*k] row space (rows ordered by expert), and the prefix
// of their NT-token chunks, which numbers the items.
struct PlanSmem {
  int act[kMaxE];       // active expert ids, increasing
  int acnt[kMaxE];      // their token counts
  int aoff[kMaxE + 1];  // their first compact row; aoff[nA] = all assignments
  int cpre[kMaxE + 1];  // chunk prefix; cpre[nA] = total chunks
  int nA;
};

// One warp: scan the counts in groups of 32 (inclusive warp scans carried
// across groups).  The caller synchronises the block afterwards.
__device__ __forceinline__ void build_plan(const int* counts, int E, int NT, PlanSmem& pl,
                                           int lane) {
  int run_off = 0, run_act = 0, run_ch = 0;
  unsigned lt;
  asm("mov.u32 %0, %%lanemask_lt;" : "=r"(lt));
  constexpr int G = kMaxE / 32;
  int cnt[G];  // every count load in flight before the first is used
#pragma unroll
  for (int g = 0; g < G; ++g) {
    const int e = 32 * g + lane;
    cnt[g] = (e < E) ? __ldcg(counts + e) : 0;
  }
#pragma unroll
  for (int g = 0; g < G; ++g) {
    const int base = 32 * g;
    if (base >= E) break;
    const int e = base + lane;
    const int c = cnt[g];
    const int ch = (c + NT - 1) / NT;
    int oc = c, och = ch;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y0 = __shfl_up_sync(0xffffffffu, oc, o);
      const int y1 = __shfl_up_sync(0xffffffffu, och, o);
      if (lane >= o) {
        oc += y0;
        och += y1;
      }
    }
    const unsigned am = __ballot_sync(0xffffffffu, c > 0);
    if (c > 0) {
      const int slot = run_act + __popc(am & lt);
      pl.act[slot] = e;
      pl.acnt[slot] = c;
      pl.aoff[slot] = run_off + oc - c;
      pl.cpre[slot] = run_ch + och - ch;
    }
    run_off += __shfl_sync(0xffffffffu, oc, 31);
    run_ch += __shfl_sync(0xffffffffu, och, 31);
    run_act += __popc(am);
  }
  if (lane == 0) {
    pl.nA = run_act;
    pl.cpre[run_act] = run_ch;
    pl.aoff[run_act] = run_off;
  }
}

// Relative cost of one stage of an item with n tokens: kStageCost + n *
// kTokenCost.  The weight tile of a stage is the same for every item; each
// token adds its own activation-row copy and scale loads (one TMA box and one
// scale row per token when the rows are copied token by token) and its output
// rows in the epilogue.  Measured on the 235B-shaped NVFP4 layer at 64 tokens:
// a CTA's finishing time grows by ~1/25 of a one-token stage per extra token
// when the rows come token by token.
constexpr int kTokenCost = 1;
__host__ __device__ constexpr int stage_cost_base(bool per_token_rows) {
  return per_token_rows ? 24 : 64;
}

// The first stage (item-major, decode_item's order) that begins at or after
// the fraction num / den of the total cost.  The cost prefix over active
// experts follows from the chunk and token prefixes: sum of (a * chunks + b *
// tokens) per row tile and K-stage.  f(0) = 0, f(den) = every stage, f
// increasing in num.  Host-callable so that the library can run the same code
// on a plan built from counts (moe_cost_split_stage).
__host__ __device__ __forceinline__ int cost_split_stage(const PlanSmem& pl, int rtiles, int KB, int NT,
                                                int a, int b, long long num, long long den) {
  const long long per = (long long)rtiles * KB;
  auto prefix = [&](int s) {
    return per * ((long long)a * pl.cpre[s] + (long long)b * pl.aoff[s]);
  };
  const long long X = prefix(pl.nA) * num / den;
  int lo = 0, hi = pl.nA;  // last slot whose cost prefix is <= X
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (prefix(mid) <= X) lo = mid; else hi = mid - 1;
  }
  if (lo == pl.nA) return pl.cpre[pl.nA] * rtiles * KB;
  const long long r = X - prefix(lo);
  const int n = pl.acnt[lo];
  const int ch = pl.cpre[lo + 1] - pl.cpre[lo];
  const long long c_rt = (long long)KB * ((long long)a * ch + (long long)b * n);
  const int rt = (int)(r / c_rt);
  const long long r2 = r - rt * c_rt;
  const int nfull = n / NT;  // chunks of NT tokens
  const long long wf = a + (long long)b * NT;
  int chunk;
  long long r3, w;
  if (r2 < nfull * KB * wf) {
    chunk = (int)(r2 / (KB * wf));
    r3 = r2 - chunk * KB * wf;
    w = wf;
  } else {  // the last, partial chunk
    chunk = nfull;
    r3 = r2 - nfull * KB * wf;
    w = a + (long long)b * (n - nfull * NT);
  }
  const int kb = (int)((r3 + w - 1) / w);  // <= KB: a stage that starts at or after X
  return ((pl.cpre[lo] * rtiles) + rt * ch + chunk) * KB + kb;
}

// Deterministic mode: a share boundary moved to the nearest item boundary
// (items are KB stages long), so that every item is summed by one CTA over
// its whole K range.  Both CTAs beside a boundary round it alike.
__host__ __device__ __forceinline__ long long item_boundary(long long s, int KB) {
  return (s + KB / 2) / KB * KB;
}

// Position of a CTA's current stage without divisions: item `it`, K-block
// `kb` inside it, ring slot and that slot's phase parity ((i / S) & 1).
template <int S>
struct StageCursor {
  int it, kb, KB, slot;
  uint32_t par;
  __device__ __forceinline__ StageCursor(int s_begin, int kb_per_item)
      : it(s_begin / kb_per_item), kb(s_begin - (s_begin / kb_per_item) * kb_per_item),
        KB(kb_per_item), slot(0), par(0u) {}
  __device__ __forceinline__ void next() {
    if (++kb == KB) {
      kb = 0;
      ++it;
    }
    if (++slot == S) {
      slot = 0;
      par ^= 1u;
    }
  }
  // jump to stage s of the sequence; the ring position runs on
  __device__ __forceinline__ void seek(int s) {
    it = s / KB;
    kb = s - it * KB;
  }
};

// StageCursor with the constructor and run test of SlabCursor below: the item
// order for kernels that take either.
template <int S>
struct ItemCursor : StageCursor<S> {
  __device__ __forceinline__ ItemCursor(const PlanSmem&, int, int kb_per_item, int, int s_begin)
      : StageCursor<S>(s_begin, kb_per_item) {}
  // last stage of the item: its sums are added out
  __device__ __forceinline__ bool ends_run() const { return this->kb + 1 == this->KB; }
};

// The same sequence of stages in slab order (FP8 tensor-core engine).  The
// stages of one (expert, row tile) group keep their place in the sequence,
// but inside a group of several token chunks the K range is cut into slabs
// of SL K-blocks, and every chunk runs over slab j before any runs over slab
// j + 1: a weight box is read from HBM by the first chunk and from L2 by the
// others while the CTA holds at most SL stages' boxes for them, where whole
// items (SL = KB) left them to be read again from HBM once the boxes of all
// CTAs' current tiles outgrew L2.  A group of one chunk is one slab of KB
// stages, the item order of decode_item.  `it` is the item (expert, row
// tile, chunk) for decode_item, `run_end` marks the last stage of a chunk's
// run in its slab: its partial sums are added out there.
template <int S>
struct SlabCursor {
  const PlanSmem* pl;
  int rtiles, KB, SL;
  int lo, rt, nch, it0;    // group: expert slot, row tile, chunks, first item
  int chunk, ks0, sl, kbs;  // chunk, first K-block and length of the slab, offset
  int it, kb, slot;
  bool run_end;
  uint32_t par;
  __host__ __device__ __forceinline__ SlabCursor(const PlanSmem& plan, int rtiles_, int kb_per_item,
                                        int slab, int s_begin)
      : pl(&plan), rtiles(rtiles_), KB(kb_per_item),
        SL(slab > 0 && slab < kb_per_item ? slab : kb_per_item), slot(0), par(0u) {
    seek(s_begin);
  }
  __host__ __device__ __forceinline__ int group_slab() const { return nch > 1 ? SL : KB; }
  __host__ __device__ __forceinline__ bool ends_run() const { return run_end; }
  __host__ __device__ __forceinline__ void settle() {
    kb = ks0 + kbs;
    it = it0 + chunk;
    run_end = (kbs + 1 == sl);
  }
  // jump to stage s of the sequence; the ring position runs on
  __host__ __device__ __forceinline__ void seek(int s) {
    int a = 0, b = pl->nA - 1;  // last slot whose first stage is <= s
    while (a < b) {
      const int mid = (a + b + 1) >> 1;
      if (pl->cpre[mid] * rtiles * KB <= s) a = mid; else b = mid - 1;
    }
    lo = a;
    nch = pl->nA > 0 ? pl->cpre[lo + 1] - pl->cpre[lo] : 1;
    if (nch < 1) nch = 1;
    const int base = pl->nA > 0 ? pl->cpre[lo] : 0;
    const int local = s - base * rtiles * KB;
    rt = local / (nch * KB);
    const int o = local - rt * nch * KB;
    it0 = base * rtiles + rt * nch;
    const int g = group_slab();
    const int nfs = KB / g;
    if (o < nfs * nch * g) {
      const int j = o / (nch * g);
      const int o1 = o - j * nch * g;
      chunk = o1 / g;
      kbs = o1 - chunk * g;
      ks0 = j * g;
      sl = g;
    } else {
      sl = KB - nfs * g;
      const int o2 = o - nfs * nch * g;
      chunk = o2 / sl;
      kbs = o2 - chunk * sl;
      ks0 = nfs * g;
    }
    settle();
  }
  __host__ __device__ __forceinline__ void next() {
    if (++kbs == sl) {
      kbs = 0;
      if (++chunk == nch) {
        chunk = 0;
        ks0 += sl;
        if (ks0 == KB) {
          ks0 = 0;
          it0 += nch;
          if (++rt == rtiles) {
            rt = 0;
            if (++lo < pl->nA) nch = pl->cpre[lo + 1] - pl->cpre[lo];
          }
        }
        const int g = group_slab();
        sl = g < KB - ks0 ? g : KB - ks0;
      }
    }
    settle();
    if (++slot == S) {
      slot = 0;
      par ^= 1u;
    }
  }
};

// ------------------------------------------------------------------ shared tail
// A CTA of the FP8 tensor-core engine streams its own share of the stages first
// (divided by cost, kStaticNum / kStaticDen of the total cost), then units of
// kUnitStages stages of the rest, taken one at a time from a global counter
// by the lead producer and handed to the CTA's other roles through a ring in
// shared memory.  A CTA whose copies land faster takes more of the tail.
// In the deterministic mode a unit is one whole item (KB stages) and the tail
// starts on an item boundary, so that every item is still summed by one CTA.
constexpr int kUnitStages = 8;
constexpr int kStaticNum = 4, kStaticDen = 5;
constexpr int kTailMinStages = 200;  // per CTA
constexpr int kUnitRing = 32;  // > the units one role can run ahead of another

struct UnitRing {
  int first[kUnitRing];  // first stage of the unit; -1: no more units
  uint64_t full[kUnitRing];
  uint64_t empty[kUnitRing];
};

// Lead producer: publish unit j (its first stage a, or -1) once every reader
// of entry j - kUnitRing has taken it.
__device__ __forceinline__ bool unit_push(UnitRing& r, int j, int a, uint64_t wait_ns,
                                          volatile int* abort) {
  const int q = j % kUnitRing;
  if (!mbar_wait_bounded(&r.empty[q], ((uint32_t)(j / kUnitRing) & 1u) ^ 1u, wait_ns, abort))
    return false;
  *reinterpret_cast<volatile int*>(&r.first[q]) = a;
  mbar_arrive(&r.full[q]);
  return true;
}

// Reader: unit j as the stage range [a, b); false at the end of the tail or
// when the wait expired (*ok = false).  A warp-wide reader calls this on all
// lanes and lane 0 reports the entry read; a one-thread reader reports it
// itself (warp_wide false).
__device__ __forceinline__ bool unit_next(UnitRing& r, int& j, int total, int us, int& a,
                                          int& b, bool warp_wide, uint64_t wait_ns,
                                          volatile int* abort, bool* ok) {
  const int q = j % kUnitRing;
  if (!mbar_wait_bounded(&r.full[q], (uint32_t)(j / kUnitRing) & 1u, wait_ns, abort)) {
    *ok = false;
    return false;
  }
  const int first = *reinterpret_cast<volatile int*>(&r.first[q]);
  if (warp_wide) {
    __syncwarp();
    if ((threadIdx.x & 31) == 0) mbar_arrive(&r.empty[q]);
  } else {
    mbar_arrive(&r.empty[q]);
  }
  ++j;
  if (first < 0) return false;
  a = first;
  b = min(first + us, total);
  return true;
}

// Lead producer, after its last unit: count this CTA done; the last CTA puts
// the counters back to zero for the next launch (every CTA has taken its
// last unit by then).
__device__ __forceinline__ void unit_done(uint32_t* units) {
  __threadfence();
  if (atomicAdd(units + 1, 1u) == gridDim.x - 1) {
    units[0] = 0u;
    units[1] = 0u;
    __threadfence();
  }
}

// The unit that follows a CTA's last one: first stage, or -1 past the end.
__device__ __forceinline__ int unit_take(uint32_t* units, int s_dyn, int total, int us) {
  const long long a = (long long)s_dyn + (long long)atomicAdd(units, 1u) * us;
  return a < total ? (int)a : -1;
}

struct ItemInfo {
  int slot, e, arow0, lrow0, nvalid, rt;
};

// Item `it` = (active expert, row tile, chunk), chunk fastest: the items of
// one expert's row tile are adjacent, so a hot expert's weight tile is read
// from HBM once and its further token chunks find it in L2.  arow0 is the
// chunk's first compact row, lrow0 the index of its first assignment in
// p.sorted.
__device__ __forceinline__ ItemInfo decode_item(long long it, int rtiles, const PlanSmem& pl,
                                                const FfnParams& p, int NT) {
  ItemInfo r;
  int lo = 0, hi = pl.nA - 1;  // last slot with cpre[slot] * rtiles <= it
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if ((long long)pl.cpre[mid] * rtiles <= it) lo = mid; else hi = mid - 1;
  }
  r.slot = lo;
  const int nch = pl.cpre[lo + 1] - pl.cpre[lo];  // chunks of this expert
  const int local = (int)(it - (long long)pl.cpre[lo] * rtiles);
  r.rt = local / nch;
  const int chunk = local - r.rt * nch;
  r.e = pl.act[lo];
  r.arow0 = pl.aoff[lo] + chunk * NT;
  r.lrow0 = (p.list_T ? r.e * p.T : pl.aoff[lo]) + chunk * NT;
  const int rem = pl.acnt[lo] - chunk * NT;
  r.nvalid = rem < NT ? rem : NT;
  return r;
}

// ------------------------------------------------------------------ between and after the phases
// SwiGLU of every assignment row: h = silu(g) * u from the fp32 gate|up
// accumulators, scaled per row by a power of two into f16 (in the unit order
// of the warp-MMA NVFP4 layout when `perm`).  One CTA per row: every thread
// loads its share of the row once (up to 8 groups of 4 columns, I <= 8192),
// the row maximum comes from a shared-memory reduction, and the scaled values
// are written from registers - two memory latencies per row.
template <int FMT>
__global__ void __launch_bounds__(256) swiglu_kernel(const FfnParams p, int rows, int perm) {
  constexpr int G = 8;  // float4 groups per thread
  __shared__ float s_max[8];
  // the down step may launch now: what it does before its own wait (plan,
  // weight copies) does not read this kernel's output
  pdl_launch_dependents();
  pdl_wait();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int n4 = p.I / 4;
  for (int row = blockIdx.x; row < rows; row += gridDim.x) {
    const float4* g4 = reinterpret_cast<const float4*>(p.gu + (size_t)row * 2 * p.I);
    const float4* u4 = reinterpret_cast<const float4*>(p.gu + (size_t)row * 2 * p.I + p.I);
    float4 hv[G];
    float amax = 0.f;
#pragma unroll
    for (int q = 0; q < G; ++q) {
      const int i = threadIdx.x + 256 * q;
      if (i < n4) {
        const float4 gv = __ldcg(g4 + i), uv = __ldcg(u4 + i);
        hv[q].x = gv.x / (1.f + expf(-gv.x)) * uv.x;
        hv[q].y = gv.y / (1.f + expf(-gv.y)) * uv.y;
        hv[q].z = gv.z / (1.f + expf(-gv.z)) * uv.z;
        hv[q].w = gv.w / (1.f + expf(-gv.w)) * uv.w;
        amax = fmaxf(amax, fmaxf(fmaxf(fabsf(hv[q].x), fabsf(hv[q].y)),
                                 fmaxf(fabsf(hv[q].z), fabsf(hv[q].w))));
      }
    }
    amax = warp_max(amax);
    if (lane == 0) s_max[warp] = amax;
    __syncthreads();
    amax = s_max[0];
#pragma unroll
    for (int w = 1; w < 8; ++w) amax = fmaxf(amax, s_max[w]);
    const float sc = pow2_scale_for(amax);
    __half* hr = p.h16 + (size_t)row * p.I;
#pragma unroll
    for (int q = 0; q < G; ++q) {
      const int i = threadIdx.x + 256 * q;
      if (i < n4) {
        const __half2 lo = __floats2half2_rn(hv[q].x * sc, hv[q].y * sc);
        const __half2 hi = __floats2half2_rn(hv[q].z * sc, hv[q].w * sc);
        uint2 o;
        o.x = *reinterpret_cast<const uint32_t*>(&lo);
        o.y = *reinterpret_cast<const uint32_t*>(&hi);
        const int f = 4 * i;  // 4 consecutive columns stay inside one 16-byte unit
        *reinterpret_cast<uint2*>(hr + (perm ? act_pos<FMT>(f) : f)) = o;
      }
    }
    if (threadIdx.x == 0) p.hinv[row] = 1.f / sc;
    __syncthreads();  // s_max is reused by the next row
  }
}

// out = bf16(oacc + residual), four columns per thread.
static __global__ void __launch_bounds__(256) finalize_kernel(const FfnParams p) {
  pdl_wait();
  // the per-expert assignment counters start the next layer call from zero
  if (p.acnt_reset && blockIdx.x == 0)
    for (int e = threadIdx.x; e < p.E; e += blockDim.x) p.acnt_reset[e] = 0u;
  const size_t n4 = (size_t)p.T * p.H / 4;
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < n4;
       i += (size_t)gridDim.x * blockDim.x) {
    float4 a = __ldcg(reinterpret_cast<const float4*>(p.oacc) + i);
    if (p.residual) {
      const uint2 r = *(reinterpret_cast<const uint2*>(p.residual) + i);
      const float2 r0 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&r.x));
      const float2 r1 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&r.y));
      a.x += r0.x;
      a.y += r0.y;
      a.z += r1.x;
      a.w += r1.y;
    }
    const __nv_bfloat162 o0 = __floats2bfloat162_rn(a.x, a.y);
    const __nv_bfloat162 o1 = __floats2bfloat162_rn(a.z, a.w);
    uint2 o;
    o.x = *reinterpret_cast<const uint32_t*>(&o0);
    o.y = *reinterpret_cast<const uint32_t*>(&o1);
    *(reinterpret_cast<uint2*>(p.out) + i) = o;
  }
}

// ------------------------------------------------------------------ the kernel
template <int FMT, int NT, int KS>
__global__ void __launch_bounds__(ffn_threads<KS>(), 1)
    ffn_kernel(const __grid_constant__ CUtensorMap tmA0, const __grid_constant__ CUtensorMap tmA1,
               const __grid_constant__ CUtensorMap tmS0, const __grid_constant__ CUtensorMap tmS1,
               const __grid_constant__ CUtensorMap tmB, const FfnParams p) {
  using G = StageGeom<FMT, NT>;
  constexpr int KEL = G::KEL;
  constexpr int NTILE = NT / 8;
  constexpr int S = G::STAGES;

  extern __shared__ __align__(1024) unsigned char smem_raw[];
  // stage ring, 1024-byte aligned in the shared window (128B-swizzle atoms)
  unsigned char* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);

  __shared__ __align__(8) uint64_t full_bar[S];
  __shared__ __align__(8) uint64_t empty_bar[S];
  __shared__ PlanSmem pl;
  __shared__ int s_tok[NT];
  __shared__ volatile int s_abort;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  constexpr int CW = kFfnMTiles * KS;  // consumer warps
  const bool is_producer = (warp == CW);

  if (threadIdx.x == 0) {
    s_abort = 0;
    for (int i = 0; i < S; ++i) {
      mbar_init(&full_bar[i], 1);
      mbar_init(&empty_bar[i], CW);
    }
    fence_mbar_init();
  }
  // Launched as a programmatic dependent: everything above overlapped the
  // previous kernel; from here on its outputs are read.
  pdl_wait();
  pdl_launch_dependents();
  if (warp == 0) build_plan(p.counts, p.E, NT, pl, lane);
  __syncthreads();

  const int N = (p.phase == 1) ? p.I : p.H;       // rows of one expert matrix
  const int K = (p.phase == 1) ? p.H : p.I;       // contraction length
  const int rtiles = (p.phase == 1) ? p.I / kRowsHalf : p.H / (2 * kRowsHalf);
  const int KB = K / KEL;
  const long long items = (long long)pl.cpre[pl.nA] * rtiles;
  const long long total = items * KB;
  long long s_begin = total * blockIdx.x / gridDim.x;
  long long s_end = total * (blockIdx.x + 1) / gridDim.x;
  if (p.det) {
    s_begin = item_boundary(s_begin, KB);
    s_end = item_boundary(s_end, KB);
  }
  const uint32_t timeout_bit = (p.phase == 1) ? kStatusTimeoutGateUp : kStatusTimeoutDown;

  if (is_producer) {
    if (lane == 0 && s_end > s_begin) {
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
          inf = decode_item(it, rtiles, pl, p, NT);
          if (p.phase == 1)
            for (int j = 0; j < inf.nvalid; ++j) s_tok[j] = __ldg(p.sorted + inf.lrow0 + j) / p.k;
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
        const int npad = (inf.nvalid + 7) & ~7;
        uint32_t bytes = 2u * kRowsHalf * kRowBytes + 2u * kRowsHalf * FmtTraits<FMT>::SBYTES;
        bytes += (p.phase == 1) ? (uint32_t)inf.nvalid * G::BROW : (uint32_t)npad * G::BROW;
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
        if (p.phase == 1) {
          for (int j = 0; j < inf.nvalid; ++j)
            tma_load_2d(st + G::B + j * G::BROW, &tmB, &full_bar[slot], kb * KEL, s_tok[j], pol_a);
        } else {
          for (int r8 = 0; r8 < npad; r8 += 8)
            tma_load_2d(st + G::B + r8 * G::BROW, &tmB, &full_bar[slot], kb * KEL, inf.arow0 + r8,
                        pol_a);
        }
      }
      // Let every copy this CTA issued land before the CTA exits.
      const long long first = issued > S ? issued - S : 0;
      for (long long j = first; j < issued; ++j) {
        if (p.test_stall && j == 0) continue;
        mbar_wait_bounded(&full_bar[j % S], (uint32_t)((j / S) & 1), p.wait_ns, nullptr);
      }
    }
    return;
  }

  // ---------------------------------------------------------------- consumers
  const int g = lane >> 2, t = lane & 3;
  // MMA row m of this warp's 16-row tile lives in shared row 16*warp + rho(m);
  // the order makes the two row groups of each quarter-warp differ in bit 2,
  // so the 128B-swizzled reads of a quarter-warp never share a bank.
  const int rho_g = ((g & 1) << 2) | (g >> 1);
  const int mtile = warp % kFfnMTiles;
  const int khalf = warp / kFfnMTiles;  // KS = 2: which half of the stage's K
  const int ra = 16 * mtile + rho_g, rb = ra + 8;

  float acc0[NTILE][4], acc1[NTILE][4];
  long long cur_item = -1;
  ItemInfo inf{};
  // per-item column data
  float colscale[NTILE][2];
  int colrow[NTILE][2];   // flush destination row (assignment row or token)
  float colgate[NTILE][2];

  auto zero_acc = [&]() {
#pragma unroll
    for (int n = 0; n < NTILE; ++n)
#pragma unroll
      for (int i = 0; i < 4; ++i) acc0[n][i] = acc1[n][i] = 0.f;
  };

  auto load_item_cols = [&]() {
#pragma unroll
    for (int n = 0; n < NTILE; ++n)
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        const int j = n * 8 + 2 * t + c;
        colscale[n][c] = 0.f;
        colrow[n][c] = -1;
        colgate[n][c] = 0.f;
        if (j < inf.nvalid) {
          const int arow = inf.arow0 + j;
          const int a = __ldg(p.sorted + inf.lrow0 + j);
          if (p.phase == 1) {
            colscale[n][c] = __ldg(p.xinv + a / p.k);
            colrow[n][c] = arow;
          } else {
            colscale[n][c] = __ldcg(p.xinv + arow);  // hinv, written by the previous kernel
            if (p.fused) {
              colrow[n][c] = a / p.k;
              colgate[n][c] = __ldg(p.gates + a);
            } else {
              colrow[n][c] = p.det ? a : arow;
              colgate[n][c] = 1.f;
            }
          }
        }
      }
  };

  // Adds the item's partial sums to the global accumulators.
  // `dead`: this warp stopped at an expired wait; it adds nothing.
  auto flush = [&](bool dead) {
    float ts0 = 1.f, ts1 = 1.f;
    if (FMT == 2) {
      ts0 = __ldg(p.ts0 + inf.e);
      ts1 = __ldg(p.ts1 + inf.e);
    }
#pragma unroll
    for (int n = 0; n < NTILE; ++n)
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        if (dead || colrow[n][c] < 0) continue;
        const float sc = colscale[n][c];
        const int dst = colrow[n][c];
#pragma unroll
        for (int half = 0; half < 2; ++half) {
          const float v0 = acc0[n][c + 2 * half] * sc * ts0;
          const float v1 = acc1[n][c + 2 * half] * sc * ts1;
          const int mrow = 16 * mtile + rho_g + 8 * half;  // row within the 128-row box
          if (p.phase == 1) {
            const int f = inf.rt * kRowsHalf + mrow;
            float* base = p.gu + (size_t)dst * 2 * p.I;
            red_add_f32(base + f, v0);
            red_add_f32(base + p.I + f, v1);
          } else {
            const int hrow = inf.rt * 2 * kRowsHalf + mrow;
            const float gw = colgate[n][c];
            float* base = p.fused ? p.oacc + (size_t)dst * p.H : p.y_perm + (size_t)dst * p.H;
            red_add_f32(base + hrow, gw * v0);
            red_add_f32(base + hrow + kRowsHalf, gw * v1);
          }
        }
      }
  };

  zero_acc();
  long long consumed = 0;
  bool dead = false;
  for (long long s = s_begin; s < s_end; ++s, ++consumed) {
    const long long it = s / KB;
    const int kb = (int)(s % KB);
    if (it != cur_item) {
      if (cur_item >= 0) {
        flush(dead);
        zero_acc();
      }
      cur_item = it;
      inf = decode_item(it, rtiles, pl, p, NT);
      load_item_cols();
    }
    if (dead) continue;
    // FP8 block scales of this stage (one per 128x128 tile of each box)
    float bs0 = 1.f, bs1 = 1.f;
    if (FMT == 1) {
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
    const int slot = (int)(consumed % S);
    const uint32_t round = (uint32_t)(consumed / S);
    if (!mbar_wait_bounded(&full_bar[slot], round & 1u, p.wait_ns, &s_abort)) {
      set_status(p.status, timeout_bit);
      s_abort = 1;
      dead = true;
      continue;
    }
    const uint32_t st = smem_u32(smem + (size_t)slot * G::BYTES);
    const int ntiles = (inf.nvalid + 7) >> 3;

    float tmp0[NTILE][4], tmp1[NTILE][4];
#pragma unroll
    for (int n = 0; n < NTILE; ++n)
#pragma unroll
      for (int i = 0; i < 4; ++i) tmp0[n][i] = tmp1[n][i] = 0.f;

    // Load phase: this warp's share of the stage (weights, scales, token
    // fragments) into registers.  With EARLY the slot is released right after,
    // so the producer can refill it while the warp computes.
    constexpr int HH = 2 / KS;                  // halves of the stage's K per warp
    constexpr int NU = FmtTraits<FMT>::NU;
    constexpr bool EARLY = (KS == 2 && NT == 8);
    uint4 qa0[HH], qb0[HH], qa1[HH], qb1[HH];
    uint32_t sa0[HH], sb0[HH], sa1[HH], sb1[HH];  // NVFP4 scale pairs (f16x2)
    uint4 xb[HH][NU][NTILE];
#pragma unroll
    for (int hh = 0; hh < HH; ++hh) {
      const int h = (KS == 2) ? khalf : hh;
      const int c = 4 * h + t;  // 16-byte weight chunk of this thread
      qa0[hh] = lds128(st + G::A0 + ra * kRowBytes + ((c ^ (ra & 7)) << 4));
      qb0[hh] = lds128(st + G::A0 + rb * kRowBytes + ((c ^ (rb & 7)) << 4));
      qa1[hh] = lds128(st + G::A1 + ra * kRowBytes + ((c ^ (ra & 7)) << 4));
      qb1[hh] = lds128(st + G::A1 + rb * kRowBytes + ((c ^ (rb & 7)) << 4));
      if (FMT == 2) {
        sa0[hh] = lds16(st + G::S0 + ra * 16 + 2 * c);
        sb0[hh] = lds16(st + G::S0 + rb * 16 + 2 * c);
        sa1[hh] = lds16(st + G::S1 + ra * 16 + 2 * c);
        sb1[hh] = lds16(st + G::S1 + rb * 16 + 2 * c);
      }
      if (EARLY) {
#pragma unroll
        for (int u = 0; u < NU; ++u)
#pragma unroll
          for (int n = 0; n < NTILE; ++n)
            if (n < ntiles)
              xb[hh][u][n] =
                  lds128(st + G::B + (n * 8 + g) * G::BROW + (act_unit<FMT>(c * NU + u) << 4));
      }
    }
    if (EARLY) {
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty_bar[slot]);
    }

#pragma unroll
    for (int hh = 0; hh < HH; ++hh) {
      const int c = 4 * ((KS == 2) ? khalf : hh) + t;
      // NVFP4: the two 16-element scales of this chunk per row, as f16x2
      // broadcasts {s, s} of the lower (k-steps 0-3) and upper (4-7) block
      uint32_t sa0lo = 0, sa0hi = 0, sb0lo = 0, sb0hi = 0;
      uint32_t sa1lo = 0, sa1hi = 0, sb1lo = 0, sb1hi = 0;
      if (FMT == 2) {
        const uint32_t fa0 = e4m3x2_to_f16x2(sa0[hh]), fb0 = e4m3x2_to_f16x2(sb0[hh]);
        const uint32_t fa1 = e4m3x2_to_f16x2(sa1[hh]), fb1 = e4m3x2_to_f16x2(sb1[hh]);
        sa0lo = __byte_perm(fa0, 0, 0x1010);
        sa0hi = __byte_perm(fa0, 0, 0x3232);
        sb0lo = __byte_perm(fb0, 0, 0x1010);
        sb0hi = __byte_perm(fb0, 0, 0x3232);
        sa1lo = __byte_perm(fa1, 0, 0x1010);
        sa1hi = __byte_perm(fa1, 0, 0x3232);
        sb1lo = __byte_perm(fb1, 0, 0x1010);
        sb1hi = __byte_perm(fb1, 0, 0x3232);
      }
      const uint32_t wa0[4] = {qa0[hh].x, qa0[hh].y, qa0[hh].z, qa0[hh].w};
      const uint32_t wb0[4] = {qb0[hh].x, qb0[hh].y, qb0[hh].z, qb0[hh].w};
      const uint32_t wa1[4] = {qa1[hh].x, qa1[hh].y, qa1[hh].z, qa1[hh].w};
      const uint32_t wb1[4] = {qb1[hh].x, qb1[hh].y, qb1[hh].z, qb1[hh].w};
#pragma unroll
      for (int u = 0; u < NU; ++u) {
        // token fragments of this unit: 8 f16 = K positions P..P+7 of this thread
        uint4 xu[NTILE];
#pragma unroll
        for (int n = 0; n < NTILE; ++n) {
          if (n < ntiles)
            xu[n] = EARLY ? xb[hh][u][n]
                          : lds128(st + G::B + (n * 8 + g) * G::BROW +
                                   (act_unit<FMT>(c * NU + u) << 4));
        }
        // weights of the two k-steps of this unit: FP8 uses one 32-bit word
        // (4 codes) per row per k-step, NVFP4 one word (8 codes) per row per 2 k-steps
        uint32_t dA0[2][4], dA1[2][4];  // [k-step][a-reg]
        if (FMT == 1) {
#pragma unroll
          for (int ss = 0; ss < 2; ++ss) {
            const int s_ = 2 * u + ss;
            e4m3x4_to_f16x4(wa0[s_], dA0[ss][0], dA0[ss][2]);
            e4m3x4_to_f16x4(wb0[s_], dA0[ss][1], dA0[ss][3]);
            e4m3x4_to_f16x4(wa1[s_], dA1[ss][0], dA1[ss][2]);
            e4m3x4_to_f16x4(wb1[s_], dA1[ss][1], dA1[ss][3]);
          }
        } else {
          // word u holds k-steps 2u (bytes 0,1) and 2u+1 (bytes 2,3); the
          // 16-element scale block of k-step s_ is 2c + (s_ >> 2)
          const uint32_t ca0 = (u < 2) ? sa0lo : sa0hi, cb0 = (u < 2) ? sb0lo : sb0hi;
          const uint32_t ca1 = (u < 2) ? sa1lo : sa1hi, cb1 = (u < 2) ? sb1lo : sb1hi;
          uint32_t qa[4], qb[4], qc[4], qd[4];
          e2m1x8_to_f16x8(wa0[u], qa);
          e2m1x8_to_f16x8(wb0[u], qb);
          e2m1x8_to_f16x8(wa1[u], qc);
          e2m1x8_to_f16x8(wb1[u], qd);
#pragma unroll
          for (int ss = 0; ss < 2; ++ss) {
            dA0[ss][0] = hmul2_u32(qa[2 * ss], ca0);
            dA0[ss][2] = hmul2_u32(qa[2 * ss + 1], ca0);
            dA0[ss][1] = hmul2_u32(qb[2 * ss], cb0);
            dA0[ss][3] = hmul2_u32(qb[2 * ss + 1], cb0);
            dA1[ss][0] = hmul2_u32(qc[2 * ss], ca1);
            dA1[ss][2] = hmul2_u32(qc[2 * ss + 1], ca1);
            dA1[ss][1] = hmul2_u32(qd[2 * ss], cb1);
            dA1[ss][3] = hmul2_u32(qd[2 * ss + 1], cb1);
          }
        }
#pragma unroll
        for (int ss = 0; ss < 2; ++ss) {
          const uint32_t* A0r = dA0[ss];
          const uint32_t* A1r = dA1[ss];
#pragma unroll
          for (int n = 0; n < NTILE; ++n) {
            if (n < ntiles) {
              const uint32_t b0 = ss ? xu[n].z : xu[n].x;
              const uint32_t b1 = ss ? xu[n].w : xu[n].y;
              mma_f16(tmp0[n], A0r[0], A0r[1], A0r[2], A0r[3], b0, b1);
              mma_f16(tmp1[n], A1r[0], A1r[1], A1r[2], A1r[3], b0, b1);
            }
          }
        }
      }
    }
    if (!EARLY) {
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty_bar[slot]);
    }
#pragma unroll
    for (int n = 0; n < NTILE; ++n)
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        acc0[n][i] = fmaf(bs0, tmp0[n][i], acc0[n][i]);
        acc1[n][i] = fmaf(bs1, tmp1[n][i], acc1[n][i]);
      }
  }
  if (cur_item >= 0) flush(dead);
}

}  // namespace moe
