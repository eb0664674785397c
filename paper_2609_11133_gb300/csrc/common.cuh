// Shared device helpers of libmoe: PTX wrappers for mbarriers, TMA tensor
// copies, bounded waits, warp MMA and the workspace layout.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_fp4.h>
#include <cuda_fp8.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>

namespace moe {

// ------------------------------------------------------------------ limits
constexpr int kMaxE = 512;          // experts per layer
constexpr int kMaxTK = 65536;       // T * k
constexpr int kMaxHI = 32768;       // H and I
constexpr int kRouteTok = 8;        // tokens per router CTA
constexpr int kRouteWarps = 8;      // warps per router CTA

// Device status bits (the first error wins; see moe_read_status).
constexpr uint32_t kStatusTimeoutGateUp = 1u;
constexpr uint32_t kStatusTimeoutDown = 2u;
constexpr uint32_t kStatusBadExpertId = 4u;
constexpr uint32_t kStatusTimeoutRoute = 8u;

// Tensor-core router (route_tc.cu), used for large batches: the logits as a
// bf16 GEMM against the fp32 router split exactly into three bf16 parts, its
// K range cut into kRouteTcSplit slices whose fp32 partial sums the router
// kernel adds in slice order.  The slice count does not depend on T, so a
// token's logits are the same in every batch that takes this router.
constexpr int kRouteTcSplit = 8;
constexpr int kRouteTcMaxE = 256;  // experts: one MMA N (a multiple of 16, <= 256)
inline int route_tc_ep(int E) { return (E + 15) / 16 * 16; }

// Bounded waits give up after this many nanoseconds of %globaltimer.
constexpr uint64_t kWaitLimitNs = 1000000000ull;  // 1 s

// ------------------------------------------------------------------ workspace
// Byte offsets of everything the kernels keep between launches.  Built on the
// host by ws_layout() and passed by value to the kernels.
// Activation forms the expert engines read.
constexpr int kActF16 = 0;      // f16 rows (power-of-two scaled), natural order
constexpr int kActF16Perm = 1;  // f16 rows in the warp-MMA NVFP4 unit order
constexpr int kActTerms = 2;    // four NVFP4 terms per row (block-scaled engine)
constexpr int kActE4M3 = 3;     // two E4M3 terms per row (FP8 tensor-core engine)

struct WsLayout {
  // control block (zeroed once; every counter is reset by its last user)
  size_t status;       // u32 device status word
  size_t acnt;         // u32 [kMaxE] assignments per expert (fused layer)
  size_t units;        // u32 [4] shared-tail counters of the two expert phases
  size_t route_chunk;  // u32 [nChunks] per-token-chunk arrival tickets
  // routing
  size_t logits;   // f32 [T, E]
  size_t ids;      // i32 [T, k]
  size_t gates;    // f32 [T, k]
  size_t counts;   // i32 [E] tokens per expert (moe_expert_ffn)
  size_t alist;    // i32 [E, T] per-expert assignment lists (fused layer)
  // activations
  size_t xinv;     // f32 [T]   power-of-two inverse scale of x16 rows
  size_t x16;      // f16 [T, H]
  size_t gu;       // f32 [T*k, 2I] gate | up pre-activations
  size_t hinv;     // f32 [T*k]
  size_t h16;      // f16 [T*k, I]
  size_t oacc;     // f32 [T, H] combine accumulator
  // activation terms of the tensor-core engines (zero-sized otherwise; x16
  // and h16 are zero-sized when these are used).  NVFP4: x codes [4T, H/2],
  // x scales [4T, H/16], h codes [4Tk, I/2], h scales [4Tk, I/16]; FP8:
  // x [2T, H] and h [2Tk, I] E4M3 (hi and lo rows).
  size_t xq;
  size_t xsf;
  size_t hq;
  size_t hsf;
  // T > 64, tensor-core engines: x terms gathered into compact-row order
  // (rows as h: terms per assignment), and their NVFP4 scales
  size_t xg;
  size_t xgsf;
  // prefill-shaped NVFP4 batches: each assignment's down row and the compact
  // row of each assignment (zero-sized otherwise); the deterministic mode of
  // the decode engines keeps the down rows too (by assignment)
  size_t yperm;    // f32 [T*k, H]
  size_t inv;      // i32 [T*k]
  // tensor-core router (zero-sized otherwise): the router's three bf16 parts,
  // the partial logits of the K slices, and the pre-normalised rows of x
  size_t w3;       // bf16 [3, Ep, H]
  size_t plog;     // f32 [kRouteTcSplit, T, Ep]
  size_t xn;       // bf16 [T, H]
  size_t total;
  int nChunks;
};

inline size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

// Rows of an h-terms array (`terms` rows per assignment), at least one full
// down-step B box (64 rows) so that a box never extends past the array.
inline size_t hq_rows(int T, int k, int terms) {
  const size_t r = (size_t)terms * T * k;
  return r < 64 ? 64 : r;
}

// The fused layer gathers the activation terms into compact-row order when
// chunks are wide (more than 64 tokens): one B box per chunk instead of one
// per token.
inline bool gather_terms(int T, int act) {
  return T > 64 && (act == kActTerms || act == kActE4M3);
}

// Prefill-shaped NVFP4 batches, at least 32 tokens per expert on average, run
// on the prefill engine (ffn_pf.cuh): items of 64 tokens, each assignment's
// down row in y_perm, summed by the combine kernel.
inline bool prefill_shape(int T, int k, int E, int act) {
  return act == kActTerms && T > 64 && (long long)T * k >= 32LL * E;
}

inline WsLayout ws_layout(int T, int k, int E, int H, int I, int act = kActF16,
                          bool det = false, bool tcr = false) {
  WsLayout L{};
  size_t o = 0;
  auto take = [&](size_t bytes) {
    size_t r = o;
    o = align_up(o + bytes, 256);
    return r;
  };
  L.nChunks = (T + kRouteTok - 1) / kRouteTok;
  const size_t TK = (size_t)T * k;
  L.status = take(4);
  L.acnt = take(4 * (size_t)kMaxE);  // fixed size: the same offset for every T and E
  L.units = take(16);
  L.route_chunk = take(4 * (size_t)(L.nChunks > 0 ? L.nChunks : 1));
  L.logits = take(4 * (size_t)T * E);
  L.ids = take(4 * TK);
  L.gates = take(4 * TK);
  L.counts = take(4 * (size_t)E);
  L.alist = take(4 * (size_t)E * T);
  L.xinv = take(4 * (size_t)T);
  const size_t nf = (act == kActF16 || act == kActF16Perm) ? 1 : 0;  // warp-MMA engine only
  L.x16 = take(nf * 2 * (size_t)T * H);
  L.gu = take(4 * TK * 2 * (size_t)I);
  L.hinv = take(4 * TK);
  L.h16 = take(nf * 2 * TK * (size_t)I);
  L.oacc = take(4 * (size_t)T * H);
  const size_t n4 = (act == kActTerms) ? 1 : 0, n8 = (act == kActE4M3) ? 1 : 0;
  L.xq = take((n4 + n8) * 2 * (size_t)T * H);  // 4T rows x H/2, or 2T rows x H
  L.xsf = take(n4 * 4 * (size_t)T * H / 16);
  L.hq = take(n4 * hq_rows(T, k, 4) * (size_t)I / 2 + n8 * hq_rows(T, k, 2) * (size_t)I);
  L.hsf = take(n4 * hq_rows(T, k, 4) * (size_t)I / 16);
  const size_t ng = gather_terms(T, act) ? 1 : 0;
  L.xg = take(ng * (n4 * hq_rows(T, k, 4) * (size_t)H / 2 + n8 * hq_rows(T, k, 2) * (size_t)H));
  L.xgsf = take(ng * n4 * hq_rows(T, k, 4) * (size_t)H / 16);
  const size_t npf = prefill_shape(T, k, E, act) ? 1 : 0;
  L.yperm = take((npf || det ? 1 : 0) * 4 * TK * (size_t)H);
  L.inv = take(npf * 4 * TK);
  const size_t nr = tcr ? 1 : 0, Ep = (size_t)route_tc_ep(E);
  L.w3 = take(nr * 3 * Ep * H * 2);
  L.plog = take(nr * kRouteTcSplit * (size_t)T * Ep * 4);
  L.xn = take(nr * (size_t)T * H * 2);
  L.total = o;
  return L;
}

// Raise a kernel's dynamic shared-memory limit once per device (the call is a
// host-side attribute change; doing it once keeps it out of graph captures
// and off the per-call path).  `mask` is one bit per device, per kernel.
template <typename K>
inline cudaError_t set_smem_once(K kern, int bytes, std::atomic<unsigned long long>& mask) {
  int dev = 0;
  cudaError_t err = cudaGetDevice(&dev);
  if (err != cudaSuccess) return err;
  const unsigned long long bit = 1ull << (dev & 63);
  if (mask.load(std::memory_order_acquire) & bit) return cudaSuccess;
  err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (err == cudaSuccess) mask.fetch_or(bit, std::memory_order_acq_rel);
  return err;
}

template <typename Ty>
__host__ __device__ inline Ty* ws_ptr(void* ws, size_t off) {
  return reinterpret_cast<Ty*>(static_cast<char*>(ws) + off);
}

// ------------------------------------------------------------------ PTX helpers
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count)
               : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Wait for phase `parity` of `bar` to complete.  Gives up (returns false) when
// the deadline passes or when *abort becomes non-zero.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity,
                                                  uint64_t limit_ns, volatile int* abort) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  while (true) {
    for (int i = 0; i < 64; ++i)
      if (mbar_try_wait(bar, parity)) return true;
    if (abort != nullptr && *abort) return false;
    if (globaltimer_ns() - t0 > limit_ns) return false;
  }
}

// 2-D tiled TMA load global -> shared, completion counted on `bar` in bytes.
// `x` is the innermost (contiguous) coordinate in elements, `y` the row.
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, uint64_t* bar,
                                            int x, int y, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      ".L2::cache_hint [%0], [%1, {%3, %4}], [%2], %5;" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_u32(bar)), "r"(x), "r"(y), "l"(policy)
      : "memory");
}

__device__ __forceinline__ void tma_prefetch_desc(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

__device__ __forceinline__ uint64_t policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}

__device__ __forceinline__ uint64_t policy_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}

// 16-byte shared-memory load.
__device__ __forceinline__ uint4 lds128(uint32_t addr) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "r"(addr));
  return v;
}

__device__ __forceinline__ uint32_t lds16(uint32_t addr) {
  unsigned short v;
  asm volatile("ld.shared.u16 %0, [%1];" : "=h"(v) : "r"(addr));
  return v;
}

// D = A * B + C, m16n8k16, f16 inputs, f32 accumulators.
__device__ __forceinline__ void mma_f16(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                        uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// Four E4M3 bytes of `w` to four exact f16 values: lo = bytes 0,1 and
// hi = bytes 2,3, lower byte in the lower half (hardware cvt, one per pair).
__device__ __forceinline__ void e4m3x4_to_f16x4(uint32_t w, uint32_t& lo, uint32_t& hi) {
  asm("{\n .reg .b16 p0, p1;\n mov.b32 {p0, p1}, %2;\n"
      " cvt.rn.f16x2.e4m3x2 %0, p0;\n cvt.rn.f16x2.e4m3x2 %1, p1;\n}\n"
      : "=r"(lo), "=r"(hi)
      : "r"(w));
}

// Two E4M3 bytes (low byte -> low half) to two exact f16 values.
__device__ __forceinline__ uint32_t e4m3x2_to_f16x2(uint32_t two_bytes) {
  uint32_t r;
  const uint16_t v = static_cast<uint16_t>(two_bytes);
  asm("cvt.rn.f16x2.e4m3x2 %0, %1;" : "=r"(r) : "h"(v));
  return r;
}

// Eight E2M1 codes of `w` (byte i holds codes 2i (low nibble) and 2i+1) to
// four f16x2 values d[i] = {code 2i, code 2i+1}, exact.
__device__ __forceinline__ void e2m1x8_to_f16x8(uint32_t w, uint32_t (&d)[4]) {
  asm("{\n .reg .b8 q0, q1, q2, q3;\n mov.b32 {q0, q1, q2, q3}, %4;\n"
      " cvt.rn.f16x2.e2m1x2 %0, q0;\n cvt.rn.f16x2.e2m1x2 %1, q1;\n"
      " cvt.rn.f16x2.e2m1x2 %2, q2;\n cvt.rn.f16x2.e2m1x2 %3, q3;\n}\n"
      : "=r"(d[0]), "=r"(d[1]), "=r"(d[2]), "=r"(d[3])
      : "r"(w));
}

__device__ __forceinline__ uint32_t hmul2_u32(uint32_t a, uint32_t b) {
  __half2 r = __hmul2(*reinterpret_cast<__half2*>(&a), *reinterpret_cast<__half2*>(&b));
  return *reinterpret_cast<uint32_t*>(&r);
}

__device__ __forceinline__ void red_add_f32(float* p, float v) {
  asm volatile("red.global.add.f32 [%0], %1;" ::"l"(p), "f"(v) : "memory");
}

// A sum into an output element: added to the zeroed accumulator, or stored
// where it is the element's only sum (the deterministic mode of the
// tensor-core engines, whose CTAs each sum whole items).
__device__ __forceinline__ void put_f32(float* p, float v, bool store) {
  if (store)
    asm volatile("st.global.f32 [%0], %1;" ::"l"(p), "f"(v) : "memory");
  else
    red_add_f32(p, v);
}

// Power-of-two factor that maps max|v| into [2^14, 2^15): f16 holds the
// scaled value exactly for every bf16 input and leaves headroom for sums.
__device__ __forceinline__ float pow2_scale_for(float amax) {
  if (!(amax > 0.f) || !isfinite(amax)) return 1.f;
  int e;
  frexpf(amax, &e);  // amax = m * 2^e, 0.5 <= m < 1
  return ldexpf(1.f, 15 - e);
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ void set_status(uint32_t* status, uint32_t bit) {
  if (status) atomicOr(status, bit);
}

// Programmatic dependent launch controls (no-ops when not launched as such).
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

}  // namespace moe

namespace moe {
// ------------------------------------------------------------------ tcgen05 helpers
// Tensor memory (TMEM): 128 lanes x 512 columns of 32-bit cells per SM.  An
// address is (lane << 16) | column.  A warp may touch lanes 32*(warp%4) ..+31.

__device__ __forceinline__ void tmem_alloc(uint32_t* holder, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(holder)),
               "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
// Arrive once on `bar` when every tcgen05 operation this thread issued so far completes.
__device__ __forceinline__ void tc_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                   smem_u32(bar))
               : "memory");
}
// 16 consecutive 32-bit columns of this thread's lane.
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&v)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, "
      "%11, %12, %13, %14, %15, %16};" ::"r"(taddr),
      "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]),
      "r"(v[8]), "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]),
      "r"(v[15])
      : "memory");
}
__device__ __forceinline__ void tmem_st_wait() {
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&v)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, "
      "%11, %12, %13, %14, %15}, [%16];"
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]),
        "=r"(v[7]), "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]),
        "=r"(v[14]), "=r"(v[15])
      : "r"(taddr)
      : "memory");
}
__device__ __forceinline__ void tmem_ld_wait() {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// Shared-memory matrix descriptor: K-major operand stored in 128-byte rows
// with the 128B swizzle, 8-row atoms 1024 bytes apart.
__device__ __forceinline__ uint64_t tc_desc_sw128(uint32_t smem_addr) {
  uint64_t d = 0;
  d |= (uint64_t)((smem_addr & 0x3FFFFu) >> 4);  // start address
  d |= (uint64_t)1u << 16;                       // leading byte offset (unused here)
  d |= (uint64_t)(1024u >> 4) << 32;             // stride byte offset: next 8-row atom
  d |= (uint64_t)1u << 46;                       // descriptor version
  d |= (uint64_t)2u << 61;                       // 128-byte swizzle
  return d;
}
}  // namespace moe
