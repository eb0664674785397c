// C ABI of libmoe (declared in include/moe.h): argument validation, workspace
// layout, TMA tensor-map encoding and kernel launches.  Host code only.
#include <cudaTypedefs.h>

#include <atomic>
#include <cstdlib>
#include <cstring>
#include <mutex>

#include "../../include/moe.h"
#include "act_terms.cuh"
#include "ffn_launch.cuh"
#include "route.cuh"

using namespace moe;

namespace {

constexpr int kAbiVersion = 100;  // 0.1.0
constexpr int kFlagTestStall = 0x100;  // test hook, see the comment in moe.h

// ------------------------------------------------------------------ device facts
struct DevInfo {
  std::atomic<int> ready{0};
  int sms = 0, ok = 0;
  long long l2 = 0;  // L2 bytes
};
DevInfo g_dev[64];

int device_check(int* sms) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return MOE_ERR_CUDA;
  DevInfo& d = g_dev[dev];
  if (!d.ready.load(std::memory_order_acquire)) {
    int major = 0, minor = 0, n = 0, l2 = 0;
    if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&l2, cudaDevAttrL2CacheSize, dev) != cudaSuccess)
      return MOE_ERR_CUDA;
    d.sms = n;
    d.l2 = l2;
    d.ok = (major == 10 && minor == 3);
    d.ready.store(1, std::memory_order_release);
  }
  if (!d.ok) return MOE_ERR_UNSUPPORTED_DEVICE;
  *sms = d.sms;
  return MOE_OK;
}

// L2 size of the current device (after device_check).
long long device_l2_bytes() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  return g_dev[dev].l2;
}

uint64_t wait_limit_ns() {
  static std::atomic<uint64_t> cached{0};
  uint64_t v = cached.load();
  if (v == 0) {
    v = kWaitLimitNs;
    if (const char* s = std::getenv("MOE_WAIT_LIMIT_MS")) {
      const long ms = std::strtol(s, nullptr, 10);
      if (ms > 0 && ms <= 60000) v = (uint64_t)ms * 1000000ull;
    }
    cached.store(v);
  }
  return v;
}

// ------------------------------------------------------------------ tensor maps
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
  });
  return fn;
}

bool map_2d(CUtensorMap* m, CUtensorMapDataType dt, const void* base, uint64_t cols,
            uint64_t rows, uint64_t row_bytes, uint32_t box_cols, uint32_t box_rows,
            CUtensorMapSwizzle sw) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {row_bytes};
  cuuint32_t box[2] = {box_cols, box_rows};
  cuuint32_t es[2] = {1, 1};
  return fn(m, dt, 2, const_cast<void*>(base), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// codes of one expert-stacked matrix [E*N, Kbytes], 128 x 128-byte boxes, 128B swizzle
bool map_codes(CUtensorMap* m, const uint8_t* codes, int E, int N, int Kbytes) {
  return map_2d(m, CU_TENSOR_MAP_DATA_TYPE_UINT8, codes, (uint64_t)Kbytes, (uint64_t)E * N,
                (uint64_t)Kbytes, kRowBytes, kRowsHalf, CU_TENSOR_MAP_SWIZZLE_128B);
}

// NVFP4 scales [E*N, K/16] bytes, 128 x 16-byte boxes
bool map_sf(CUtensorMap* m, const void* sf, int E, int N, int K) {
  return map_2d(m, CU_TENSOR_MAP_DATA_TYPE_UINT8, sf, (uint64_t)(K / 16), (uint64_t)E * N,
                (uint64_t)(K / 16), 16, kRowsHalf, CU_TENSOR_MAP_SWIZZLE_NONE);
}

// Activation-term arrays [rows, 4 terms, row_bytes] as a 3-D map whose box is
// the first kPfTerms terms of kPfTok rows: the prefill engine's B operand
// (codes, 128 bytes of K per row, 128B swizzle) and its scales (16 bytes per
// row, no swizzle); B row 3j + t = term t of row j.
bool map_terms3(CUtensorMap* m, const void* base, int row_bytes, int rows, bool codes) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[3] = {(cuuint64_t)row_bytes, (cuuint64_t)kTerms, (cuuint64_t)rows};
  cuuint64_t strides[2] = {(cuuint64_t)row_bytes, (cuuint64_t)row_bytes * kTerms};
  cuuint32_t box[3] = {codes ? (cuuint32_t)kRowBytes : 16u, (cuuint32_t)kPfTerms,
                       (cuuint32_t)kPfTok};
  cuuint32_t es[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_UINT8, 3, const_cast<void*>(base), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE,
            codes ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// Expert engines: the block-scaled tcgen05 engine (ffn_bs.cuh) for NVFP4 and
// the FP8 tcgen05 engine (ffn_f8.cuh) for FP8.  MOE_ENGINE=mma runs both
// formats on the warp-MMA engine (ffn.cuh) instead (for comparisons).
enum Engine { kEngMma = 0, kEngBs = 1, kEngF8 = 2 };

int engine_for(int fmt) {
  static int force_mma = -1;
  if (force_mma < 0) {
    const char* s = std::getenv("MOE_ENGINE");
    force_mma = (s && std::strcmp(s, "mma") == 0) ? 1 : 0;
  }
  if (force_mma) return kEngMma;
  return fmt == MOE_FMT_NVFP4 ? kEngBs : kEngF8;
}

int act_for(int fmt, int eng) {
  if (eng == kEngBs) return kActTerms;
  if (eng == kEngF8) return kActE4M3;
  return fmt == MOE_FMT_NVFP4 ? kActF16Perm : kActF16;
}

// Token-chunk size of the expert kernels (the N side of the MMA; the
// tensor-core engines use 4 (NVFP4) or 2 (FP8) rows of N per token).
// MOE_NT overrides the choice (for measurements).
int nt_for(int T, int eng) {
  if (const char* s = std::getenv("MOE_NT")) {
    const int v = std::atoi(s);
    if (v == 8 || v == 16 || (v == 32 && eng != kEngBs)) return v;
  }
  // 8-token chunks while few experts get more tokens than that (T <= 64 with
  // top-8 of >= 128 experts); larger batches take wider chunks so that a hot
  // expert's weights are streamed fewer times.
  if (eng == kEngBs) return T <= 64 ? 8 : 16;
  if (eng == kEngF8) return T <= 64 ? 8 : 32;
  return T <= 64 ? 8 : 32;
}

// Slab order of the FP8 engine (SlabCursor, ffn.cuh) in a step whose whole
// items would not keep their weight tiles in L2: the grid's current tiles
// (KB stages of two 16 KB weight boxes per CTA) larger than the L2.  Measured
// on the 480B-shaped layer with Zipf routing at T = 256: the gate/up step
// (KB = 48, 239 MB of tiles on 152 CTAs) 839 -> 696 us with slabs of 16;
// the down step (KB = 20, 100 MB) was slower with every slab length tried
// (398 -> 517 us at 16, 612 at 8): its tiles stayed in L2 with whole items,
// and every slab end adds the chunks' partial sums out.  MOE_F8_SLAB=n sets
// the slab length (0: whole items always; for comparisons).
constexpr int kF8Slab = 16;
int f8_slab(int KB, int grid) {
  static int v = -1;
  if (v < 0) {
    const char* s = std::getenv("MOE_F8_SLAB");
    v = s ? std::atoi(s) : kF8Slab;
    if (v < 0) v = 0;
  }
  const long long tiles = (long long)grid * KB * 2 * kRowsHalf * kRowBytes;
  return tiles > device_l2_bytes() ? v : 0;
}

// Experts per router CTA: small batches spread the router rows over more
// CTAs (one expert per CTA, its row split over 8 warps); larger ones keep
// four experts per CTA so that the token rows staged in shared memory are
// reused, and eight (two rounds of four) once the grid would not fit two CTAs
// per SM: fewer waves of each CTA's fixed work (staging, activation terms,
// ticket).  Measured: 235B-shaped layer at 128 tokens 25 -> 19 us; more
// experts per CTA (16, 32) made the 480B-shaped router at 256 tokens slower.
int route_epb(int T, int E, int sms) {
  if (T <= 16) return 1;
  const int chunks = (T + kRouteTok - 1) / kRouteTok;
  return (long long)((E + 3) / 4) * chunks > 2LL * sms ? 8 : 4;
}

// Batches with T * H >= kRouteTcMinTH (E <= 256) compute the router logits on
// the tensor cores (route_tc.cu).  Measured (route and gather, us, GEMV ->
// tensor cores): H=4096 T=256 51.7 -> 60.4, T=512 76.5 -> 68.1, T=1024 125.8
// -> 81.0, T=2048 238.2 -> 134.6; H=6144 T=256 71.8 -> 70.5, T=512 114.2 ->
// 87.4.  MOE_ROUTE_TC=0 keeps every batch on the CUDA-core GEMV of
// route_kernel, MOE_ROUTE_TC=1 sends every batch with E <= 256 to the tensor
// cores (for comparisons).
constexpr long long kRouteTcMinTH = 1LL << 21;
bool use_route_tc(int T, int H, int E) {
  static int mode = -2;  // -1 default, 0 off, 1 on
  if (mode == -2) {
    const char* s = std::getenv("MOE_ROUTE_TC");
    mode = !s ? -1 : (std::strcmp(s, "0") == 0 ? 0 : (std::strcmp(s, "1") == 0 ? 1 : -1));
  }
  if (E > kRouteTcMaxE || mode == 0) return false;
  return mode == 1 || (long long)T * H >= kRouteTcMinTH;
}

// Prefill-shaped NVFP4 batches run on the prefill engine (ffn_pf.cuh);
// MOE_PF=0 keeps them on the decode engine (for comparisons).
bool use_prefill(int T, int k, int E, int eng) {
  static int off = -1;
  if (off < 0) {
    const char* s = std::getenv("MOE_PF");
    off = (s && std::strcmp(s, "0") == 0) ? 1 : 0;
  }
  return !off && eng == kEngBs && prefill_shape(T, k, E, act_for(MOE_FMT_NVFP4, eng));
}

// ------------------------------------------------------------------ validation
int check_weights(const moe_expert_weights_t* w) {
  if (!w) return MOE_ERR_INVALID_ARG;
  if (w->fmt != MOE_FMT_FP8_B128 && w->fmt != MOE_FMT_NVFP4) return MOE_ERR_INVALID_ARG;
  if (!w->w_gate || !w->w_up || !w->w_down || !w->s_gate || !w->s_up || !w->s_down)
    return MOE_ERR_INVALID_ARG;
  if (w->fmt == MOE_FMT_NVFP4 && (!w->ts_gate || !w->ts_up || !w->ts_down))
    return MOE_ERR_INVALID_ARG;
  if (w->E < 1 || w->E > kMaxE) return MOE_ERR_UNSUPPORTED_SHAPE;
  if (w->H < 256 || w->H > 8192 || w->H % 256) return MOE_ERR_UNSUPPORTED_SHAPE;
  const int imod = (w->fmt == MOE_FMT_FP8_B128) ? 128 : 256;
  if (w->I < imod || w->I > 8192 || w->I % imod) return MOE_ERR_UNSUPPORTED_SHAPE;
  if (!aligned(w->w_gate, 16) || !aligned(w->w_up, 16) || !aligned(w->w_down, 16))
    return MOE_ERR_INVALID_ARG;
  const size_t sa = (w->fmt == MOE_FMT_NVFP4) ? 16 : 4;
  if (!aligned(w->s_gate, sa) || !aligned(w->s_up, sa) || !aligned(w->s_down, sa))
    return MOE_ERR_INVALID_ARG;
  return MOE_OK;
}

int check_tk(int T, int k, int E) {
  if (T < 0 || k < 1) return MOE_ERR_INVALID_ARG;
  if (k > E || k > kMaxK) return MOE_ERR_UNSUPPORTED_SHAPE;
  if ((long long)T * k > kMaxTK) return MOE_ERR_UNSUPPORTED_SHAPE;
  return MOE_OK;
}

constexpr int kLayerFlags =
    MOE_FLAG_NO_RENORM | MOE_FLAG_PRENORM_RMS | MOE_FLAG_DETERMINISTIC | kFlagTestStall;

// Workspace of a moe_decode_layer call: the deterministic mode keeps one fp32
// down row per assignment (the prefill engine keeps them anyway).
WsLayout layer_layout(const moe_expert_weights_t* w, int T, int k, int flags) {
  return ws_layout(T, k, w->E, w->H, w->I, act_for(w->fmt, engine_for(w->fmt)),
                   (flags & MOE_FLAG_DETERMINISTIC) != 0, use_route_tc(T, w->H, w->E));
}

// ------------------------------------------------------------------ the expert steps
struct ExpertRun {
  const moe_expert_weights_t* w;
  int T, k, nt, sms;
  void* ws;
  WsLayout L;
  const int* sorted;  // assignment lists (see FfnParams::list_T)
  int list_T;
  const int* counts;  // tokens per expert
  int gathered;       // x terms already in compact-row order (xg, xgsf)
  const float* gates;
  int fused;
  float* y_perm;
  __nv_bfloat16* out;
  const __nv_bfloat16* residual;
  int test_stall;
  int det;  // deterministic mode (FfnParams::det)
};

int run_experts(const ExpertRun& r, cudaStream_t st, cudaEvent_t ev_mid) {
  const moe_expert_weights_t* w = r.w;
  const int E = w->E, H = w->H, I = w->I;
  const bool fp4 = (w->fmt == MOE_FMT_NVFP4);
  const int KEL = fp4 ? 256 : 128;
  const int hb = fp4 ? H / 2 : H, ib = fp4 ? I / 2 : I;  // bytes per row
  FfnMaps m1{}, m2{};
  bool ok = map_codes(&m1.a0, w->w_gate, E, I, hb) && map_codes(&m1.a1, w->w_up, E, I, hb) &&
            map_codes(&m2.a0, w->w_down, E, H, ib);
  m2.a1 = m2.a0;
  if (fp4) {
    ok = ok && map_sf(&m1.s0, w->s_gate, E, I, H) && map_sf(&m1.s1, w->s_up, E, I, H) &&
         map_sf(&m2.s0, w->s_down, E, H, I);
    m2.s1 = m2.s0;
  } else {
    m1.s0 = m1.s1 = m1.a0;
    m2.s0 = m2.s1 = m2.a0;
  }
  __half* x16 = ws_ptr<__half>(r.ws, r.L.x16);
  __half* h16 = ws_ptr<__half>(r.ws, r.L.h16);
  const int eng = engine_for(w->fmt);
  if (eng == kEngBs) {
    // activation terms: x rows 4t..4t+3 (one box per token) or, gathered,
    // the chunk's rows (one box of 4*nt rows); h rows of a chunk likewise
    if (r.gathered)
      ok = ok && map_2d(&m1.b, CU_TENSOR_MAP_DATA_TYPE_UINT8, ws_ptr<uint8_t>(r.ws, r.L.xg),
                        (uint64_t)H / 2, (uint64_t)hq_rows(r.T, r.k, kTerms), (uint64_t)H / 2,
                        kRowBytes, (uint32_t)(kTerms * r.nt), CU_TENSOR_MAP_SWIZZLE_128B);
    else
      ok = ok && map_2d(&m1.b, CU_TENSOR_MAP_DATA_TYPE_UINT8, ws_ptr<uint8_t>(r.ws, r.L.xq),
                        (uint64_t)H / 2, (uint64_t)r.T * kTerms, (uint64_t)H / 2, kRowBytes,
                        kTerms, CU_TENSOR_MAP_SWIZZLE_128B);
    ok = ok && map_2d(&m2.b, CU_TENSOR_MAP_DATA_TYPE_UINT8, ws_ptr<uint8_t>(r.ws, r.L.hq),
                      (uint64_t)I / 2, (uint64_t)hq_rows(r.T, r.k, kTerms), (uint64_t)I / 2,
                      kRowBytes, (uint32_t)(kTerms * r.nt), CU_TENSOR_MAP_SWIZZLE_128B);
  } else if (eng == kEngF8) {
    // E4M3 terms: x rows 2t, 2t+1 (one box per token) or gathered (one box
    // of 2*nt rows), h rows of a chunk
    if (r.gathered)
      ok = ok && map_2d(&m1.b, CU_TENSOR_MAP_DATA_TYPE_UINT8, ws_ptr<uint8_t>(r.ws, r.L.xg),
                        (uint64_t)H, (uint64_t)hq_rows(r.T, r.k, kF8Terms), (uint64_t)H,
                        kRowBytes, (uint32_t)(kF8Terms * r.nt), CU_TENSOR_MAP_SWIZZLE_128B);
    else
      ok = ok && map_2d(&m1.b, CU_TENSOR_MAP_DATA_TYPE_UINT8, ws_ptr<uint8_t>(r.ws, r.L.xq),
                        (uint64_t)H, (uint64_t)r.T * kF8Terms, (uint64_t)H, kRowBytes, kF8Terms,
                        CU_TENSOR_MAP_SWIZZLE_128B);
    ok = ok && map_2d(&m2.b, CU_TENSOR_MAP_DATA_TYPE_UINT8, ws_ptr<uint8_t>(r.ws, r.L.hq),
                      (uint64_t)I, (uint64_t)hq_rows(r.T, r.k, kF8Terms), (uint64_t)I, kRowBytes,
                      (uint32_t)(kF8Terms * r.nt), CU_TENSOR_MAP_SWIZZLE_128B);
  } else {
    ok = ok && map_2d(&m1.b, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, x16, (uint64_t)H, (uint64_t)r.T,
                      (uint64_t)H * 2, (uint32_t)KEL, 1, CU_TENSOR_MAP_SWIZZLE_NONE);
    ok = ok && map_2d(&m2.b, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, h16, (uint64_t)I,
                      (uint64_t)r.T * r.k, (uint64_t)I * 2, (uint32_t)KEL, 8,
                      CU_TENSOR_MAP_SWIZZLE_NONE);
  }
  if (!ok) return MOE_ERR_CUDA;

  FfnParams p{};
  p.T = r.T;
  p.k = r.k;
  p.E = E;
  p.H = H;
  p.I = I;
  p.counts = r.counts;
  p.sorted = r.sorted;
  p.list_T = r.list_T;
  p.gates = r.gates;
  p.status = ws_ptr<uint32_t>(r.ws, r.L.status);
  p.units = ws_ptr<uint32_t>(r.ws, r.L.units);
  p.wait_ns = wait_limit_ns();
  p.det = r.det;

  FfnParams p1 = p;
  p1.phase = 1;
  p1.s0 = static_cast<const float*>(w->s_gate);
  p1.s1 = static_cast<const float*>(w->s_up);
  p1.ts0 = w->ts_gate;
  p1.ts1 = w->ts_up;
  p1.xinv = ws_ptr<float>(r.ws, r.L.xinv);
  p1.gu = ws_ptr<float>(r.ws, r.L.gu);
  p1.h16 = h16;
  p1.hinv = ws_ptr<float>(r.ws, r.L.hinv);
  p1.bsf = ws_ptr<uint8_t>(r.ws, r.gathered ? r.L.xgsf : r.L.xsf);
  p1.b_compact = r.gathered;
  p1.hq = ws_ptr<uint8_t>(r.ws, r.L.hq);
  p1.hsf = ws_ptr<uint8_t>(r.ws, r.L.hsf);
  p1.test_stall = r.test_stall;
  p1.slab = f8_slab(H / 128, r.sms);

  FfnParams p2 = p;
  p2.phase = 2;
  p2.fused = r.fused;
  p2.s0 = static_cast<const float*>(w->s_down);
  p2.s1 = p2.s0;
  p2.ts0 = w->ts_down;
  p2.ts1 = w->ts_down;
  p2.xinv = ws_ptr<float>(r.ws, r.L.hinv);
  p2.oacc = ws_ptr<float>(r.ws, r.L.oacc);
  p2.y_perm = r.y_perm;
  p2.out = r.out;
  p2.residual = r.residual;
  p2.bsf = ws_ptr<uint8_t>(r.ws, r.L.hsf);
  p2.acnt_reset = r.list_T ? ws_ptr<uint32_t>(r.ws, r.L.acnt) : nullptr;
  p2.slab = f8_slab(I / 128, r.sms);

  auto launch = [&](const FfnMaps& m, const FfnParams& pp) {
    if (eng == kEngBs) return launch_ffn_bs(r.nt, r.sms, m, pp, st);
    if (eng == kEngF8) return launch_ffn_f8(r.nt, r.sms, m, pp, st);
    return fp4 ? launch_ffn<2>(r.nt, r.sms, m, pp, st, true)
               : launch_ffn<1>(r.nt, r.sms, m, pp, st, true);
  };
  cudaError_t err = launch(m1, p1);
  if (err != cudaSuccess) return MOE_ERR_CUDA;
  if (ev_mid && cudaEventRecord(ev_mid, st) != cudaSuccess) return MOE_ERR_CUDA;
  if (eng == kEngBs)
    err = launch_swiglu_terms(r.T * r.k, r.sms, p1, st);
  else if (eng == kEngF8)
    err = launch_swiglu_e4m3(r.T * r.k, r.sms, p1, st);
  else if (fp4)
    err = launch_swiglu<2>(r.T * r.k, r.sms, p1, true, st);  // h16 in the unit order
  else
    err = launch_swiglu<1>(r.T * r.k, r.sms, p1, false, st);
  if (err != cudaSuccess) return MOE_ERR_CUDA;
  err = launch(m2, p2);
  if (err != cudaSuccess) return MOE_ERR_CUDA;
  if (r.fused) err = launch_finalize(r.sms, p2, st);
  return err == cudaSuccess ? MOE_OK : MOE_ERR_CUDA;
}

// The expert steps of a prefill-shaped NVFP4 batch: gate/up on the prefill
// engine into the fp32 gate|up rows, SwiGLU into activation terms, down on
// the prefill engine into each assignment's row of y_perm, and the combine
// (gates, residual, bf16), which also zeroes the per-expert counters.
int run_prefill(const moe_expert_weights_t* w, int T, int k, int sms, void* ws,
                const WsLayout& L, const float* gates, const void* residual, void* out,
                int test_stall, cudaEvent_t ev_mid, cudaStream_t st) {
  const int E = w->E, H = w->H, I = w->I;
  FfnMaps m1{}, m2{};
  bool ok = map_codes(&m1.a0, w->w_gate, E, I, H / 2) && map_codes(&m1.a1, w->w_up, E, I, H / 2) &&
            map_sf(&m1.s0, w->s_gate, E, I, H) && map_sf(&m1.s1, w->s_up, E, I, H) &&
            map_terms3(&m1.b, ws_ptr<uint8_t>(ws, L.xg), H / 2, T * k, true) &&
            map_terms3(&m1.sb, ws_ptr<uint8_t>(ws, L.xgsf), H / 16, T * k, false) &&
            map_codes(&m2.a0, w->w_down, E, H, I / 2) && map_sf(&m2.s0, w->s_down, E, H, I) &&
            map_terms3(&m2.b, ws_ptr<uint8_t>(ws, L.hq), I / 2, T * k, true) &&
            map_terms3(&m2.sb, ws_ptr<uint8_t>(ws, L.hsf), I / 16, T * k, false);
  if (!ok) return MOE_ERR_CUDA;
  m2.a1 = m2.a0;
  m2.s1 = m2.s0;
  FfnParams p{};
  p.T = T;
  p.k = k;
  p.E = E;
  p.H = H;
  p.I = I;
  p.counts = ws_ptr<int>(ws, L.acnt);
  p.sorted = ws_ptr<int>(ws, L.alist);
  p.list_T = 1;
  p.b_compact = 1;
  p.gates = gates;
  p.status = ws_ptr<uint32_t>(ws, L.status);
  p.units = ws_ptr<uint32_t>(ws, L.units);
  p.wait_ns = wait_limit_ns();
  FfnParams p1 = p;
  p1.phase = 1;
  p1.ts0 = w->ts_gate;
  p1.ts1 = w->ts_up;
  p1.xinv = ws_ptr<float>(ws, L.xinv);
  p1.gu = ws_ptr<float>(ws, L.gu);
  p1.bsf = ws_ptr<uint8_t>(ws, L.xgsf);
  p1.hq = ws_ptr<uint8_t>(ws, L.hq);
  p1.hsf = ws_ptr<uint8_t>(ws, L.hsf);
  p1.hinv = ws_ptr<float>(ws, L.hinv);
  p1.test_stall = test_stall;
  FfnParams p2 = p;
  p2.phase = 2;
  p2.ts0 = w->ts_down;
  p2.ts1 = w->ts_down;
  p2.xinv = ws_ptr<float>(ws, L.hinv);
  p2.y_perm = ws_ptr<float>(ws, L.yperm);
  p2.bsf = ws_ptr<uint8_t>(ws, L.hsf);
  if (launch_ffn_pf(sms, m1, p1, st) != cudaSuccess) return MOE_ERR_CUDA;
  if (ev_mid && cudaEventRecord(ev_mid, st) != cudaSuccess) return MOE_ERR_CUDA;
  if (launch_swiglu_terms(T * k, sms, p1, st, kPfTerms) != cudaSuccess) return MOE_ERR_CUDA;
  if (launch_ffn_pf(sms, m2, p2, st) != cudaSuccess) return MOE_ERR_CUDA;
  CombineParams c{p2.y_perm, gates, ws_ptr<int>(ws, L.inv), T, k, H,
                  static_cast<const __nv_bfloat16*>(residual), static_cast<__nv_bfloat16*>(out),
                  ws_ptr<unsigned>(ws, L.acnt), E};
  return launch_combine(c, st) == cudaSuccess ? MOE_OK : MOE_ERR_CUDA;
}

}  // namespace

// ====================================================================== ABI
extern "C" {

const char* moe_status_string(int s) {
  switch (s) {
    case MOE_OK: return "MOE_OK";
    case MOE_ERR_INVALID_ARG: return "MOE_ERR_INVALID_ARG";
    case MOE_ERR_UNSUPPORTED_SHAPE: return "MOE_ERR_UNSUPPORTED_SHAPE";
    case MOE_ERR_WORKSPACE_TOO_SMALL: return "MOE_ERR_WORKSPACE_TOO_SMALL";
    case MOE_ERR_CUDA: return "MOE_ERR_CUDA";
    case MOE_ERR_DEVICE_TIMEOUT: return "MOE_ERR_DEVICE_TIMEOUT";
    case MOE_ERR_BAD_EXPERT_ID: return "MOE_ERR_BAD_EXPERT_ID";
    case MOE_ERR_UNSUPPORTED_DEVICE: return "MOE_ERR_UNSUPPORTED_DEVICE";
    default: return "MOE_ERR_UNKNOWN";
  }
}

int moe_version(void) { return kAbiVersion; }

int moe_workspace_size_flags(const moe_expert_weights_t* w, int T, int k, int flags,
                             size_t* bytes) {
  if (!bytes || (flags & ~kLayerFlags)) return MOE_ERR_INVALID_ARG;
  int rc = check_weights(w);
  if (rc) return rc;
  rc = check_tk(T, k, w->E);
  if (rc) return rc;
  *bytes = layer_layout(w, T, k, flags).total;
  return MOE_OK;
}

int moe_workspace_size(const moe_expert_weights_t* w, int T, int k, size_t* bytes) {
  return moe_workspace_size_flags(w, T, k, 0, bytes);
}

int moe_layer_kernel_count(const moe_expert_weights_t* w, int T, int k, int* count) {
  if (!count) return MOE_ERR_INVALID_ARG;
  int rc = check_weights(w);
  if (rc) return rc;
  rc = check_tk(T, k, w->E);
  if (rc) return rc;
  // (router prep and GEMM), route, (gather), gate/up, SwiGLU, down, finalize
  *count = (T == 0) ? 0
                    : 5 + (gather_terms(T, act_for(w->fmt, engine_for(w->fmt))) ? 1 : 0) +
                          (use_route_tc(T, w->H, w->E) ? 2 : 0);
  return MOE_OK;
}

int moe_route_workspace_size(int T, int E, size_t* bytes) {
  if (!bytes || T < 0) return MOE_ERR_INVALID_ARG;
  if (E < 1 || E > kMaxE) return MOE_ERR_UNSUPPORTED_SHAPE;
  *bytes = ws_layout(T, 1, E, 256, 0).logits + align_up(4 * (size_t)T * E, 256);
  return MOE_OK;
}

// The plan the kernels build in shared memory, built here by a plain scan.
static int host_plan(const int32_t* counts, int E, int NT, PlanSmem& pl, long long* assignments) {
  long long off = 0, ch = 0;
  int n = 0;
  for (int e = 0; e < E; ++e) {
    const int c = counts[e];
    if (c < 0) return MOE_ERR_INVALID_ARG;
    if (c == 0) continue;
    pl.act[n] = e;
    pl.acnt[n] = c;
    pl.aoff[n] = (int)off;
    pl.cpre[n] = (int)ch;
    off += c;
    ch += (c + NT - 1) / NT;
    ++n;
    if (off > (1 << 24)) return MOE_ERR_UNSUPPORTED_SHAPE;
  }
  pl.nA = n;
  pl.aoff[n] = (int)off;
  pl.cpre[n] = (int)ch;
  *assignments = off;
  return MOE_OK;
}

int moe_cost_split_stage(const int32_t* counts, int E, int NT, int rtiles, int KB, int a, int b,
                         long long num, long long den, int* stage) {
  if (!counts || !stage || NT < 1 || NT > 256 || rtiles < 1 || KB < 1) return MOE_ERR_INVALID_ARG;
  if (a < 1 || b < 0 || den < 1 || num < 0 || num > den) return MOE_ERR_INVALID_ARG;
  if (E < 1 || E > kMaxE) return MOE_ERR_UNSUPPORTED_SHAPE;
  PlanSmem pl;
  long long off = 0;
  const int rc = host_plan(counts, E, NT, pl, &off);
  if (rc) return rc;
  const long long ch = pl.cpre[pl.nA];
  // stage indices are int; the scaled cost prefix C * num is long long
  const long long stages = ch * rtiles * KB;
  if (stages >= (1ll << 31)) return MOE_ERR_UNSUPPORTED_SHAPE;
  if (a > (1 << 16) || b > (1 << 16)) return MOE_ERR_UNSUPPORTED_SHAPE;
  const long long C = (long long)rtiles * KB * ((long long)a * ch + (long long)b * off);
  if (C > 0 && num > (1ll << 62) / C) return MOE_ERR_UNSUPPORTED_SHAPE;
  *stage = cost_split_stage(pl, rtiles, KB, NT, a, b, num, den);
  return MOE_OK;
}

int moe_stage_order(const int32_t* counts, int E, int NT, int rtiles, int KB, int slab,
                    int s_begin, int n, int32_t* item, int32_t* kb, int32_t* run_end) {
  if (!counts || NT < 1 || NT > 256 || rtiles < 1 || KB < 1 || slab < 0 || s_begin < 0 || n < 0)
    return MOE_ERR_INVALID_ARG;
  if (n > 0 && (!item || !kb || !run_end)) return MOE_ERR_INVALID_ARG;
  if (E < 1 || E > kMaxE) return MOE_ERR_UNSUPPORTED_SHAPE;
  PlanSmem pl;
  long long off = 0;
  const int rc = host_plan(counts, E, NT, pl, &off);
  if (rc) return rc;
  const long long stages = (long long)pl.cpre[pl.nA] * rtiles * KB;
  if (stages >= (1ll << 31)) return MOE_ERR_UNSUPPORTED_SHAPE;
  if ((long long)s_begin + n > stages) return MOE_ERR_INVALID_ARG;
  if (n == 0) return MOE_OK;
  SlabCursor<1> c(pl, rtiles, KB, slab, s_begin);
  for (int i = 0; i < n; ++i, c.next()) {
    item[i] = c.it;
    kb[i] = c.kb;
    run_end[i] = c.run_end ? 1 : 0;
  }
  return MOE_OK;
}

int moe_workspace_init(void* ws, size_t ws_bytes, void* stream) {
  if (!ws) return MOE_ERR_INVALID_ARG;
  return cudaMemsetAsync(ws, 0, ws_bytes, (cudaStream_t)stream) == cudaSuccess ? MOE_OK
                                                                               : MOE_ERR_CUDA;
}

int moe_read_status(void* ws, size_t ws_bytes, int* status, void* stream) {
  if (!ws || !status || ws_bytes < 4) return MOE_ERR_INVALID_ARG;
  uint32_t word = 0;
  cudaStream_t st = (cudaStream_t)stream;
  if (cudaMemcpyAsync(&word, ws, 4, cudaMemcpyDeviceToHost, st) != cudaSuccess ||
      cudaStreamSynchronize(st) != cudaSuccess)
    return MOE_ERR_CUDA;
  if (word) {
    if (cudaMemsetAsync(ws, 0, 4, st) != cudaSuccess || cudaStreamSynchronize(st) != cudaSuccess)
      return MOE_ERR_CUDA;
  }
  if (word & (kStatusTimeoutGateUp | kStatusTimeoutDown | kStatusTimeoutRoute))
    *status = MOE_ERR_DEVICE_TIMEOUT;
  else if (word & kStatusBadExpertId)
    *status = MOE_ERR_BAD_EXPERT_ID;
  else
    *status = MOE_OK;
  return MOE_OK;
}

int moe_route_topk(const void* x, const float* router_w, const float* router_bias, int T, int H,
                   int E, int k, int renorm, int32_t* topk_ids, float* topk_w, float* logits_out,
                   void* ws, size_t ws_bytes, void* stream) {
  if (E < 1 || E > kMaxE) return MOE_ERR_UNSUPPORTED_SHAPE;
  int rc = check_tk(T, k, E);
  if (rc) return rc;
  if (T == 0) return MOE_OK;
  if (!x || !router_w || !topk_ids || !topk_w || !ws) return MOE_ERR_INVALID_ARG;
  if (H < 256 || H > 8192 || H % 256) return MOE_ERR_UNSUPPORTED_SHAPE;
  if (!aligned(x, 16) || !aligned(router_w, 16) || !aligned(ws, 256)) return MOE_ERR_INVALID_ARG;
  size_t need = 0;
  moe_route_workspace_size(T, E, &need);
  if (ws_bytes < need) return MOE_ERR_WORKSPACE_TOO_SMALL;
  if (T == 0) return MOE_OK;
  int sms = 0;
  rc = device_check(&sms);
  if (rc) return rc;
  const WsLayout L = ws_layout(T, 1, E, 256, 0);
  RouteParams p{};
  p.x = static_cast<const __nv_bfloat16*>(x);
  p.wr = router_w;
  p.bias = router_bias;
  p.T = T;
  p.H = H;
  p.E = E;
  p.k = k;
  p.renorm = renorm ? 1 : 0;
  p.fmt = 1;
  p.logits = logits_out ? logits_out : ws_ptr<float>(ws, L.logits);
  p.ids = topk_ids;
  p.gates = topk_w;
  p.chunk_cnt = ws_ptr<unsigned>(ws, L.route_chunk);
  p.epb = route_epb(T, E, sms);
  return launch_route(p, (cudaStream_t)stream) == cudaSuccess ? MOE_OK : MOE_ERR_CUDA;
}

int moe_permute(const int32_t* topk_ids, int T, int k, int E, int32_t* counts, int32_t* offsets,
                int32_t* sorted_assign, int32_t* inv_perm, int32_t* active, void* stream) {
  if (!counts || !offsets || !sorted_assign || !inv_perm || !active) return MOE_ERR_INVALID_ARG;
  if (E < 1 || E > kMaxE) return MOE_ERR_UNSUPPORTED_SHAPE;
  int rc = check_tk(T, k, E);
  if (rc) return rc;
  if (T > 0 && !topk_ids) return MOE_ERR_INVALID_ARG;
  int sms = 0;
  rc = device_check(&sms);
  if (rc) return rc;
  return launch_permute_standalone(topk_ids, T, k, E, counts, offsets, sorted_assign, inv_perm,
                                   active, (cudaStream_t)stream) == cudaSuccess
             ? MOE_OK
             : MOE_ERR_CUDA;
}

int moe_expert_ffn(const void* x, const moe_expert_weights_t* w, const int32_t* offsets,
                   const int32_t* sorted_assign, const int32_t* active, int T, int k,
                   float* y_perm, void* ws, size_t ws_bytes, void* stream) {
  int rc = check_weights(w);
  if (rc) return rc;
  rc = check_tk(T, k, w->E);
  if (rc) return rc;
  if (T == 0) return MOE_OK;
  if (!x || !offsets || !sorted_assign || !active || !y_perm || !ws) return MOE_ERR_INVALID_ARG;
  if (!aligned(x, 16) || !aligned(y_perm, 16) || !aligned(ws, 256)) return MOE_ERR_INVALID_ARG;
  const WsLayout L = ws_layout(T, k, w->E, w->H, w->I, act_for(w->fmt, engine_for(w->fmt)));
  if (ws_bytes < L.total) return MOE_ERR_WORKSPACE_TOO_SMALL;
  if (T == 0) return MOE_OK;
  int sms = 0;
  rc = device_check(&sms);
  if (rc) return rc;
  cudaStream_t st = (cudaStream_t)stream;
  const int eng = engine_for(w->fmt);
  const int nt = nt_for(T, eng);
  PrepParams pp{};
  pp.x = static_cast<const __nv_bfloat16*>(x);
  pp.T = T;
  pp.H = w->H;
  pp.E = w->E;
  pp.k = k;
  pp.fmt = w->fmt;
  pp.act = act_for(w->fmt, eng);
  pp.x16 = ws_ptr<__half>(ws, L.x16);
  pp.xq = ws_ptr<uint8_t>(ws, L.xq);
  pp.xsf = ws_ptr<uint8_t>(ws, L.xsf);
  pp.xinv = ws_ptr<float>(ws, L.xinv);
  pp.offsets = offsets;
  pp.counts = ws_ptr<int>(ws, L.counts);
  pp.zero_a = reinterpret_cast<float4*>(y_perm);
  pp.zero_a_n4 = (size_t)T * k * w->H / 4;
  pp.zero_b = ws_ptr<float4>(ws, L.gu);
  pp.zero_b_n4 = (size_t)T * k * 2 * w->I / 4;
  if (launch_prep(pp, st) != cudaSuccess) return MOE_ERR_CUDA;
  ExpertRun r{};
  r.w = w;
  r.T = T;
  r.k = k;
  r.nt = nt;
  r.sms = sms;
  r.ws = ws;
  r.L = L;
  r.sorted = sorted_assign;
  r.list_T = 0;
  r.counts = ws_ptr<int>(ws, L.counts);
  r.fused = 0;
  r.y_perm = y_perm;
  return run_experts(r, st, nullptr);
}

int moe_combine(const float* y_perm, const float* topk_w, const int32_t* inv_perm, int T, int k,
                int H, const void* residual, void* out, void* stream) {
  if (T < 0 || k < 1 || H < 4 || H % 4) return MOE_ERR_INVALID_ARG;
  if (T == 0) return MOE_OK;
  if (!y_perm || !topk_w || !inv_perm || !out) return MOE_ERR_INVALID_ARG;
  if (!aligned(y_perm, 16) || !aligned(out, 8) || (residual && !aligned(residual, 8)))
    return MOE_ERR_INVALID_ARG;
  if (T == 0) return MOE_OK;
  CombineParams p{y_perm, topk_w, inv_perm, T, k, H,
                  static_cast<const __nv_bfloat16*>(residual), static_cast<__nv_bfloat16*>(out)};
  return launch_combine(p, (cudaStream_t)stream) == cudaSuccess ? MOE_OK : MOE_ERR_CUDA;
}

int moe_decode_layer_ex(const void* x, const float* router_w, const float* router_bias,
                        const moe_expert_weights_t* w, int T, int k, int flags,
                        const void* residual, void* out, void* ws, size_t ws_bytes,
                        float* logits_out, int32_t* topk_ids_out, float* topk_w_out,
                        void* const* events, void* stream) {
  if (flags & ~kLayerFlags) return MOE_ERR_INVALID_ARG;
  int rc = check_weights(w);
  if (rc) return rc;
  rc = check_tk(T, k, w->E);
  if (rc) return rc;
  if (T == 0) return MOE_OK;  // an empty batch may come with null row pointers
  if (!x || !router_w || !out || !ws) return MOE_ERR_INVALID_ARG;
  if (!aligned(x, 16) || !aligned(router_w, 16) || !aligned(ws, 256) || !aligned(out, 8) ||
      (residual && !aligned(residual, 8)))
    return MOE_ERR_INVALID_ARG;
  if (out == x) return MOE_ERR_INVALID_ARG;
  const int E = w->E, H = w->H, I = w->I;
  const WsLayout L = layer_layout(w, T, k, flags);
  if (ws_bytes < L.total) return MOE_ERR_WORKSPACE_TOO_SMALL;
  if (T == 0) return MOE_OK;
  int sms = 0;
  rc = device_check(&sms);
  if (rc) return rc;
  cudaStream_t st = (cudaStream_t)stream;
  cudaEvent_t ev[4] = {nullptr, nullptr, nullptr, nullptr};
  if (events)
    for (int i = 0; i < 4; ++i) ev[i] = static_cast<cudaEvent_t>(events[i]);
  const int eng = engine_for(w->fmt);
  const int nt = nt_for(T, eng);
  const bool pf = use_prefill(T, k, E, eng);
  // deterministic mode of the decode engines (the prefill engine sums every
  // item in one CTA and each token's rows in the combine kernel anyway)
  const bool det = (flags & MOE_FLAG_DETERMINISTIC) && !pf;

  RouteParams p{};
  p.x = static_cast<const __nv_bfloat16*>(x);
  p.wr = router_w;
  p.bias = router_bias;
  p.T = T;
  p.H = H;
  p.E = E;
  p.k = k;
  p.renorm = (flags & MOE_FLAG_NO_RENORM) ? 0 : 1;
  p.prenorm = (flags & MOE_FLAG_PRENORM_RMS) ? 1 : 0;
  p.fmt = w->fmt;
  p.fused = 1;
  p.epb = route_epb(T, E, sms);
  p.act = act_for(w->fmt, eng);
  p.logits = logits_out ? logits_out : ws_ptr<float>(ws, L.logits);
  p.ids = ws_ptr<int>(ws, L.ids);
  p.gates = ws_ptr<float>(ws, L.gates);
  p.ids2 = topk_ids_out;
  p.gates2 = topk_w_out;
  p.chunk_cnt = ws_ptr<unsigned>(ws, L.route_chunk);
  p.x16 = ws_ptr<__half>(ws, L.x16);
  p.xq = ws_ptr<uint8_t>(ws, L.xq);
  p.xsf = ws_ptr<uint8_t>(ws, L.xsf);
  p.xinv = ws_ptr<float>(ws, L.xinv);
  // the decode engines add their partial sums into zeroed accumulators (the
  // token rows, or in the deterministic mode each assignment's row); the
  // prefill engine, and the tensor-core engines in the deterministic mode,
  // store complete sums and need none
  const bool stores = pf || (det && eng != kEngMma);
  p.zero_a = ws_ptr<float4>(ws, L.gu);
  p.zero_a_n4 = stores ? 0 : (size_t)T * k * 2 * I / 4;
  p.zero_b = ws_ptr<float4>(ws, det ? L.yperm : L.oacc);
  p.zero_b_n4 = stores ? 0 : (size_t)T * (det ? k : 1) * H / 4;
  p.acnt = ws_ptr<unsigned>(ws, L.acnt);
  p.alist = ws_ptr<int>(ws, L.alist);
  if (ev[0] && cudaEventRecord(ev[0], st) != cudaSuccess) return MOE_ERR_CUDA;
  if (use_route_tc(T, H, E)) {
    // logits on the tensor cores; route_kernel adds the slices and routes
    RouteTcParams q{};
    q.wr = router_w;
    q.x = p.x;
    q.xn = ws_ptr<__nv_bfloat16>(ws, L.xn);
    q.w3 = ws_ptr<__nv_bfloat16>(ws, L.w3);
    q.plog = ws_ptr<float>(ws, L.plog);
    q.T = T;
    q.H = H;
    q.E = E;
    q.Ep = route_tc_ep(E);
    q.prenorm = p.prenorm;
    q.act = p.act;
    q.xq = p.xq;
    q.xsf = p.xsf;
    q.xinv = p.xinv;
    q.status = ws_ptr<uint32_t>(ws, L.status);
    q.wait_ns = wait_limit_ns();
    CUtensorMap ta, tb;
    if (!map_2d(&ta, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, q.prenorm ? (const void*)q.xn : x,
                (uint64_t)H, (uint64_t)T, (uint64_t)H * 2, 64, 128, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !map_2d(&tb, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, q.w3, (uint64_t)H, 3 * (uint64_t)q.Ep,
                (uint64_t)H * 2, 64, (uint32_t)q.Ep, CU_TENSOR_MAP_SWIZZLE_128B))
      return MOE_ERR_CUDA;
    if (launch_router_prep(q, st) != cudaSuccess || launch_route_tc(ta, tb, q, st) != cudaSuccess)
      return MOE_ERR_CUDA;
    p.plog = q.plog;
    p.nsplit = kRouteTcSplit;
    p.ep = q.Ep;
    // without the GEMV a CTA's work is the chunk's staging, its share of the
    // activation terms and of the zeroing, and the partial sums of its
    // experts: about one wave of CTAs, each chunk's experts split between them
    const int chunks = (T + kRouteTok - 1) / kRouteTok;
    int per = (sms + chunks - 1) / chunks;
    per = per < 1 ? 1 : (per > (E + 3) / 4 ? (E + 3) / 4 : per);
    p.epb = (E + per - 1) / per;
    if (p.act == kActTerms || p.act == kActE4M3) {
      p.terms_done = 1;  // the prep kernel wrote the activation terms
    } else if (p.prenorm) {  // the router kernel stages the normalised rows
      p.x = q.xn;
    }
    p.prenorm = 0;
  }
  if (launch_route(p, st) != cudaSuccess) return MOE_ERR_CUDA;
  const bool gathered = gather_terms(T, p.act);
  if (gathered) {
    const bool fp4 = (p.act == kActTerms);
    GatherParams g{};
    g.q = p.xq;
    g.sf = fp4 ? p.xsf : nullptr;
    g.gq = ws_ptr<uint8_t>(ws, L.xg);
    g.gsf = ws_ptr<uint8_t>(ws, L.xgsf);
    g.acnt = p.acnt;
    g.alist = p.alist;
    g.T = T;
    g.k = k;
    g.E = E;
    g.terms = fp4 ? kTerms : kF8Terms;
    g.qrow = fp4 ? H / 2 : H;
    g.sfrow = H / 16;
    g.inv = pf ? ws_ptr<int>(ws, L.inv) : nullptr;
    g.status = ws_ptr<uint32_t>(ws, L.status);
    g.wait_ns = wait_limit_ns();
    if (launch_gather(g, st) != cudaSuccess) return MOE_ERR_CUDA;
  }
  if (ev[1] && cudaEventRecord(ev[1], st) != cudaSuccess) return MOE_ERR_CUDA;
  if (pf) {
    rc = run_prefill(w, T, k, sms, ws, L, p.gates, residual, out,
                     (flags & kFlagTestStall) ? 1 : 0, ev[2], st);
    if (rc) return rc;
    if (ev[3] && cudaEventRecord(ev[3], st) != cudaSuccess) return MOE_ERR_CUDA;
    return MOE_OK;
  }

  ExpertRun r{};
  r.w = w;
  r.T = T;
  r.k = k;
  r.nt = nt;
  r.sms = sms;
  r.ws = ws;
  r.L = L;
  r.sorted = p.alist;
  r.list_T = 1;
  r.gathered = gathered ? 1 : 0;
  r.counts = reinterpret_cast<const int*>(p.acnt);
  r.gates = p.gates;
  r.fused = det ? 0 : 1;  // deterministic: down rows by assignment, then the combine
  r.y_perm = det ? ws_ptr<float>(ws, L.yperm) : nullptr;
  r.det = det ? 1 : 0;
  r.out = static_cast<__nv_bfloat16*>(out);
  r.residual = static_cast<const __nv_bfloat16*>(residual);
  r.test_stall = (flags & kFlagTestStall) ? 1 : 0;
  rc = run_experts(r, st, ev[2]);
  if (rc) return rc;
  if (det) {
    // a token's k rows in the order j = 0..k-1; also zeroes the counters
    CombineParams c{r.y_perm, p.gates, nullptr, T, k, H,
                    static_cast<const __nv_bfloat16*>(residual), static_cast<__nv_bfloat16*>(out),
                    p.acnt, E};
    if (launch_combine(c, st) != cudaSuccess) return MOE_ERR_CUDA;
  }
  if (ev[3] && cudaEventRecord(ev[3], st) != cudaSuccess) return MOE_ERR_CUDA;
  return MOE_OK;
}

int moe_decode_layer(const void* x, const float* router_w, const float* router_bias,
                     const moe_expert_weights_t* w, int T, int k, int flags, const void* residual,
                     void* out, void* ws, size_t ws_bytes, void* stream) {
  return moe_decode_layer_ex(x, router_w, router_bias, w, T, k, flags, residual, out, ws,
                             ws_bytes, nullptr, nullptr, nullptr, nullptr, stream);
}

}  // extern "C"
