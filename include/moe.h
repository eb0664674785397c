/*
 * moe.h - C ABI of libmoe.so: one decode step of a Mixture-of-Experts FFN
 * layer on one GB300 GPU (sm_103a).
 *
 * The operation is the decode-lane work of the paper's served MoE models
 * (Qwen3-Coder-480B FP8 and Qwen3-235B-A22B NVFP4, Section 4 "Setup"); the
 * paper states that decode is weight-read bound (Section 2.1) and that MoE
 * sparsity leaves the decode lane under-saturated (Appendix A.3).  The paper
 * gives no kernel or number format for it; the numeric readings below are
 * this library's.
 *
 *   logits[t,e] = sum_h x[t,h] * Wr[e,h] (+ bias[e])          fp32
 *   ids[t,:]    = top-k of logits[t,:], by (value desc, index asc)
 *   w[t,j]      = exp(l_j - l_max) / sum_{i in top-k} exp(l_i - l_max)
 *   h           = silu(x_t Wg_e^T) * (x_t Wu_e^T),  silu(z) = z / (1 + e^-z)
 *   y           = h Wd_e^T
 *   out[t]      = bf16( sum_j w[t,j] * y_{t,ids[t,j]}  (+ residual[t]) )
 *
 * Conventions shared by every entry point
 * - Pointers named x, out, residual point to bf16 data (IEEE binary32 top
 *   halves); every other pointer has the element type stated.  All data
 *   pointers are DEVICE pointers unless a comment says otherwise.
 * - Row-major, innermost index contiguous.  T tokens, H hidden, E experts,
 *   k experts per token, I expert intermediate size.
 * - `stream` is a cudaStream_t (NULL = the legacy default stream).  Every
 *   call only enqueues work on it and returns; nothing synchronises.
 * - The caller owns every buffer.  The library allocates no device memory.
 * - Return value: MOE_OK (0) or a negative moe_status_t.  Argument errors
 *   are detected on the host before anything is enqueued.  Errors detected
 *   by a running kernel (a bounded wait that expired, an expert id out of
 *   range) are recorded in a status word inside the workspace and read
 *   with moe_read_status().  No exception or abort crosses the ABI.
 *
 * Arithmetic of the GPU path: fp32 router and gates; expert products
 * accumulate in fp32.  Large batches compute the router logits on the tensor
 * cores from the fp32 router split exactly into three bf16 parts (every
 * product exact in fp32, fp32 accumulation: the fp32 GEMV up to the order of
 * its additions).  Both formats feed their weights to the tensor cores
 * as stored, and the activations (x, and h between the gate/up and down
 * steps) are encoded in the weights' format family:
 * - NVFP4: block-scaled MMA (E2M1 x UE4M3 per 16 K); each activation row is
 *   a sum of four NVFP4 terms, each term coding the previous terms'
 *   residual, which leaves less than 2^-9.5 of each 16-element block's
 *   maximum uncoded.
 * - FP8: E4M3 x E4M3 MMA per 128-K block, the block scales applied in fp32;
 *   each activation row is two E4M3 terms, hi = e4m3(v) and lo = e4m3(v -
 *   hi), after a power-of-two row scale.
 * The environment variable MOE_ENGINE=mma selects instead a warp-MMA engine
 * that decodes the weights exactly to f16 and multiplies them with exact f16
 * activations (bf16 inputs after a power-of-two row scale).
 *
 * Environment (read by the library; none is needed):
 *   MOE_ENGINE=mma        the warp-MMA engine above (read once per process)
 *   MOE_NT=8|16|32        token-chunk width of the expert kernels instead of
 *                         the default (8 up to 64 tokens, else 16 for NVFP4
 *                         and 32 for FP8); 32 is not taken for NVFP4
 *   MOE_WAIT_LIMIT_MS=n   limit in ms of every bounded device wait, 1-60000
 *                         (default 1000; read once per process)
 *   MOE_PF=0              prefill-shaped NVFP4 batches (T > 64, T*k >= 32*E)
 *                         stay on the decode engine instead of the prefill
 *                         engine (read once per process)
 *   MOE_ROUTE_TC=0|1      router logits on the CUDA cores for every batch (0),
 *                         or on the tensor cores for every batch with E <= 256
 *                         (1), instead of the tensor cores from T*H >= 2^21
 *                         (read once per process)
 *   MOE_F8_SLAB=n         K-blocks per slab of the FP8 engine's experts with
 *                         several 32-token chunks (T > 64), in a step whose
 *                         whole items' weight tiles exceed the L2 (default 16;
 *                         0 keeps whole items; read once per process)
 *
 * Expert weight formats (moe_expert_weights_t)
 *   gate and up are [E, I, H]-shaped (N = I rows, K = H contiguous),
 *   down is [E, H, I]-shaped (N = H rows, K = I contiguous).
 * - MOE_FMT_FP8_B128: codes are OCP OFP8 E4M3 bytes [E, N, K]; scales are
 *   float32 [E, N/128, K/128], one per 128x128 tile; W = e4m3(code)*scale.
 *   Codes 0x7F/0xFF (NaN) must not occur.
 * - MOE_FMT_NVFP4: codes are OCP E2M1 nibbles, two per byte [E, N, K/2]
 *   (low nibble = even K index); scales are E4M3 bytes [E, N, K/16], one per
 *   16 consecutive K elements; ts_* are float32 [E], one per expert matrix;
 *   W = e2m1(code) * e4m3(scale) * ts.
 *
 * Supported shapes: H % 256 == 0; I % 128 == 0 (FP8) or I % 256 == 0
 * (NVFP4); 1 <= k <= min(E, 32); E <= 512; 0 <= T; T*k <= 65536; H, I <= 8192.
 * T == 0 is a no-op.  Anything else returns MOE_ERR_UNSUPPORTED_SHAPE.
 */
#ifndef MOE_H_
#define MOE_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  MOE_OK = 0,
  MOE_ERR_INVALID_ARG = -1,        /* null pointer, negative size, bad flag */
  MOE_ERR_UNSUPPORTED_SHAPE = -2,  /* shape outside the supported set above */
  MOE_ERR_WORKSPACE_TOO_SMALL = -3,
  MOE_ERR_CUDA = -4,               /* a CUDA runtime call or launch failed */
  MOE_ERR_DEVICE_TIMEOUT = -5,     /* a kernel's bounded wait expired */
  MOE_ERR_BAD_EXPERT_ID = -6,      /* moe_permute met an id outside [0, E) */
  MOE_ERR_UNSUPPORTED_DEVICE = -7  /* not an sm_103 (GB300) device */
} moe_status_t;

typedef enum { MOE_FMT_FP8_B128 = 1, MOE_FMT_NVFP4 = 2 } moe_format_t;

/* Flags of moe_decode_layer. */
#define MOE_FLAG_NO_RENORM 0x1   /* gates = full-softmax probabilities at the top-k */
#define MOE_FLAG_PRENORM_RMS 0x2 /* route and run the experts on bf16(RMSNorm(x)),
                                    unit weight, eps 1e-6; residual is still added */
#define MOE_FLAG_DETERMINISTIC 0x4 /* the same output bits on every run: see
                                      moe_decode_layer */

/* The expert weights of one layer.  All pointers are device pointers to the
 * caller's buffers; the struct itself is read on the host during the call. */
typedef struct {
  int fmt; /* moe_format_t */
  int E, H, I;
  const uint8_t *w_gate, *w_up, *w_down;
  const void *s_gate, *s_up, *s_down;     /* float32 (FP8) or uint8 E4M3 (NVFP4) */
  const float *ts_gate, *ts_up, *ts_down; /* NVFP4 only; NULL for FP8 */
} moe_expert_weights_t;

/* Human-readable name of a status code.  Never NULL; static storage. */
const char* moe_status_string(int status);

/* ABI version (major*10000 + minor*100 + patch). */
int moe_version(void);

/* Bytes of device workspace needed by moe_decode_layer / moe_expert_ffn for
 * these weights and T tokens with k experts each (*bytes, host pointer).
 * Pure host computation. */
int moe_workspace_size(const moe_expert_weights_t* w, int T, int k, size_t* bytes);

/* As moe_workspace_size, for a moe_decode_layer call with these flags
 * (MOE_FLAG_*): MOE_FLAG_DETERMINISTIC adds T*k*H*4 bytes (one fp32 down row
 * per assignment) unless the batch already keeps them; the other flags add
 * nothing.  MOE_ERR_INVALID_ARG for an unknown flag bit. */
int moe_workspace_size_flags(const moe_expert_weights_t* w, int T, int k, int flags,
                             size_t* bytes);

/* Kernels one moe_decode_layer call launches for these weights and T tokens
 * with k experts each (*count, host pointer): the router, the gather of the
 * activation terms (tensor-core engines, T > 64), gate/up, SwiGLU, down and
 * the bf16 finalize.  0 for T = 0.  Pure host computation; errors as
 * moe_workspace_size. */
int moe_layer_kernel_count(const moe_expert_weights_t* w, int T, int k, int* count);

/* Bytes of device workspace needed by moe_route_topk for T tokens, E experts. */
int moe_route_workspace_size(int T, int E, size_t* bytes);

/* How the tensor-core expert kernels divide their stages between CTAs: the
 * first stage that begins at or after the fraction num / den of the layer's
 * total cost.  Runs the kernels' own split function on the host, on the plan
 * the kernels build from the per-expert token counts.  Pure host computation;
 * a diagnostic for tests and tuning, not a step of the decode layer.
 *   counts [E] int32, host: tokens per expert (the plan lists the experts with
 *     tokens in increasing id order).
 *   Stage order: active expert, row tile (rtiles of them), chunk of NT tokens,
 *     K-block (KB of them).  A stage of a chunk with n tokens costs a + b * n.
 *   *stage (host): the first stage s whose preceding stages cost at least
 *     floor(C * num / den), C the total cost; 0 for num = 0, every stage for
 *     num = den.
 *   MOE_ERR_INVALID_ARG: null pointer, negative count, NT outside [1, 256],
 *     rtiles, KB or a below 1, b below 0, den below 1, num outside [0, den].
 *   MOE_ERR_UNSUPPORTED_SHAPE: E outside [1, 512], 2^31 stages or more, more
 *     than 2^24 tokens, a or b above 2^16, or C * num above 2^62. */
int moe_cost_split_stage(const int32_t* counts, int E, int NT, int rtiles, int KB, int a, int b,
                         long long num, long long den, int* stage);

/* The order in which the FP8 tensor-core kernel walks its stages: stages
 * s_begin .. s_begin + n - 1 of the sequence, as the kernel's own cursor
 * gives them, run on the host on the plan built from the counts.  Pure host
 * computation; a diagnostic for tests, not a step of the decode layer.
 *   Each (active expert, row tile) group holds the same stages as in
 *   moe_cost_split_stage's order and keeps its place in the sequence.  Inside
 *   a group whose expert has several chunks of NT tokens, the K-blocks are cut
 *   into slabs of `slab` K-blocks (the last one shorter when slab does not
 *   divide KB), and every chunk runs over one slab, K-blocks in order, before
 *   any chunk runs over the next.  A group of one chunk, or slab = 0 or
 *   slab >= KB, keeps the item order: chunk, then K-block.
 *   item[i] (host, int32): the item (active expert, row tile, chunk), numbered
 *     as in moe_cost_split_stage's order (chunk fastest); kb[i] its K-block;
 *     run_end[i] = 1 on the last stage of a chunk's run within its slab,
 *     where the kernel adds that chunk's partial sums out, else 0.
 *   MOE_ERR_INVALID_ARG: null pointer (the outputs may be null when n = 0),
 *     negative count, NT outside [1, 256], rtiles or KB below 1, slab, s_begin
 *     or n negative, or s_begin + n past the last stage.
 *   MOE_ERR_UNSUPPORTED_SHAPE: E outside [1, 512], more than 2^24 tokens or
 *     2^31 stages or more. */
int moe_stage_order(const int32_t* counts, int E, int NT, int rtiles, int KB, int slab,
                    int s_begin, int n, int32_t* item, int32_t* kb, int32_t* run_end);

/* Zero a workspace (cudaMemsetAsync).  A workspace must be zeroed once
 * before its first use; the library keeps it consistent afterwards (its
 * counters are reset by their last user).  After moe_read_status() reports
 * an error, zero it again before the next call. */
int moe_workspace_init(void* ws, size_t ws_bytes, void* stream);

/* Copy the device status word of a workspace to *status (host pointer) and
 * clear it.  Synchronises `stream`.  *status is MOE_OK or the negative code
 * of the first device-side error since the last read. */
int moe_read_status(void* ws, size_t ws_bytes, int* status, void* stream);

/* Router GEMV, softmax and top-k (steps a1-a2 of the decode layer).
 *   x [T, H] bf16; router_w [E, H] float32; router_bias [E] float32 or NULL.
 *   topk_ids [T, k] int32, topk_w [T, k] float32: outputs, column j is the
 *     j-th largest logit (ties to the lower expert index).
 *   logits_out [T, E] float32 or NULL: the fp32 logits the selection used.
 *   renorm: 1 = gates renormalised over the top-k, 0 = full-softmax values.
 *   ws: workspace of at least moe_route_workspace_size() bytes. */
int moe_route_topk(const void* x, const float* router_w, const float* router_bias, int T, int H,
                   int E, int k, int renorm, int32_t* topk_ids, float* topk_w, float* logits_out,
                   void* ws, size_t ws_bytes, void* stream);

/* Token-to-expert permutation (step a3).  Assignment a = t*k + j.
 *   topk_ids [T, k] int32 in [0, E) (out-of-range ids are skipped and
 *     reported as MOE_ERR_BAD_EXPERT_ID through `ws`-less status: the call
 *     writes -1 into active[0]).
 *   counts [E]: assignments per expert; offsets [E+1]: exclusive prefix sum;
 *   sorted_assign [T*k]: assignments sorted stably by expert;
 *   inv_perm [T*k]: position of each assignment in sorted_assign;
 *   active [E+1]: active[0] = number of experts with counts > 0, then their
 *     ids in increasing order. */
int moe_permute(const int32_t* topk_ids, int T, int k, int E, int32_t* counts, int32_t* offsets,
                int32_t* sorted_assign, int32_t* inv_perm, int32_t* active, void* stream);

/* Expert FFN over permuted assignments (steps a4-a5), no gating.
 *   x [T, H] bf16; w: expert weights; offsets, sorted_assign, active as
 *   produced by moe_permute for the same T, k, E.
 *   y_perm [T*k, H] float32 output: row p = expert ids[sorted_assign[p]]
 *     applied to token sorted_assign[p] / k.
 *   ws: workspace of at least moe_workspace_size(w, T, k) bytes. */
int moe_expert_ffn(const void* x, const moe_expert_weights_t* w, const int32_t* offsets,
                   const int32_t* sorted_assign, const int32_t* active, int T, int k,
                   float* y_perm, void* ws, size_t ws_bytes, void* stream);

/* Gate-weighted combine (step a6).
 *   out[t, :] = bf16( sum_j topk_w[t, j] * y_perm[inv_perm[t*k + j], :]
 *                     (+ residual[t, :]) ),  round to nearest even.
 *   residual [T, H] bf16 or NULL; out [T, H] bf16 (may alias residual). */
int moe_combine(const float* y_perm, const float* topk_w, const int32_t* inv_perm, int T, int k,
                int H, const void* residual, void* out, void* stream);

/* The whole decode layer (steps a1-a6) in three kernels on `stream`.
 *   x [T, H] bf16; router_w [E, H] float32; router_bias [E] float32 or NULL;
 *   w: expert weights (w->H must equal the row length of x and router_w);
 *   flags: MOE_FLAG_*; residual [T, H] bf16 or NULL (may alias out);
 *   out [T, H] bf16, must not alias x;
 *   alignment: x and router_w 16 bytes, out and residual 8 bytes, ws 256 bytes;
 *   ws: at least moe_workspace_size_flags(w, T, k, flags) bytes, zeroed
 *   once before first use (moe_workspace_init).
 * Reproducibility.  The expert kernels split the work of an expert's row tile
 * over K between CTAs, and the partial sums meet in fp32 atomic adds, as do
 * the k expert rows of a token; the order of those adds varies from run to
 * run, and so may the last bits of `out`.  MOE_FLAG_DETERMINISTIC removes
 * every such order: each (expert, 128-row tile, token chunk) is summed over
 * its whole K range by one CTA (CTA shares end on those boundaries), each
 * assignment's down row is written to its own fp32 row, and a combine kernel
 * adds a token's k rows in the order j = 0..k-1.  The same call then gives
 * the same bits on every run, whatever the stream, the concurrent work or the
 * order in which the routing lists an expert's tokens.  It costs the larger
 * workspace and a less even division of the stages between the SMs (most at
 * T = 1, where few items meet many SMs). */
int moe_decode_layer(const void* x, const float* router_w, const float* router_bias,
                     const moe_expert_weights_t* w, int T, int k, int flags, const void* residual,
                     void* out, void* ws, size_t ws_bytes, void* stream);

/* moe_decode_layer plus optional observation points, for tests and timing.
 *   logits_out [T, E] float32, topk_ids_out [T, k] int32, topk_w_out [T, k]
 *   float32: copies of the routing the layer used (each may be NULL).
 *   events: NULL, or 4 cudaEvent_t handles recorded on `stream` before the
 *   route kernel, before the gate/up kernel, before the down kernel and
 *   after it. */
int moe_decode_layer_ex(const void* x, const float* router_w, const float* router_bias,
                        const moe_expert_weights_t* w, int T, int k, int flags,
                        const void* residual, void* out, void* ws, size_t ws_bytes,
                        float* logits_out, int32_t* topk_ids_out, float* topk_w_out,
                        void* const* events, void* stream);

/* moe_decode_layer without a caller-provided workspace, for callers that must
 * not allocate device memory when they run the layer (for example an
 * inference engine's plugin enqueue path, which gets a stream and its tensors
 * but no allocator, or a serving loop that cannot afford a cudaMalloc that may
 * synchronise the device).  The paper has no counterpart of this call.
 *   Arguments as moe_decode_layer, minus ws / ws_bytes.
 *   Scratch: a 16 MiB device array inside libmoe.so; every GPU that loads the
 *     library holds it until the process exits.  Shapes whose
 *     moe_workspace_size_flags() exceeds 16 MiB return MOE_ERR_WORKSPACE_TOO_SMALL:
 *     the 235B-shaped NVFP4 layer (H=4096, E=128, k=8, I=1536) fits up to
 *     T = 74 tokens, the 480B-shaped FP8 layer (H=6144, E=160, k=8, I=2560)
 *     up to T = 64; with MOE_FLAG_DETERMINISTIC up to T = 59 and T = 38.
 *   The first call on a device looks up the array's device address and
 *     clears the array's status word; make that first call before capturing
 *     the stream into a CUDA graph.  A lookup that fails returns MOE_ERR_CUDA
 *     and is tried again by the next call.
 *   Every call shares the one array and clears its counters itself; calls
 *     that overlap on the GPU (two streams, or two host threads) race and must
 *     be serialised by the caller.
 *   Device-side errors (an expired bounded wait) are recorded in the array's
 *     status word; read them with moe_noalloc_read_status().
 *   Allocates nothing: no cudaMalloc, no cudaFree. */
int moe_decode_layer_noalloc(const void* x, const float* router_w, const float* router_bias,
                             const moe_expert_weights_t* w, int T, int k, int flags,
                             const void* residual, void* out, void* stream);

/* The device status word of moe_decode_layer_noalloc's array on the current
 * device, as moe_read_status does for a workspace: *status (host pointer)
 * gets MOE_OK or the code of the first device-side error of any
 * moe_decode_layer_noalloc call since the last read, and the word is
 * cleared.  Synchronises `stream`.  Allocates nothing.  The paper has no
 * counterpart of this call. */
int moe_noalloc_read_status(int* status, void* stream);

#ifdef __cplusplus
}
#endif
#endif /* MOE_H_ */
