/*
 * moeca.h -- C ABI of the GB300 branch-cached MoE layer stack (MoECa).
 *
 * One call of moeca_step() runs a stack of L DiT-MoE expert layers for one
 * denoising step with branch-level feature reuse:
 *   route (Eq. 7) -> EMA statistic, entropy, per-expert threshold (Eq. 10-12)
 *   -> match each routed (token, expert) branch against the token's cached
 *   branches, score it and decide recompute / reuse (Sec. 4.2, Eq. 9)
 *   -> run the expert FFN only on recomputed branches (Eq. 5 / Eq. 6)
 *   -> combine fresh and cached branch outputs with the current gate weights
 *   and add the residual (Eq. 8) -> refresh the cached branch norms.
 * Full-computation and cache steps alternate as in Sec. 4.1.
 * With n_heads > 0 every layer is a DiT-MoE block: a multi-head
 * self-attention sub-layer, whose output a_i is cached beside the branches,
 * runs before the MoE sub-layer.  On a cache step a token recomputes its
 * attention exactly when its recompute set is non-empty (Sec. 4.1, the
 * synchronized MoE / attention update); the decision is taken on
 * u'_i = x_i + a_i^{t0}, and a token that recomputes continues with
 * u_i = x_i + a_i^t.
 *
 * Conventions
 *  - All tensors are row-major.  "device" pointers are CUDA global memory of
 *    the handle's device; "host" pointers are ordinary host memory.
 *  - Weights and activation buffers are BORROWED: the caller owns them and
 *    keeps them alive (weights for the handle's lifetime).  The library owns
 *    every state and workspace buffer it allocates in moeca_create().
 *  - Every function returns a moeca_status; none throws or aborts.  Kernels
 *    never trap: a device-side problem (an index out of range, a bounded wait
 *    that ran out) is written to a status word that the next moeca_step()
 *    or moeca_get_stats() reports as MOECA_ERR_DEVICE_STATUS / _TIMEOUT.
 *  - Calls that take a `stream` enqueue work on that cudaStream_t (NULL = the
 *    legacy default stream) and return without waiting for the GPU.
 *  - A handle is not thread-safe; use one handle per host thread.
 */
#ifndef MOECA_H_
#define MOECA_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct moeca_handle moeca_handle; /* opaque, owned by the library */

typedef enum {
  MOECA_OK = 0,
  MOECA_ERR_INVALID_ARG = -1,   /* bad pointer, size, alias or config value     */
  MOECA_ERR_UNSUPPORTED = -2,   /* valid but not built (e.g. D not a multiple of 64 on bf16) */
  MOECA_ERR_CUDA = -3,          /* a CUDA runtime call failed (see moeca_last_error) */
  MOECA_ERR_OOM = -4,           /* device allocation failed                       */
  MOECA_ERR_STATE = -5,         /* call not valid in the handle's state           */
  MOECA_ERR_TIMEOUT = -6,       /* a bounded device wait ran out                  */
  MOECA_ERR_DEVICE_STATUS = -7  /* a kernel flagged bad data (index out of range) */
} moeca_status;

typedef enum {
  MOECA_F32 = 0,  /* fp32 storage, fp32 FFMA everywhere (debug-precision path)   */
  MOECA_BF16 = 1  /* bf16 activations/weights/cache, fp32 accumulation and logic */
} moeca_dtype;

typedef enum {
  MOECA_FFN_AUTO = 0, /* tcgen05 tensor-core grouped GEMM for bf16, SIMT for fp32 */
  MOECA_FFN_SIMT = 1  /* CUDA-core grouped GEMM for both dtypes (cross-check path) */
} moeca_ffn_impl;

/* Shapes, hyper-parameters and the readings of points the paper leaves open. */
typedef struct {
  int32_t n_layers;    /* L >= 1                                                  */
  int32_t hidden;      /* D: multiple of 8 (fp32: 4); bf16 tensor path: of 64     */
  int32_t ffn;         /* F: expert FFN width; bf16 tensor path: multiple of 64   */
  int32_t n_experts;   /* E routed experts, 1..64                                  */
  int32_t top_k;       /* k, 1..8 and <= E                                         */
  int32_t n_shared;    /* always-on shared experts (Eq. 6): 0 or 1, width F        */
  int32_t max_tokens;  /* largest T = batch * tokens a step may carry (>= 1)      */
  int32_t dtype;       /* moeca_dtype                                              */
  float lambda1;       /* Eq. 9 weight of the temporal drift Delta                 */
  float lambda2;       /* Eq. 9 weight of the historical contribution o            */
  float tau0;          /* Eq. 12 base threshold (may be +-inf)                     */
  float alpha;         /* Eq. 12 expert adaptation strength, [0, 1)                */
  float beta;          /* Eq. 10 EMA decay, [0, 1)                                 */
  int32_t refresh_period;     /* N: full-computation step when step % N == 0 (0: only step 0 / forced) */
  int32_t renorm_topk;        /* 1: top-k gate weights renormalised to sum 1 (default) */
  int32_t entropy_norm;       /* 0: Hbar = H / ln T (default); 1: min-max over the layer's experts */
  int32_t shared_policy;      /* 0: shared expert recomputed iff the token's recompute set is
                                 non-empty or the step is full (Sec. 4.1 sync rule, default); 1: always */
  int32_t reused_meta_policy; /* 0: a reused slot keeps w^{t0} (default); 1: it takes w^t */
  int32_t gelu_tanh;          /* 1: tanh-form GELU (default); 0: erf form */
  int32_t ffn_impl;           /* moeca_ffn_impl */
  int32_t ffn_tile_n;         /* tensor-core FFN tile width: 0 = chosen per launch from the group
                                 sizes (default), else 64 / 128 / 192 / 256 where it divides N */
  int32_t ffn_split_k;        /* tensor-core FFN K splits: 0 = chosen per launch (default), else 1..4 */
  int32_t score_terms;        /* Eq. 9 terms in the branch score, a bit mask (Table 5's signal
                                 ablation): 1 = w, 2 = lambda1 Delta, 4 = lambda2 o; 7 (default) = all */
  int32_t granularity;        /* 0: branch-level decisions (MoECa, default); 1: token-level, a
                                 token's k branches share one decision: all are recomputed when
                                 the branch rule would recompute any of them (Sec. 3) */
  int32_t n_heads;            /* 0 (default): each layer is the MoE sub-layer alone; H > 0: each
                                 layer is a DiT-MoE block whose attention sub-layer has H heads of
                                 D / H (64, 72, 80, 96 or 128) channels; bf16 only */
  int32_t seq_len;            /* token rows per sample: attention runs within each run of seq_len
                                 consecutive rows (0: all T rows are one sample); T must be a
                                 multiple of it and it a multiple of 8 */
  int32_t attn_policy;        /* attention output on cache steps: 0 = recomputed for the tokens
                                 with a non-empty recompute set (Sec. 4.1 sync rule, default);
                                 1 = reused for every token ("without sync update", Table 4);
                                 2 = recomputed for every token, routing on the fresh input */
  int32_t attn_impl;          /* attention core: 0 = chosen per sample length (default: tcgen05 /
                                 TMEM kernel from 512 tokens per sample, warp-level mma.sync kernel
                                 below, where a CTA sees too few key blocks to fill its pipeline);
                                 1 = mma.sync kernel; 2 = tcgen05 kernel */
  int32_t adaln;              /* 1: each DiT-MoE block (n_heads > 0) enters both sub-layers through
                                 AdaLN, the residual form x + AdaLN o f(x) of Sec. 3 in DiT's shape:
                                 per sample b, SiLU(c_b) w_ada^T + b_ada gives six D-vectors
                                 (shift_a, scale_a, gate_a, shift_m, scale_m, gate_m);
                                 h = LN(x)(1 + scale_a) + shift_a, a = Attn(h),
                                 u = x + gate_a a, m = LN(u)(1 + scale_m) + shift_m,
                                 out = u + gate_m MoE(m); LN over D without affine parameters.
                                 The caches hold the ungated a and branch outputs, every step
                                 applies its own modulation, and under the sync rule the router
                                 sees m' from u' = x + gate_a a^{t0}.  moeca_step_args.cond then
                                 carries c.  bf16 only; hidden <= 2560; (max_tokens / seq_len) x
                                 hidden x 4 bytes <= 200 KB (the staged conditioning), else
                                 MOECA_ERR_UNSUPPORTED at create.  0 (default): no normalisation
                                 or modulation */
  float ln_eps;               /* AdaLN layer-normalisation epsilon (default 1e-6) */
  int32_t keep_route_in;      /* 1: keep each AdaLN block's router input (m' on sync cache steps)
                                 for moeca_get_layer_trace, one more [T, D] write per layer;
                                 0 (default) */
  int32_t token_reuse_policy; /* what a token whose recompute set R_i is empty returns on a cache
                                 step: 0 (default) = Eq. 8, its cached branch outputs combined with
                                 the current gate weights w^t; 1 = Sec. 4.1's "reuse cached states"
                                 read at token level: its last computed MoE output y^{t0} (routed
                                 branches and shared expert, before the AdaLN gate) unchanged.
                                 1 keeps y for every token: one [T, D] fp32 buffer per layer
                                 (moeca_layer_state.cache_y), written by every token that computes */
  int32_t combine_direct;     /* Eq. 8 combine kernel form: 1 (default) = direct, one warp per
                                 token, the lanes load the rows themselves; 0 = staged where a
                                 warp's two token buffers take at most 24 KB, each warp bringing a
                                 token's rows into shared memory with bulk copies while it combines
                                 the previous one (the direct form otherwise, and always under the
                                 token-level reading above).  Both give the same bits */
  int32_t weight_prefetch_mb; /* bf16 layers run by the fused preparation kernel: while that kernel
                                 routes and decides, its blocks bring up to this many MB of the
                                 layer's routed first-GEMM weights (W1, from expert 0 on, the order
                                 in which the grouped GEMM takes them) into L2, so that the GEMM's
                                 first phase reads them from L2 instead of HBM.  A cache hint: the
                                 results do not depend on it.  0 = none; default 16; at most 4096 */
} moeca_config;

/* Fill `cfg` with the defaults above and the paper's hyper-parameters
 * (tau0 0.8, alpha 0.6, beta 0.65, Sec. 5.3; lambda1 1.0 and lambda2 0.5 are
 * this library's choice: the paper does not print its values). */
void moeca_config_default(moeca_config* cfg);

/* Device pointers of one layer's weights (dtype of the config; bias fp32).
 * Eq. 7 router and Eq. 5 / Eq. 6 experts; every matrix is "K-major":
 *   w_gate [E, D], b_gate [E] fp32 or NULL,
 *   w1 [E, F, D], w2 [E, D, F]  (FFN_e(u) = w2_e GELU(w1_e u), no bias),
 *   ws1 [F, D], ws2 [D, F] for the shared expert (NULL when n_shared == 0).
 * Attention sub-layer (n_heads > 0; NULL otherwise), a = Attn(x):
 *   w_qkv [3D, D]: rows [0, D) queries, [D, 2D) keys, [2D, 3D) values, head h
 *   at rows h*dh .. h*dh + dh - 1 of each; b_qkv [3D] fp32 or NULL;
 *   w_o [D, D] output projection; b_o [D] fp32 or NULL.
 * AdaLN projection (adaln = 1; NULL otherwise): w_ada [6D, D] bf16, the six
 *   D-row blocks in the order shift_a, scale_a, gate_a, shift_m, scale_m,
 *   gate_m; b_ada [6D] fp32 or NULL.
 * Base pointers must be 16-byte aligned. */
typedef struct {
  const void* w_gate;
  const float* b_gate;
  const void* w1;
  const void* w2;
  const void* ws1;
  const void* ws2;
  const void* w_qkv;
  const float* b_qkv;
  const void* w_o;
  const float* b_o;
  const void* w_ada;
  const float* b_ada;
} moeca_layer_weights;

/* Per-step arguments. */
typedef struct {
  int32_t n_tokens;      /* T, 0..max_tokens; T = 0 is a no-op; a new T forces a full step */
  int32_t step_index;    /* denoising step counter used by the refresh schedule             */
  int32_t force_refresh; /* 1: make this a full-computation step (Sec. 4.1)                 */
  float tau0_override;   /* NaN: use config tau0; otherwise the Eq. 12 base threshold now   */
  const float* cond;     /* adaln = 1: [n_tokens / seq_len, D] fp32 device, each sample's
                            conditioning c (timestep + class embedding); caller-owned, read by
                            the step's first kernel, so it must stay valid until the stream
                            reaches it; NULL otherwise (an AdaLN stack refuses NULL with
                            MOECA_ERR_INVALID_ARG before any launch) */
} moeca_step_args;

/* Branch counters, cumulative since create / moeca_reset_stats (Fig. 8 inputs). */
typedef struct {
  int64_t layer_steps;          /* layer evaluations                                    */
  int64_t refresh_layer_steps;  /* of which full-computation                            */
  int64_t branches;             /* routed branches, T * k per layer step                */
  int64_t cache_step_branches;  /* routed branches on cache steps                       */
  int64_t matched;              /* cache-step branches whose expert is cached for the token */
  int64_t recomputed;           /* branches recomputed (every branch on full steps)     */
  int64_t reused;               /* branches served from the cache                       */
  int64_t tokens_fully_reused;  /* cache-step tokens with an empty recompute set        */
  int64_t shared_recomputed;    /* shared-expert rows recomputed                        */
  int64_t near_margin_route;    /* tokens whose ranks 1..k+1 logits differ by < 1e-5 relative */
  int64_t near_margin_score;    /* matched branches with |s - tau| < 1e-5 |tau|         */
  int32_t device_status;        /* 0, or the first kernel status code seen              */
  int32_t device_detail;        /* kernel-specific detail of that status                */
  int64_t attn_recomputed;      /* token rows whose attention output was computed (n_heads > 0) */
} moeca_stats;

/* Caller-owned DEVICE buffers for one layer's cached state, T rows each.
 * Any pointer may be NULL in moeca_get_layer_state (that field is skipped);
 * moeca_set_layer_state needs all of them (shared_h only when n_shared == 1,
 * attn_a only when n_heads > 0, cache_y only when token_reuse_policy == 1).
 *   cache_e [T, k] int32   cached expert ids e^{t0}        (Eq. 7)
 *   cache_w [T, k] fp32    cached gate weights w^{t0}      (Eq. 7)
 *   cache_norm [T, k] fp32 ||h^{t0}|| over D                (Eq. 9, o)
 *   cache_h [T, k, D] dtype cached branch outputs h^{t0}    (Eq. 7)
 *   shared_h [T, D] dtype  cached shared-expert output      (Eq. 6)
 *   ema [T, E] fp32        C_{e,i} stored at [i * E + e]     (Eq. 10)
 *   attn_a [T, D] dtype    cached attention output a^{t0}   (Sec. 4.1; n_heads > 0)
 *   cache_y [T, D] fp32    each token's last computed MoE output y^{t0}, before the AdaLN
 *                          gate (token_reuse_policy = 1; ignored otherwise) */
typedef struct {
  int32_t* cache_e;
  float* cache_w;
  float* cache_norm;
  void* cache_h;
  void* shared_h;
  float* ema;
  void* attn_a;
  float* cache_y;
} moeca_layer_state;

/* Caller-owned DEVICE buffers for what one layer computed on the last step.
 * Any pointer may be NULL (skipped).  G = E + n_shared work groups.
 *   route_e [T, k] int32, route_w [T, k] fp32   routing B_i^t (Eq. 7)
 *   tau [E] fp32                                 thresholds (Eq. 12)
 *   recompute [T, k] uint8, slot [T, k] int8     decision and cache slot of branch p
 *   matched [T, k] uint8                         expert found in the token's cache
 *   token_any [T] uint8                          recompute set non-empty (Sec. 4.1)
 *   counts [G] int32, offsets [G + 1] int32      rows per expert group
 *   list [offsets[G]] int32                      rows: token * k + slot (routed), token (shared)
 *   layer_in [T, D] dtype                        the MoE sub-layer's input: the layer input, or
 *                                                for a DiT-MoE block u = x + a after the
 *                                                attention update (the FFN rows and the residual)
 *   block_in [T, D] dtype                        the DiT-MoE block's input x (n_heads > 0)
 *   route_in [T, D] dtype                        an AdaLN block's router input: m on full
 *                                                steps, m' on sync cache steps (keep_route_in
 *                                                = 1; skipped otherwise)
 *   resid [T, D] dtype                           the residual stream u the MoE output is added
 *                                                to (n_heads > 0); for an AdaLN block layer_in
 *                                                is m, the FFN rows' input
 *   mod [T / seq_len, 6D] fp32                   an AdaLN block's modulation this step */
typedef struct {
  int32_t* route_e;
  float* route_w;
  float* tau;
  uint8_t* recompute;
  int8_t* slot;
  uint8_t* matched;
  uint8_t* token_any;
  int32_t* counts;
  int32_t* offsets;
  int32_t* list;
  void* layer_in;
  void* block_in;
  void* route_in;
  void* resid;
  float* mod;
} moeca_layer_trace;

/* Kernel kinds timed by moeca_set_kernel_timing(). */
enum {
  MOECA_K_ROUTER = 0,  /* gate logits, softmax, top-k, EMA, entropy -> tau  */
  MOECA_K_SELECT = 1,  /* match, score, threshold, slots, group counts      */
  MOECA_K_COMPACT = 2, /* per-expert row lists and row gather               */
  MOECA_K_FFN1 = 3,    /* grouped GEMM X W1^T + GELU                        */
  MOECA_K_FFN2 = 4,    /* grouped GEMM Hmid W2^T -> cache rows              */
  MOECA_K_COMBINE = 5, /* Eq. 8 combine + residual + cached norms           */
  MOECA_K_PREP = 6,    /* router + select + compact fused in one launch (bf16) */
  MOECA_K_FFN = 7,     /* both grouped GEMMs in one persistent launch (bf16) */
  MOECA_K_QKV = 8,     /* attention: query / key / value projection GEMM     */
  MOECA_K_ATTN = 9,    /* attention: softmax(q k^T / sqrt(dh)) v of the recomputed rows */
  MOECA_K_OPROJ = 10,  /* attention: output projection GEMM + x + a          */
  MOECA_K_ATTN_AUX = 11, /* attention: u = x + a^{t0}, recomputed-token list, FFN row gather */
  MOECA_K_ADALN = 12,  /* AdaLN: modulation vectors, layer norm + modulation of the rows */
  MOECA_K_COUNT = 13
};

typedef struct {
  double total_ms[MOECA_K_COUNT]; /* summed CUDA-event time per kernel kind */
  int64_t launches[MOECA_K_COUNT];
} moeca_kernel_times;

/* Create a handle on CUDA device `device` and allocate its state (caches for
 * max_tokens rows per layer) and workspace.  `layers` points to n_layers host
 * structs of device weight pointers.  Errors: INVALID_ARG (NULL, a field out
 * of range), UNSUPPORTED (shape the kernels do not take), OOM, CUDA.  On error
 * *out is set to NULL and nothing is leaked. */
moeca_status moeca_create(const moeca_config* cfg, const moeca_layer_weights* layers,
                          int32_t device, moeca_handle** out);

/* Run the stack for one denoising step on `stream`.  x_in [T, D] and
 * x_out [T, D] are device buffers of the config dtype that must not overlap
 * (both may be NULL when T = 0, which does nothing).
 * The step is a full-computation step when forced, on the first step after
 * create / reset, when T differs from the previous step, or when
 * refresh_period > 0 divides step_index (Sec. 4.1); otherwise a cache step.
 * Asynchronous: no host synchronisation inside.  Errors: INVALID_ARG,
 * STATE (handle destroyed), DEVICE_STATUS / TIMEOUT (from an earlier kernel),
 * CUDA (launch failure). */
moeca_status moeca_step(moeca_handle* h, const void* x_in, void* x_out,
                        const moeca_step_args* args, void* stream);

/* One step from and to HOST buffers: the serving form of moeca_step.
 * x_in_host [T, D] and x_out_host [T, D] are host memory in the config dtype
 * (page-locked memory makes the copies asynchronous; pageable memory works
 * but each copy then blocks the calling thread); args->cond, when the stack
 * is AdaLN, is a HOST pointer to [T / seq_len, D] fp32 here.  The library
 * uploads the input (and cond) into one of two device staging buffers on its
 * own upload stream, runs moeca_step on `stream`, and reads the output back
 * on its own read-back stream, so the upload of the next call and the
 * read-back of this one overlap the neighbouring steps' compute.
 * Asynchronous: x_out_host is written once the read-back has run; call
 * moeca_host_join(h, stream) and then synchronise `stream` (or an event
 * recorded on it after the join) before reading it.  The caller keeps
 * x_in_host and cond unchanged, and x_out_host alive, until then.
 * The first call allocates the staging buffers (4 x max_tokens x D elements,
 * plus the conditioning) and the two copy streams: make it before any stream
 * capture.  Errors: as moeca_step, plus OOM / CUDA from that first call. */
moeca_status moeca_step_host(moeca_handle* h, const void* x_in_host, void* x_out_host,
                             const moeca_step_args* args, void* stream);

/* Make `stream` wait for every upload and read-back that earlier
 * moeca_step_host calls enqueued: work enqueued on `stream` afterwards (an
 * event, a synchronisation) comes after the last output reached host memory.
 * No-op when moeca_step_host was never called. */
moeca_status moeca_host_join(moeca_handle* h, void* stream);

/* ---- Token-sharded stacks --------------------------------------------------
 * Tokens are independent in every step of the layer except one: Eq. 11's
 * per-expert sums S_e = sum_i C_{e,i} and U_e = sum_i C ln C run over all T
 * token rows of the batch.  A stack can therefore be split by tokens over
 * `world` ranks (processes or GPUs), each holding a contiguous slice of
 * n_tokens rows (rank r: global rows [r n_tokens, (r + 1) n_tokens)) with
 * the weights replicated, exchanging only the per-block partial sums of
 * S_e and U_e once per layer per step.  Every rank then reduces every
 * rank's partials in the same global block order as a single-rank step
 * over the whole batch, so thresholds, decisions, row lists and outputs are
 * bit-identical to that step's.
 *
 *   moeca_shard_exchange_bytes(h, n_tokens, &bytes);     // per rank
 *   (send: bytes, recv: world x bytes, caller-owned device buffers)
 *   moeca_shard_begin(h, x_in, x_out, args, shard, send, recv, stream);  // layer 0 routed
 *   do {
 *     all-gather `bytes` from every rank's send into recv in rank order, on
 *       `stream` (e.g. ncclAllGather);
 *     moeca_shard_next(h, stream, &done);   // finish this layer, route the next
 *   } while (!done);
 *
 * Supported for the bf16 MoE layer stack run by the fused preparation kernel
 * (n_heads 0, ffn_impl AUTO, token_reuse_policy 0); n_tokens must be a
 * multiple of that kernel's token block (32 or 16) and equal on every rank;
 * total_tokens = world x n_tokens (else INVALID_ARG / UNSUPPORTED).  The
 * refresh schedule and state are as moeca_step's.  send and recv are
 * 16-byte aligned device buffers the caller keeps until the step is done;
 * each layer's partials are written to send by the kernels before the
 * exchange and read from recv by those after it.  Asynchronous on `stream`
 * like moeca_step; a started step must be finished with moeca_shard_next
 * before another step (MOECA_ERR_STATE otherwise; moeca_reset abandons it). */
typedef struct {
  int32_t rank;          /* this rank, 0 .. world - 1                        */
  int32_t world;         /* ranks holding a slice of the batch               */
  int32_t total_tokens;  /* token rows of the whole batch (world x n_tokens) */
} moeca_shard;
/* Bytes one rank contributes to each layer's exchange for n_tokens rows. */
moeca_status moeca_shard_exchange_bytes(moeca_handle* h, int32_t n_tokens, int64_t* bytes_per_rank);
moeca_status moeca_shard_begin(moeca_handle* h, const void* x_in, void* x_out, const moeca_step_args* args,
                               const moeca_shard* shard, void* send, const void* recv, void* stream);
/* Finish the layer in progress from the gathered partials in recv and route
 * the next one into send; *done = 1 after the last layer (x_out then holds
 * the output). */
moeca_status moeca_shard_next(moeca_handle* h, void* stream, int32_t* done);

/* Copy the counters of `layer` (or the sum over layers for layer = -1) into
 * *out.  Synchronises the device. */
moeca_status moeca_get_stats(moeca_handle* h, int32_t layer, moeca_stats* out);
moeca_status moeca_reset_stats(moeca_handle* h);

/* Copy one layer's cached state into caller device buffers (async on stream);
 * *n_tokens receives the T the state holds (0 if none). */
moeca_status moeca_get_layer_state(moeca_handle* h, int32_t layer, const moeca_layer_state* dst,
                                   int32_t* n_tokens, void* stream);

/* Load one layer's cached state from caller device buffers (async on stream)
 * for n_tokens rows (1..max_tokens) and mark the caches valid, so the next
 * step with that T is a cache step unless the schedule says otherwise.  Used to
 * resume a trajectory and to teacher-force parity tests.  Every layer must
 * hold the same T. */
moeca_status moeca_set_layer_state(moeca_handle* h, int32_t layer, const moeca_layer_state* src,
                                   int32_t n_tokens, void* stream);

/* Copy what `layer` computed on the last step (see moeca_layer_trace). */
moeca_status moeca_get_layer_trace(moeca_handle* h, int32_t layer, const moeca_layer_trace* dst,
                                   void* stream);

/* Drop every cache and zero the EMA statistics; the next step is a full step.
 * Synchronises the device, then clears a recorded device status (a timeout or
 * a bad index reported by an earlier kernel) and re-arms every internal
 * counter a cut-short launch may have left mid-count: the way back after
 * MOECA_ERR_TIMEOUT or MOECA_ERR_DEVICE_STATUS. */
moeca_status moeca_reset(moeca_handle* h);

/* Host-side fault injection for tests of failure detection (no counterpart
 * in the paper).  MOECA_FAULT_BARRIER_STALL: the next step's fused
 * preparation kernels wait at their grid-wide exchanges for values tagged
 * with a launch number that no launch writes, as if a block never arrived;
 * every block gives up after about one second of %globaltimer,
 * records MOECA_ERR_TIMEOUT in the device status and skips its later phases,
 * so the step's outputs are garbage and the next call that checks the device
 * status returns MOECA_ERR_TIMEOUT until moeca_reset.  Nothing faults or
 * hangs.  Returns MOECA_ERR_UNSUPPORTED when the handle does not run the
 * fused preparation kernel (fp32, or shapes it does not fit). */
typedef enum { MOECA_FAULT_BARRIER_STALL = 1 } moeca_fault;
moeca_status moeca_inject_fault(moeca_handle* h, int32_t kind);

/* Record CUDA events around every kernel launch (enable = 1) and accumulate
 * their durations; moeca_get_kernel_times() synchronises and reads them, and
 * resets the sums when reset = 1. */
moeca_status moeca_set_kernel_timing(moeca_handle* h, int32_t enable);
moeca_status moeca_get_kernel_times(moeca_handle* h, moeca_kernel_times* out, int32_t reset);

/* Free everything the handle owns.  NULL is accepted. */
moeca_status moeca_destroy(moeca_handle* h);

/* ---- Allocation-free router call ---------------------------------------
 * The paper has no counterpart to this call.  It exists for callers that
 * cannot allocate device memory, so cannot create a handle (moeca_create
 * allocates the caches and the workspace): code running inside a host
 * framework that owns every device allocation through its own pool, or a
 * deployment whose device memory budget is fixed when it starts.
 *
 * moeca_route_noalloc runs the router of one layer on caller-owned device
 * buffers: gate logits, softmax, top-k (Eq. 7), the EMA statistic update
 * (Eq. 10) and the per-expert thresholds (Eq. 11-12), the same computation
 * moeca_step runs first in every layer.  It allocates nothing (no cudaMalloc,
 * no cudaFree, no allocating library routine).  Its only scratch memory, the
 * per-block entropy partial sums and a completion counter, is one fixed
 * array compiled into the library: 256 KB + 256 B, held by every GPU that
 * loads the library until the process exits.
 *
 * Limit: ceil(n_tokens / 16) * n_experts <= 32768 (up to 8192 tokens with 64
 * experts, 32768 tokens with 16).  A larger call returns MOECA_ERR_UNSUPPORTED
 * and launches nothing.  Other errors: MOECA_ERR_INVALID_ARG (NULL or
 * misaligned pointer, a size out of range), MOECA_ERR_CUDA (the scratch
 * address lookup or the launch failed).
 *
 * The first call on each device looks up that device's address of the scratch
 * array (cudaGetSymbolAddress, with that device current), so make the first
 * call on a device before any stream capture.  Every call shares the one
 * array, which keeps the last call's contents; each call clears what must
 * start at zero itself.  Calls that overlap on the GPU (on different streams
 * or from different host threads) race on the scratch: serialise them.
 * Runs on the current device, asynchronously on `stream`. */
typedef struct {
  int32_t dtype;         /* moeca_dtype of x and w_gate                       */
  int32_t n_tokens;      /* T >= 1                                             */
  int32_t hidden;        /* D: multiple of 8 (bf16) or 4 (fp32)                */
  int32_t n_experts;     /* E, 1..64                                           */
  int32_t top_k;         /* k, 1..min(8, E)                                    */
  int32_t renorm_topk;   /* as in moeca_config                                 */
  int32_t entropy_norm;  /* as in moeca_config                                 */
  float beta;            /* Eq. 10 EMA decay, [0, 1)                           */
  float tau0;            /* Eq. 12 base threshold                              */
  float alpha;           /* Eq. 12 adaptation strength, [0, 1)                 */
  const void* x;         /* [T, D] device, 16-byte aligned                     */
  const void* w_gate;    /* [E, D] device, 16-byte aligned                     */
  const float* b_gate;   /* [E] device, or NULL                                */
  float* ema;            /* [T, E] device, C_{e,i} at [i*E + e]: read, then updated in place */
  int32_t* route_e;      /* [T, k] device output: expert ids, descending logit */
  float* route_w;        /* [T, k] device output: gate weights                */
  float* tau;            /* [E] device output: thresholds tau_e               */
} moeca_route_args;

moeca_status moeca_route_noalloc(const moeca_route_args* args, void* stream);

/* ---- Sampler (Eq. 1) ------------------------------------------------------
 * The reverse transition of Eq. 1 with the denoiser's output eps:
 *   x_{t-1} = (x_t - (1 - alpha_t) / sqrt(1 - abar_t) eps) / sqrt(alpha_t) + sigma_t z.
 *
 * moeca_ddpm_schedule fills host arrays [n_steps] for a sampling run of
 * n_steps steps over a linear training schedule of n_train betas from
 * beta_start to beta_end (abar_s = prod_{r <= s} (1 - beta_r)): run step j
 * visits training step t_j = floor(j (n_train - 1) / (n_steps - 1) + 1/2) and
 * takes abar'_j = abar_{t_j}, alpha'_j = abar'_j / abar'_{j-1} (abar'_{-1} = 1),
 * beta'_j = 1 - alpha'_j.  A run goes from j = n_steps - 1 down to 0; Eq. 1's
 * variance gives sigma_j = sqrt(beta'_j), and the last step (j = 0) adds no
 * noise.  Any output pointer may be NULL.  INVALID_ARG unless
 * 2 <= n_steps <= n_train and 0 < beta_start <= beta_end < 1. */
moeca_status moeca_ddpm_schedule(int32_t n_steps, int32_t n_train, double beta_start, double beta_end,
                                 int32_t* t, double* alpha, double* alpha_bar, double* beta);

/* moeca_ddpm_step runs the update on device buffers, asynchronously on
 * `stream` (the current device).  x_prev may alias x_t; x_next (optional)
 * receives x_prev in eps_dtype, the next denoiser input.  n must be a
 * multiple of 8 and every pointer 16-byte aligned (INVALID_ARG otherwise);
 * z may be NULL only when sigma == 0.  The noise z is the caller's draw.
 * Every buffer is caller-owned device memory and must stay valid until the
 * stream has run the update.  Errors: INVALID_ARG (checked on the host,
 * nothing launched), CUDA (the launch failed); the message is in
 * moeca_last_error(NULL). */
typedef struct {
  int64_t n;             /* elements                                   */
  int32_t eps_dtype;     /* moeca_dtype of eps and x_next              */
  double alpha;          /* alpha'_j                                   */
  double alpha_bar;      /* abar'_j (< 1)                              */
  double sigma;          /* sigma_j >= 0                               */
  const float* x_t;      /* [n] fp32                                   */
  const void* eps;       /* [n] eps_dtype                              */
  const float* z;        /* [n] fp32 standard normal draw, or NULL     */
  float* x_prev;         /* [n] fp32                                   */
  void* x_next;          /* [n] eps_dtype, or NULL                     */
} moeca_ddpm_args;
moeca_status moeca_ddpm_step(const moeca_ddpm_args* args, void* stream);

const char* moeca_status_string(moeca_status s);
/* Message of the last error on this handle ("" if none); NULL handle: the
 * last failure of a call without a handle on this thread (moeca_create,
 * moeca_ddpm_schedule, moeca_ddpm_step). */
const char* moeca_last_error(const moeca_handle* h);

#ifdef __cplusplus
}
#endif
#endif /* MOECA_H_ */
