// Internal launch interface between the host engine and the MoECa kernels.
// Plain structs of device pointers and sizes; `bf16` selects the element type
// (__nv_bfloat16 when true, float otherwise) of every activation, weight and
// cached-output buffer.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace moeca {

// Counters per layer, in this order (device uint64).
enum StatIndex {
  kStLayerSteps = 0, kStRefreshSteps, kStBranches, kStCacheBranches, kStMatched,
  kStRecomputed, kStReused, kStTokensFullyReused, kStSharedRecomputed,
  kStNearRoute, kStNearScore, kStAttnRows, kStCount
};

// cudaFuncSetAttribute(MaxDynamicSharedMemorySize, bytes) for `func` on the
// current device, once per (device, kernel) unless a larger value is asked
// for: the attribute belongs to the kernel on each device, so a process that
// uses several devices sets it on each.  Thread-safe.
cudaError_t set_dyn_smem_on_device(const void* func, int bytes);

constexpr int kMaxExperts = 64;
constexpr int kMaxTopK = 8;
constexpr int kRouterTokensPerBlock = 16;   // 8 warps x 2 tokens
constexpr int kSelectTokensPerBlock = 128;  // one token per thread

// Eq. 7 router + Eq. 10 EMA + Eq. 11-12 threshold (finished by the last block).
struct RouterArgs {
  const void* x;        // [T, D]
  const void* w_gate;   // [E, D]
  const float* b_gate;  // [E] or null
  int T, D, E, k;
  int renorm;
  float beta;
  float tau0, alpha;
  int entropy_norm;
  int32_t* route_e;     // [T, k]
  float* route_w;       // [T, k]
  float* ema;           // [T, E]
  float* partials;      // [gridDim.x, E, 2]   (sum C, sum C ln C) per block
  unsigned* done;       // last-block ticket, left at 0
  float* tau;           // [E]
  unsigned long long* stats;
  int* status;          // device status word (or null)
};
cudaError_t launch_router(const RouterArgs& a, bool bf16, cudaStream_t s);

// Sec. 4.2 match / Eq. 9 score / threshold / slots + per-group counts (the
// last block scans them into offsets).
struct SelectArgs {
  int T, k, E, G;       // G = E + n_shared
  int refresh;
  float lambda1, lambda2;
  int reused_meta_policy, shared_policy, n_shared;
  int score_terms;      // Eq. 9 terms kept: 1 = w, 2 = lambda1 Delta, 4 = lambda2 o
  int token_level;      // 1: a token's branches share one decision
  const int32_t* route_e;
  const float* route_w;
  const float* tau;
  int32_t* cache_e;     // [T, k]  updated in place
  float* cache_w;       // [T, k]  updated in place
  const float* cache_norm;
  uint8_t* recompute;   // [T, k]
  int8_t* slot;         // [T, k]
  uint8_t* matched;     // [T, k]
  uint8_t* token_any;   // [T]
  int32_t* block_counts;   // [nblk, G]
  int32_t* block_offsets;  // [nblk, G]
  int32_t* counts;         // [G]
  int32_t* offsets;        // [G + 1]
  unsigned* done;
  unsigned long long* stats;
  int* status;
};
cudaError_t launch_select(const SelectArgs& a, cudaStream_t s);

// Per-group row lists in ascending token order + gather of the rows' inputs.
struct CompactArgs {
  int T, k, E, G, D, n_shared;
  int refresh, shared_policy;
  const int32_t* route_e;
  const uint8_t* recompute;
  const int8_t* slot;
  const uint8_t* token_any;
  const int32_t* block_offsets;
  const int32_t* offsets;
  int32_t* list;        // [rows]
  const void* x;        // [T, D]
  void* xg;             // [rows, D] gathered inputs, or null when the GEMM gathers itself
  int* status;
};
// compact_kernel (row lists), then, unless xg is null, gather_kernel (rows).
cudaError_t launch_compact(const CompactArgs& a, bool bf16, cudaStream_t s);
// gather_kernel alone: the listed rows of a.x into a.xg (lists already built).
cudaError_t launch_gather(const CompactArgs& a, bool bf16, cudaStream_t s);

// Grouped expert FFN over the compacted rows (Eq. 5 / Eq. 6 on R only).
struct FfnArgs {
  int G, E, D, F, k, T;
  int max_rows;          // capacity of xg / hmid rows
  const int32_t* counts;
  const int32_t* offsets;
  const int32_t* list;
  const void* xg;        // [rows, D]   gathered inputs (SIMT path)
  const void* x;         // [T, D]      layer input: the tensor-core path gathers rows from it
  void* hmid;            // [rows, F]
  const void* w1;        // [E, F, D]
  const void* w2;        // [E, D, F]
  const void* ws1;       // [F, D]   shared expert (group E) or null
  const void* ws2;       // [D, F]
  void* cache_h;         // [T*k, D]   destination rows of routed groups
  void* shared_h;        // [T, D]     destination rows of the shared group
  int gelu_tanh;
  int tile_n;            // tensor-core tile width to force (0: chosen per launch)
  int split_k;           // tensor-core K splits to force (0: chosen per launch)
  float* partial;        // split-K workspace: tensor-core path, or the fp32 path's [simt_split, max_rows, D]
  int simt_split;        // fp32 path: K splits of the second GEMM (1: none)
  int* tile_sem;         // split-K arrival counters, zeroed once
  int* dep;              // tensor-core fused launch: per m-tile counter pairs, zeroed once (or null)
  int max_mtiles;        // capacity of dep, tc_dep_pairs(max_rows, G)
  int* work;             // tensor-core path: unit ticket counter; 0 before every launch (the combine
                         // kernel that follows re-arms it)
  int* status;
};
cudaError_t launch_ffn_simt(const FfnArgs& a, bool bf16, int phase, cudaStream_t s);

// tcgen05 / TMA grouped GEMM (bf16 only).  Tensor maps are built once per
// handle; `TcPlan` owns them.
struct TcPlan;
TcPlan* tc_plan_create(const FfnArgs& a, int n_sms, char* err, int errlen);
size_t tc_split_units(int n_sms);      // split-K units the workspace holds
size_t tc_partial_bytes(int n_sms);    // bytes of the split-K partial workspace
size_t tc_dep_pairs(int max_rows, int G);  // m-tile counter pairs a fused launch can need
void tc_plan_destroy(TcPlan* p);
// phase 1 or 2: that GEMM alone; phase 0: both, fused into one persistent
// launch when a.dep is set and no K split is forced (else two launches).
cudaError_t launch_ffn_tc(TcPlan* p, const FfnArgs& a, int phase, cudaStream_t s);

// Fused router + select + compact (one cooperative launch, bf16 only).
struct PrepArgs {
  const void* x;          // [T, D] layer input
  const void* w_gate;     // [E, D]
  const float* b_gate;    // [E] or null
  int T, D, E, k, G;      // G = E + n_shared groups
  int renorm, entropy_norm;
  float beta, tau0, alpha;
  int32_t* route_e;       // [T, k]
  float* route_w;         // [T, k]
  float* ema;             // [T, E]
  unsigned long long* part_words;   // [blocks, E, 2] tagged (sum C, sum C ln C) per block (exchange 1)
  unsigned long long* count_words;  // [blocks, groups] tagged recomputed rows per group (exchange 2)
  unsigned epoch;         // this launch's tag (never 0, never reused before a reset)
  unsigned wait_epoch;    // the tag the exchanges wait for (epoch, unless a stall is injected)
  float* shard_send;      // token-sharded MODE 1: [blocks, E] float2 block partials (sum C, sum C ln C)
  const float* shard_recv;  // MODE 2: [shard_blocks, E] float2, every rank's partials in rank order
  int shard_blocks;       // MODE 2: blocks of all ranks
  int shard_tokens;       // MODE 2: tokens of all ranks (T of Eq. 11's normalisation)
  float* tau;             // [E] (written by block 0)
  SelectArgs sel;         // decision inputs and outputs (its tau is replaced in-kernel)
  int32_t* counts;        // [G]
  int32_t* offsets;       // [G + 1]
  int32_t* list;          // [rows]
  void* xg;               // [rows, D], or null: the rows are gathered later (launch_gather)
  const void* attn_a;     // DiT-MoE block cache step: [T, D] cached attention rows a^{t0}, or null;
                          // then the rows staged from x become u = x + a^{t0}, written to u_out
  void* u_out;            // [T, D]
  int gather_final_only;  // 1: gather only the rows of tokens without recomputed branches
  int32_t* row_of;        // or null: [T, k + n_shared] list position of each branch's row
                          // (p < k routed, p = k shared), -1 when not recomputed
  int n_shared;
  int attn_list;          // 1: also list the tokens with a non-empty recompute set (group G)
  int32_t* attn_rows;     //   [T] ascending tokens,
  int* attn_n;            //   their count,
  int32_t* attn_inv;      //   [T] each token's place (-1 if absent),
  int32_t* sample_lo;     //   [T / seq + 1] where each sample's tokens start
  int seq;                //   tokens per sample
  const void* l2_pf;      // or null: [l2_pf_bytes] brought into L2 while the block routes (a hint)
  size_t l2_pf_bytes;     // a multiple of 16; l2_pf 16-byte aligned
  unsigned long long* stats;
  int* status;
};
struct PrepShape {
  int tokens_per_block;   // 0: the fused kernel cannot run this shape
  int epad;               // experts padded to a multiple of 8
  int kmax;               // compile-time bound on top-k (2, 4 or 8)
  size_t smem;            // dynamic shared memory per block
  bool attn;              // the DiT-MoE block build of the kernel
};
constexpr size_t kPrepSmemMax = 200 * 1024;
PrepShape prep_plan(int D, int E, int k, int max_tokens, int n_sms, bool attn);
// The two builds of prep.cu (plain, and prep_attn.cu for DiT-MoE blocks).
PrepShape prep_plan_plain(int D, int E, int k, int max_tokens, int n_sms);
PrepShape prep_plan_attn(int D, int E, int k, int max_tokens, int n_sms);
cudaError_t launch_prep_plain(const PrepArgs& a, const PrepShape& p, cudaStream_t s);
cudaError_t launch_prep_attn(const PrepArgs& a, const PrepShape& p, cudaStream_t s);
cudaError_t launch_prep(const PrepArgs& a, const PrepShape& p, cudaStream_t s);
// Token-sharded launches of the plain build: mode 1 routes and writes the
// block partials to shard_send, mode 2 reduces shard_recv and decides.
cudaError_t launch_prep_shard(const PrepArgs& a, const PrepShape& p, int mode, cudaStream_t s);

// Eq. 8 combine + residual + cached branch norms.
struct CombineArgs {
  int T, D, k, n_shared;
  const void* x;          // [T, D]
  void* out;              // [T, D]
  const void* cache_h;    // [T, k, D]
  const void* shared_h;   // [T, D] or null
  const float* route_w;   // [T, k]
  const int8_t* slot;     // [T, k]
  float* cache_norm;      // [T, k]
  int* rearm;             // a counter the previous kernel leaves for re-arming (the GEMM's unit
                          // ticket), set to 0 after the dependency wait, or null
  const float* gate;      // AdaLN block (bf16): out = x + gate * y, gate row of token i at
  int gate_ld, seq;       //   gate + (i / seq) * gate_ld; null: out = x + y
  float* cache_y;         // [T, D] fp32 last computed y per token (token_reuse_policy 1), or null
  const uint8_t* token_any;  // [T] recompute set non-empty (with cache_y)
  int copy_y;             // 1: a token with token_any 0 takes y = cache_y (a cache step under
                          //   token_reuse_policy 1); 0: every token computes y (and stores it)
  int n_sms;              // the device's SM count (the staged form's persistent grid)
  int direct;             // 1: force the direct form (one warp per token, rows loaded by the lanes)
  int early;              // 1: in the direct form, a token with token_any 0 is combined without
                          //   waiting for the previous kernel (a cache step, no token-level copy,
                          //   the shared row, if any, recomputed only for tokens with token_any)
  int* status;
};
cudaError_t launch_combine(const CombineArgs& a, bool bf16, cudaStream_t s);

// ---- Attention path of a DiT-MoE block (Sec. 4.1), bf16 only ----

// Tensor-core projection GEMM: C = A B^T + bias (proj_tc.cu).
enum ProjMode { kProjStore = 0, kProjResidual = 1, kProjQKV = 2, kProjResidualGated = 3 };
struct ProjArgs {
  const void* A;          // [a_rows, K] bf16, row-major
  int a_rows;             // rows A holds (>= M)
  const void* B;          // [N, K] bf16 weights
  const float* bias;      // [N] or null
  int M, N, K;            // N a multiple of 64, K of 64
  int tile_n;             // output tile width (0: the widest of 256 / 128 / 64 dividing N)
  const int* m_dev;       // device row count (<= M), or null
  int mode;               // ProjMode
  void* out;              // kProjStore: [M, ldo] bf16
  int ldo;
  const int32_t* rows;    // kProjResidual: token of row m, or null (m)
  int n_tok;              // kProjResidual: rows of x / a_out / u_out
  const void* x;          // kProjResidual: [n_tok, N]
  void* a_out;            // kProjResidual: [n_tok, N]  a_i
  void* u_out;            // kProjResidual: [n_tok, N]  x_i + a_i
  unsigned long long* row_stat;  // or null: the launch adds its row count here
  const int32_t* row_of;  // kProjResidual, or null: [n_tok, row_w] FFN row positions of the token
  int row_w;              //   (-1: none); u is also written to those rows of xg
  void* xg;               // [rows, N] FFN input rows
  const int32_t* inv;     // kProjQKV (N = 3D): list place of token m, -1 if not listed, or null (m)
  void* q_out;            // kProjQKV: [list rows, D] q of the listed tokens, in list order
  void* k_out;            // kProjQKV: [n_tok, D] k
  void* vt_out;           // kProjQKV: [D, n_tok] v transposed
  const float* gate;      // kProjResidualGated: u = x + gate * a, the gate row of token t at
  int gate_ld, seq;       //   gate + (t / seq) * gate_ld (AdaLN block)
  int* status;
};
// Tile width a launch uses for N: `want` (64 / 128 / 256) if it divides N,
// else (want = 0) the widest that does; 0 when none fits.
int proj_tile_n(int N, int want);
cudaError_t launch_proj_tc(const ProjArgs& a, cudaStream_t s);

// ---- AdaLN modulation of a DiT-MoE block (Sec. 3) and the sampler step (Eq. 1) ----

// mod[l][b][j] = sum_d SiLU(cond[b][d]) w[l][j][d] + b[l][j] for every layer l,
// sample b < B and row j < 6D, in one launch (adaln.cu).
struct AdaModArgs {
  int L, B, D;
  const float* cond;                    // [B, D] fp32
  const void* const* w;                 // device array [L] of [6D, D] bf16 matrices
  const float* const* b;                // device array [L] of [6D] fp32 vectors (entries may be null)
  float* out;                           // [L, B, 6D]
};
// Bytes of shared memory the launch needs (B * D fp32), and whether it fits.
size_t ada_mod_smem(int B, int D);
cudaError_t launch_ada_mod(const AdaModArgs& a, int n_sms, cudaStream_t s);

// Row-wise layer normalisation and modulation of one AdaLN block, one warp per
// row t (rows[i], or i < T):
//   h = bf16(LN(x) (1 + scale_a) + shift_a)              when h_out is set
//   u = bf16(x + gate_a a), written to u                 when a is set (else u is read)
//   m = bf16(LN(u) (1 + scale_m) + shift_m)              when m_out is set (and m_copy)
// with the six D-vectors of the row's sample at mod + (t / seq) * 6D in the
// order shift_a, scale_a, gate_a, shift_m, scale_m, gate_m.  bf16 only.
struct AdaLnArgs {
  int T, D, seq;
  float eps;
  const float* mod;       // [T / seq, 6D]
  const void* x;          // [T, D]
  const void* a;          // [T, D] or null
  void* h_out;            // [T, D] or null
  void* u;                // [T, D]
  void* m_out;            // [T, D] or null
  void* m_copy;           // [T, D] or null
  const int32_t* rows;    // or null (every row)
  const int* n_rows;      // device count of rows (with rows)
  int* status;
};
constexpr int kAdaLnMaxD = 2560;
cudaError_t launch_adaln_rows(const AdaLnArgs& a, cudaStream_t s);

// x_prev = (x_t - c1 eps) inv_sqrt_alpha + sigma z (Eq. 1), n elements, and
// optionally x_next = x_prev in the denoiser's dtype.
struct DdpmArgs {
  long long n;
  int bf16;               // eps and x_next are bf16 (else fp32)
  float c1, inv_sqrt_alpha, sigma;
  const float* x_t;
  const void* eps;
  const float* z;         // or null (sigma == 0)
  float* x_prev;
  void* x_next;           // or null
};
cudaError_t launch_ddpm(const DdpmArgs& a, cudaStream_t s);

// u = x + a, row by row (the MoE input of a token that keeps its cached attention).
cudaError_t launch_attn_residual(const void* x, const void* a, void* u, int T, int D, int* status,
                                 cudaStream_t s);

// Ascending list of tokens whose recompute set is non-empty, its length,
// where each sample's tokens start in it (sample_lo [T / S + 1]), and each
// token's place in it (inv [T], -1 if absent).
cudaError_t launch_attn_rows(const uint8_t* token_any, int T, int S, int32_t* rows, int* n_rows,
                             int32_t* sample_lo, int32_t* inv, cudaStream_t s);

// Multi-head self-attention rows: o[r] = concat_h softmax(q_t k_S^T / sqrt(dh)) v_S for the
// r-th listed token t, keys and values of t's sample (S consecutive token rows).
struct AttnArgs {
  const void* q;          // [rows, D] bf16: q of the listed tokens in list order (head h at columns h dh ..)
  const void* k;          // [T, D] bf16
  const void* vt;         // [D, T] bf16: v transposed
  int T, D, H, S;         // S tokens per sample (a multiple of 8), T a multiple of S
  const int32_t* rows;    // ascending token list, or null: every token (row r = token r)
  const int32_t* sample_lo;  // with rows: sample b's tokens are rows[sample_lo[b] .. sample_lo[b + 1])
  void* o;                // [rows, D] bf16
  int* status;
};
bool attn_supported(int D, int H);
cudaError_t launch_attn_core(const AttnArgs& a, cudaStream_t s);   // mma.sync (warp-level) core
cudaError_t launch_attn_tc(const AttnArgs& a, cudaStream_t s);     // tcgen05 / TMEM core (attn_tc.cu)

}  // namespace moeca
