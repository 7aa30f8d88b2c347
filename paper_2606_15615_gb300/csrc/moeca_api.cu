// Host engine and C ABI of the branch-cached MoE layer stack (include/moeca.h).
//
// Per step and layer the engine enqueues, on the caller's stream and with no
// host synchronisation:
//   router (Eq. 7, Eq. 10-12) -> select (Sec. 4.2, Eq. 9) -> compact ->
//   grouped FFN phase 1 and 2 over the recompute rows (Eq. 5 / Eq. 6) ->
//   combine (Eq. 8) writing the next layer's input.
// A DiT-MoE block (n_heads > 0) adds its attention sub-layer (Sec. 4.1):
//   full step:  q/k/v projection -> attention of every row -> output
//               projection writing a and u = x + a -> the MoE sub-layer on u;
//   cache step: u = x + a^{t0} -> router / decisions on u -> (sync rule)
//               list of tokens with a non-empty recompute set -> q/k/v
//               projection -> attention of the listed rows -> output
//               projection updating their a and u -> FFN row gather from u
//               -> FFN -> combine with the residual u.
// An AdaLN block (adaln = 1, Sec. 3) first computes every layer's modulation
// vectors from the step's conditioning (one launch), then per layer:
//   full step:  h = LN-modulate(x) -> q/k/v from h -> attention -> output
//               projection writing a and u = x + g_a a -> m = LN-modulate(u)
//               -> the MoE sub-layer on m -> out = u + g_m y;
//   cache step: u' = x + g_a a^{t0}, m' = LN-modulate(u') (and h) in one pass
//               -> decisions on m' -> (sync rule) the listed tokens' attention
//               from h, their a, u and m -> FFN row gather from m -> FFN ->
//               combine out = u + g_m y.
// It decides full-computation vs cache steps (Sec. 4.1), owns every state and
// workspace buffer, and reports errors as status codes.
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <map>
#include <mutex>
#include <new>
#include <string>
#include <utility>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "common.cuh"
#include "kernels.h"
#include "moeca.h"

using namespace moeca;

namespace moeca {

cudaError_t set_dyn_smem_on_device(const void* func, int bytes) {
  static std::mutex mu;
  static std::map<std::pair<int, const void*>, int> done;  // (device, kernel) -> bytes set
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lock(mu);
  auto it = done.find({dev, func});
  if (it != done.end() && it->second >= bytes) return cudaSuccess;
  e = cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e != cudaSuccess) return e;
  done[{dev, func}] = bytes;
  return cudaSuccess;
}

}  // namespace moeca

namespace {

thread_local std::string g_create_error;

// Phase 1 of the tensor-core FFN can gather its A rows from the layer input
// with TMA tile::gather4 instead of reading rows that compact_kernel copied
// into a contiguous buffer.  Measured on GB300 the gather issue rate (32
// gather4 per 64-wide k-block from one thread) costs more than the copy, so
// the copy path is the default.
constexpr bool kGemmGathersRows = false;

struct LayerBuf {
  moeca_layer_weights w;
  int32_t* cache_e = nullptr;
  float* cache_w = nullptr;
  float* cache_norm = nullptr;
  void* cache_h = nullptr;
  void* shared_h = nullptr;
  float* ema = nullptr;
  int32_t* route_e = nullptr;
  float* route_w = nullptr;
  float* tau = nullptr;
  uint8_t* recompute = nullptr;
  int8_t* slot = nullptr;
  uint8_t* matched = nullptr;
  uint8_t* token_any = nullptr;
  int32_t* counts = nullptr;
  int32_t* offsets = nullptr;
  int32_t* list = nullptr;
  unsigned long long* stats = nullptr;
  void* attn_a = nullptr;    // [T, D] cached attention output a^{t0} (DiT-MoE block)
  void* attn_u = nullptr;    // [T, D] MoE sub-layer input u of the last step (AdaLN: the residual u)
  void* attn_m = nullptr;    // [T, D] AdaLN block: the MoE input m of the last step
  void* route_m = nullptr;   // [T, D] AdaLN block: its router input (keep_route_in)
  float* cache_y = nullptr;  // [T, D] fp32 each token's last computed MoE output (token_reuse_policy 1)
  TcPlan* tc = nullptr;
  bool valid = false;
};

struct PendingTiming {
  int kind;
  cudaEvent_t start, stop;
};

}  // namespace

struct moeca_handle {
  moeca_config cfg{};
  int device = 0;
  bool bf16 = false;
  size_t es = 4;
  int G = 0;
  int n_sms = 0;
  int max_rows = 0;
  std::vector<LayerBuf> layers;
  float* partials = nullptr;
  unsigned* done = nullptr;  // [0] router ticket, [1] select ticket
  int32_t* block_counts = nullptr;
  int32_t* block_offsets = nullptr;
  void* xg = nullptr;
  void* hmid = nullptr;
  float* tc_partial = nullptr;
  float* simt_partial = nullptr;  // fp32 path: second-GEMM K-split partials [simt_split, max_rows, D]
  int simt_split = 1;
  int* tc_sem = nullptr;
  int* tc_dep = nullptr;        // fused GEMM launch: m-tile dependency counters, left at 0
  int* tc_work = nullptr;       // GEMM unit tickets {next, CTAs done}, left at 0
  int tc_dep_pairs_n = 0;
  PrepShape prep{0, 0, 0, 0, false};  // fused router + select + compact, when it fits
  unsigned prep_epoch = 0;      // tag of the last fused launch (its exchanges' words)
  bool inject_stall = false;    // moeca_inject_fault: next step's exchanges wait for a tag nobody writes
  unsigned long long* prep_words = nullptr;  // tagged exchange words: partials, then row counts
  size_t prep_words_n = 0;
  size_t prep_count_off = 0;    // where the row-count words start
  void* qkv = nullptr;          // attention workspace: q [T, D] (list order), k [T, D], v^T [D, T]
  int32_t* attn_inv = nullptr;  // [T] each token's place in attn_rows (-1: absent)
  void* attn_o = nullptr;       // [T, D] attention rows before the output projection
  int32_t* attn_rows = nullptr; // [T] tokens that recompute their attention
  int* attn_n = nullptr;        // their count
  int32_t* attn_samp = nullptr; // [T + 1] where each sample's tokens start in attn_rows
  int32_t* attn_rowof = nullptr; // [T, k + n_shared] FFN row of each branch (fused sync path)
  float* mod = nullptr;         // AdaLN: [L, B, 6D] modulation vectors of the current step
  int mod_b = 0;                // samples the last step's modulation holds
  void* ada_h = nullptr;        // AdaLN: [T, D] attention input h = LN-modulate(x)
  void** ada_w = nullptr;       // AdaLN: device array [L] of w_ada pointers
  float** ada_b = nullptr;      // AdaLN: device array [L] of b_ada pointers
  std::vector<void*> act;  // input of layer l (l >= 1)
  int* status_host = nullptr;
  int* status_dev = nullptr;
  int state_T = 0;
  const void* last_x_in = nullptr;
  std::string last_error;
  std::vector<void*> allocs;
  // moeca_step_host: double-buffered device staging, an upload and a
  // read-back stream, and the events that order them against the steps.
  struct HostIo {
    bool ready = false;
    void* in[2] = {nullptr, nullptr};
    void* out[2] = {nullptr, nullptr};
    float* cond[2] = {nullptr, nullptr};
    cudaStream_t up_stream = nullptr, back_stream = nullptr;
    cudaEvent_t up[2] = {nullptr, nullptr}, done[2] = {nullptr, nullptr}, back[2] = {nullptr, nullptr};
    long long calls = 0;
  } hio;
  // Token-sharded step in progress (moeca_shard_begin / moeca_shard_next).
  struct ShardRun {
    bool active = false;
    int layer = 0, T = 0, world = 1, total = 0;
    bool refresh = false;
    float tau0 = 0.f;
    const void* x_in = nullptr;
    void* x_out = nullptr;
  } sh;
  float* shard_send = nullptr;  // caller's [blocks, E] float2: this rank's block partials
  float* shard_recv = nullptr;  // caller's [world x blocks, E] float2: every rank's, in rank order
  bool timing = false;
  std::vector<cudaEvent_t> event_pool;
  std::vector<PendingTiming> pending;
  double total_ms[MOECA_K_COUNT] = {};
  int64_t launches[MOECA_K_COUNT] = {};
};

namespace {

moeca_status fail(moeca_handle* h, moeca_status s, const std::string& msg) {
  if (h) h->last_error = msg;
  else g_create_error = msg;
  return s;
}

moeca_status cuda_fail(moeca_handle* h, cudaError_t e, const char* what) {
  return fail(h, MOECA_ERR_CUDA, std::string(what) + ": " + cudaGetErrorString(e));
}

bool dev_alloc(moeca_handle* h, void** p, size_t bytes) {
  if (bytes == 0) bytes = 16;
  if (cudaMalloc(p, bytes) != cudaSuccess) {
    cudaGetLastError();
    *p = nullptr;
    return false;
  }
  h->allocs.push_back(*p);
  if (cudaMemset(*p, 0, bytes) != cudaSuccess) return false;
  return true;
}

void free_all(moeca_handle* h) {
  for (auto& L : h->layers)
    if (L.tc) tc_plan_destroy(L.tc);
  auto& io = h->hio;
  for (int b = 0; b < 2; ++b) {
    if (io.up[b]) cudaEventDestroy(io.up[b]);
    if (io.done[b]) cudaEventDestroy(io.done[b]);
    if (io.back[b]) cudaEventDestroy(io.back[b]);
    io.up[b] = io.done[b] = io.back[b] = nullptr;
  }
  if (io.up_stream) cudaStreamDestroy(io.up_stream);
  if (io.back_stream) cudaStreamDestroy(io.back_stream);
  io.up_stream = io.back_stream = nullptr;
  io.ready = false;
  for (void* p : h->allocs) cudaFree(p);
  h->allocs.clear();
  if (h->status_host) cudaFreeHost(h->status_host);
  h->status_host = nullptr;
  for (auto ev : h->event_pool) cudaEventDestroy(ev);
  for (auto& pt : h->pending) {
    cudaEventDestroy(pt.start);
    cudaEventDestroy(pt.stop);
  }
  h->event_pool.clear();
  h->pending.clear();
}

cudaEvent_t take_event(moeca_handle* h) {
  if (!h->event_pool.empty()) {
    cudaEvent_t e = h->event_pool.back();
    h->event_pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  cudaEventCreate(&e);
  return e;
}

// Launch `fn` with optional CUDA events around it.
// Scoped NVTX range for profilers (layer and kernel launches of a step).
struct NvtxRange {
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};

template <typename Fn>
cudaError_t timed(moeca_handle* h, int kind, cudaStream_t s, Fn&& fn) {
  // An NVTX range per launch (a no-op unless a profiler is attached).
  static const char* const kNames[MOECA_K_COUNT] = {"router", "select", "compact", "ffn1", "ffn2", "combine",
                                                   "prep", "ffn", "qkv", "attn", "oproj", "attn_aux",
                                                   "adaln"};
  NvtxRange range(kNames[kind]);
  if (!h->timing) return fn();
  PendingTiming pt{kind, take_event(h), take_event(h)};
  cudaEventRecord(pt.start, s);
  cudaError_t e = fn();
  cudaEventRecord(pt.stop, s);
  h->pending.push_back(pt);
  return e;
}

moeca_status check_device_status(moeca_handle* h) {
  volatile int* st = h->status_host;
  const int code = st[0];
  if (code == 0) return MOECA_OK;
  char buf[160];
  snprintf(buf, sizeof buf, "device status %d (detail %d) from an earlier kernel", code, st[1]);
  return fail(h, code == kStatusWaitTimeout ? MOECA_ERR_TIMEOUT : MOECA_ERR_DEVICE_STATUS, buf);
}

bool overlaps(const void* a, const void* b, size_t n) {
  const char* x = static_cast<const char*>(a);
  const char* y = static_cast<const char*>(b);
  return x < y + n && y < x + n;
}

// Launch arguments shared by the whole-step path and the token-sharded one.
SelectArgs select_args(const moeca_handle* h, const LayerBuf& L, int T, bool refresh) {
  const moeca_config& c = h->cfg;
  SelectArgs sa{};
  sa.T = T; sa.k = c.top_k; sa.E = c.n_experts; sa.G = h->G; sa.refresh = refresh;
  sa.lambda1 = c.lambda1; sa.lambda2 = c.lambda2;
  sa.score_terms = c.score_terms; sa.token_level = c.granularity;
  sa.reused_meta_policy = c.reused_meta_policy; sa.shared_policy = c.shared_policy; sa.n_shared = c.n_shared;
  sa.route_e = L.route_e; sa.route_w = L.route_w; sa.tau = L.tau;
  sa.cache_e = L.cache_e; sa.cache_w = L.cache_w; sa.cache_norm = L.cache_norm;
  sa.recompute = L.recompute; sa.slot = L.slot; sa.matched = L.matched; sa.token_any = L.token_any;
  sa.block_counts = h->block_counts; sa.block_offsets = h->block_offsets;
  sa.counts = L.counts; sa.offsets = L.offsets; sa.done = h->done + 1;
  sa.stats = L.stats; sa.status = h->status_dev;
  return sa;
}

// The fused preparation kernel's arguments for the MoE layer alone (no
// attention sub-layer); the epoch is taken by the caller.
PrepArgs prep_args_plain(const moeca_handle* h, const LayerBuf& L, const void* moe_in, int T, float tau0,
                         const SelectArgs& sa, void* xg) {
  const moeca_config& c = h->cfg;
  PrepArgs pa{};
  pa.x = moe_in; pa.w_gate = L.w.w_gate; pa.b_gate = L.w.b_gate;
  pa.n_shared = c.n_shared;
  pa.T = T; pa.D = c.hidden; pa.E = c.n_experts; pa.k = c.top_k; pa.G = h->G;
  pa.renorm = c.renorm_topk; pa.entropy_norm = c.entropy_norm;
  pa.beta = c.beta; pa.tau0 = tau0; pa.alpha = c.alpha;
  pa.route_e = L.route_e; pa.route_w = L.route_w; pa.ema = L.ema; pa.tau = L.tau;
  pa.sel = sa;
  pa.part_words = h->prep_words; pa.count_words = h->prep_words + h->prep_count_off;
  pa.counts = L.counts; pa.offsets = L.offsets; pa.list = L.list;
  pa.xg = xg; pa.stats = L.stats; pa.status = h->status_dev;
  // The head of the routed W1, in the GEMM's expert order (a whole number of 16-byte units).
  const size_t w1_bytes = static_cast<size_t>(c.n_experts) * c.ffn * c.hidden * h->es;
  pa.l2_pf = L.w.w1;
  pa.l2_pf_bytes = std::min(w1_bytes, static_cast<size_t>(c.weight_prefetch_mb) << 20) & ~size_t(15);
  return pa;
}

FfnArgs ffn_args(const moeca_handle* h, const LayerBuf& L, int T, const void* moe_in) {
  const moeca_config& c = h->cfg;
  FfnArgs fa{};
  fa.G = h->G; fa.E = c.n_experts; fa.D = c.hidden; fa.F = c.ffn; fa.k = c.top_k; fa.T = T;
  fa.max_rows = T * (c.top_k + c.n_shared);
  fa.counts = L.counts; fa.offsets = L.offsets; fa.list = L.list;
  fa.xg = h->xg; fa.hmid = h->hmid; fa.x = kGemmGathersRows ? moe_in : nullptr;
  fa.w1 = L.w.w1; fa.w2 = L.w.w2; fa.ws1 = L.w.ws1; fa.ws2 = L.w.ws2;
  fa.cache_h = L.cache_h; fa.shared_h = L.shared_h; fa.gelu_tanh = c.gelu_tanh; fa.status = h->status_dev;
  fa.partial = h->simt_partial ? h->simt_partial : h->tc_partial; fa.tile_sem = h->tc_sem;
  fa.simt_split = h->simt_split;
  fa.dep = h->tc_dep; fa.max_mtiles = h->tc_dep_pairs_n; fa.work = h->tc_work;
  return fa;
}

CombineArgs combine_args(const moeca_handle* h, const LayerBuf& L, int T, const void* resid, void* out, bool refresh,
                         bool use_tc) {
  const moeca_config& c = h->cfg;
  CombineArgs cb{};
  cb.T = T; cb.D = c.hidden; cb.k = c.top_k; cb.n_shared = c.n_shared;
  cb.x = resid; cb.out = out; cb.cache_h = L.cache_h; cb.shared_h = L.shared_h;
  cb.route_w = L.route_w; cb.slot = L.slot; cb.cache_norm = L.cache_norm; cb.status = h->status_dev;
  cb.n_sms = h->n_sms; cb.direct = c.combine_direct;
  if (L.cache_y) {
    // Sec. 4.1, token level: a token with an empty recompute set returns y^{t0}.
    cb.cache_y = L.cache_y; cb.token_any = L.token_any; cb.copy_y = refresh ? 0 : 1;
  }
  cb.rearm = use_tc ? h->tc_work : nullptr;
  // A fully reused token's rows are not written by this layer's GEMM.
  cb.token_any = L.token_any;
  cb.early = !refresh && !L.cache_y && (c.n_shared == 0 || c.shared_policy == 0) ? 1 : 0;
  return cb;
}

}  // namespace

extern "C" {

void moeca_config_default(moeca_config* c) {
  if (!c) return;
  std::memset(c, 0, sizeof *c);
  c->n_layers = 1;
  c->n_shared = 0;
  c->max_tokens = 1;
  c->dtype = MOECA_BF16;
  c->lambda1 = 1.0f;
  c->lambda2 = 0.5f;
  c->tau0 = 0.8f;
  c->alpha = 0.6f;
  c->beta = 0.65f;
  c->refresh_period = 0;
  c->renorm_topk = 1;
  c->entropy_norm = 0;
  c->shared_policy = 0;
  c->reused_meta_policy = 0;
  c->score_terms = 7;
  c->granularity = 0;
  c->gelu_tanh = 1;
  c->ffn_impl = MOECA_FFN_AUTO;
  c->n_heads = 0;
  c->seq_len = 0;
  c->attn_policy = 0;
  c->attn_impl = 0;
  c->adaln = 0;
  c->ln_eps = 1e-6f;
  c->keep_route_in = 0;
  c->token_reuse_policy = 0;
  c->combine_direct = 1;
  c->weight_prefetch_mb = 16;
}

const char* moeca_status_string(moeca_status s) {
  switch (s) {
    case MOECA_OK: return "ok";
    case MOECA_ERR_INVALID_ARG: return "invalid argument";
    case MOECA_ERR_UNSUPPORTED: return "unsupported";
    case MOECA_ERR_CUDA: return "CUDA error";
    case MOECA_ERR_OOM: return "out of device memory";
    case MOECA_ERR_STATE: return "invalid state";
    case MOECA_ERR_TIMEOUT: return "device wait timed out";
    case MOECA_ERR_DEVICE_STATUS: return "device status error";
  }
  return "unknown status";
}

const char* moeca_last_error(const moeca_handle* h) {
  return h ? h->last_error.c_str() : g_create_error.c_str();
}

moeca_status moeca_create(const moeca_config* cfg, const moeca_layer_weights* layers,
                          int32_t device, moeca_handle** out) {
  g_create_error.clear();
  if (!out) return fail(nullptr, MOECA_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  if (!cfg || !layers) return fail(nullptr, MOECA_ERR_INVALID_ARG, "cfg or layers is NULL");
  const moeca_config& c = *cfg;
  const bool bf16 = c.dtype == MOECA_BF16;
  if (c.dtype != MOECA_F32 && c.dtype != MOECA_BF16) return fail(nullptr, MOECA_ERR_INVALID_ARG, "dtype");
  if (c.n_layers < 1 || c.hidden < 1 || c.ffn < 1 || c.max_tokens < 1)
    return fail(nullptr, MOECA_ERR_INVALID_ARG, "n_layers, hidden, ffn and max_tokens must be >= 1");
  if (c.n_experts < 1 || c.n_experts > kMaxExperts)
    return fail(nullptr, MOECA_ERR_INVALID_ARG, "n_experts must be in [1, 64]");
  if (c.top_k < 1 || c.top_k > kMaxTopK || c.top_k > c.n_experts)
    return fail(nullptr, MOECA_ERR_INVALID_ARG, "top_k must be in [1, min(8, n_experts)]");
  if (c.n_shared != 0 && c.n_shared != 1) return fail(nullptr, MOECA_ERR_INVALID_ARG, "n_shared must be 0 or 1");
  if (!(c.alpha >= 0.f && c.alpha < 1.f) || !(c.beta >= 0.f && c.beta < 1.f))
    return fail(nullptr, MOECA_ERR_INVALID_ARG, "alpha and beta must be in [0, 1)");
  if (std::isnan(c.tau0) || !std::isfinite(c.lambda1) || !std::isfinite(c.lambda2))
    return fail(nullptr, MOECA_ERR_INVALID_ARG, "tau0, lambda1, lambda2");
  if (c.score_terms < 1 || c.score_terms > 7 || (c.granularity != 0 && c.granularity != 1))
    return fail(nullptr, MOECA_ERR_INVALID_ARG, "score_terms must be 1..7 and granularity 0 or 1");
  if (c.refresh_period < 0) return fail(nullptr, MOECA_ERR_INVALID_ARG, "refresh_period < 0");
  if (c.token_reuse_policy != 0 && c.token_reuse_policy != 1)
    return fail(nullptr, MOECA_ERR_INVALID_ARG, "token_reuse_policy must be 0 or 1");
  if (c.combine_direct != 0 && c.combine_direct != 1)
    return fail(nullptr, MOECA_ERR_INVALID_ARG, "combine_direct must be 0 or 1");
  if (c.weight_prefetch_mb < 0 || c.weight_prefetch_mb > 4096)
    return fail(nullptr, MOECA_ERR_INVALID_ARG, "weight_prefetch_mb must be in [0, 4096]");
  if (c.ffn_impl != MOECA_FFN_AUTO && c.ffn_impl != MOECA_FFN_SIMT)
    return fail(nullptr, MOECA_ERR_INVALID_ARG, "ffn_impl");
  if ((c.ffn_tile_n != 0 && c.ffn_tile_n != 64 && c.ffn_tile_n != 128 && c.ffn_tile_n != 192 &&
       c.ffn_tile_n != 256) || c.ffn_split_k < 0 || c.ffn_split_k > 4)
    return fail(nullptr, MOECA_ERR_INVALID_ARG, "ffn_tile_n must be 0/64/128/192/256, ffn_split_k 0..4");
  if (c.n_heads < 0 || c.seq_len < 0 || c.attn_policy < 0 || c.attn_policy > 2 || c.attn_impl < 0 ||
      c.attn_impl > 2)
    return fail(nullptr, MOECA_ERR_INVALID_ARG, "n_heads and seq_len must be >= 0, attn_policy 0..2, attn_impl 0..2");
  const bool attn = c.n_heads > 0;
  if (attn && !bf16) return fail(nullptr, MOECA_ERR_UNSUPPORTED, "the attention sub-layer is built for bf16 only");
  if (attn && (!attn_supported(c.hidden, c.n_heads) || c.hidden % 64))
    return fail(nullptr, MOECA_ERR_UNSUPPORTED,
                "attention needs hidden a multiple of 64 and hidden / n_heads in {64, 72, 80, 96, 128}");
  const bool ada = c.adaln != 0;
  if (c.adaln != 0 && c.adaln != 1) return fail(nullptr, MOECA_ERR_INVALID_ARG, "adaln must be 0 or 1");
  if (ada && !attn) return fail(nullptr, MOECA_ERR_UNSUPPORTED, "AdaLN modulates a DiT-MoE block: n_heads > 0");
  if (ada && c.hidden > kAdaLnMaxD) return fail(nullptr, MOECA_ERR_UNSUPPORTED, "AdaLN blocks support hidden <= 2560");
  if (ada && !(c.ln_eps > 0.f && std::isfinite(c.ln_eps))) return fail(nullptr, MOECA_ERR_INVALID_ARG, "ln_eps must be > 0");
  const int mod_b_max = ada ? std::max(1, c.seq_len ? c.max_tokens / c.seq_len : 1) : 0;
  if (ada && ada_mod_smem(mod_b_max, c.hidden) > 200 * 1024)
    return fail(nullptr, MOECA_ERR_UNSUPPORTED, "AdaLN: samples x hidden x 4 bytes must fit 200 KB of shared memory");
  const int vec = bf16 ? 8 : 4;
  if (c.hidden % vec) return fail(nullptr, MOECA_ERR_UNSUPPORTED, "hidden must be a multiple of 8 (bf16) / 4 (fp32)");
  const bool use_tc = bf16 && c.ffn_impl == MOECA_FFN_AUTO;
  if (use_tc && (c.hidden % 64 || c.ffn % 64))
    return fail(nullptr, MOECA_ERR_UNSUPPORTED, "the tensor-core FFN needs hidden and ffn multiples of 64");
  const size_t es = bf16 ? 2 : 4;
  const long long rows_ll = static_cast<long long>(c.max_tokens) * (c.top_k + c.n_shared);
  if (rows_ll > (1LL << 30) || static_cast<long long>(c.max_tokens) * c.top_k > (1LL << 30))
    return fail(nullptr, MOECA_ERR_INVALID_ARG, "max_tokens too large");
  for (int l = 0; l < c.n_layers; ++l) {
    const moeca_layer_weights& w = layers[l];
    if (!w.w_gate || !w.w1 || !w.w2) return fail(nullptr, MOECA_ERR_INVALID_ARG, "layer weight pointer is NULL");
    if (c.n_shared && (!w.ws1 || !w.ws2)) return fail(nullptr, MOECA_ERR_INVALID_ARG, "shared expert weights are NULL");
    if (attn && (!w.w_qkv || !w.w_o)) return fail(nullptr, MOECA_ERR_INVALID_ARG, "attention weights are NULL");
    if (ada && !w.w_ada) return fail(nullptr, MOECA_ERR_INVALID_ARG, "AdaLN weights are NULL");
    const void* ps[] = {w.w_gate, w.w1, w.w2, w.ws1, w.ws2, attn ? w.w_qkv : nullptr, attn ? w.b_qkv : nullptr,
                        attn ? w.w_o : nullptr, attn ? w.b_o : nullptr, ada ? w.w_ada : nullptr,
                        ada ? w.b_ada : nullptr};
    for (const void* p : ps)
      if (reinterpret_cast<uintptr_t>(p) % 16) return fail(nullptr, MOECA_ERR_INVALID_ARG, "weights must be 16-byte aligned");
  }
  int ndev = 0;
  cudaError_t ce = cudaGetDeviceCount(&ndev);
  if (ce != cudaSuccess) { cudaGetLastError(); return fail(nullptr, MOECA_ERR_CUDA, std::string("no CUDA device: ") + cudaGetErrorString(ce)); }
  if (device < 0 || device >= ndev) return fail(nullptr, MOECA_ERR_INVALID_ARG, "device out of range");
  if ((ce = cudaSetDevice(device)) != cudaSuccess) return fail(nullptr, MOECA_ERR_CUDA, cudaGetErrorString(ce));

  moeca_handle* h = new (std::nothrow) moeca_handle();
  if (!h) return fail(nullptr, MOECA_ERR_OOM, "host allocation failed");
  h->cfg = c;
  h->device = device;
  h->bf16 = bf16;
  h->es = es;
  h->G = c.n_experts + c.n_shared;
  h->max_rows = static_cast<int>(rows_ll);
  cudaDeviceGetAttribute(&h->n_sms, cudaDevAttrMultiProcessorCount, device);
  const size_t T = c.max_tokens, k = c.top_k, D = c.hidden, E = c.n_experts, G = h->G, F = c.ffn;
  bool ok = true;
  auto A = [&](void** p, size_t bytes) { ok = ok && dev_alloc(h, p, bytes); };
  h->layers.resize(c.n_layers);
  for (int l = 0; l < c.n_layers && ok; ++l) {
    LayerBuf& L = h->layers[l];
    L.w = layers[l];
    A((void**)&L.cache_e, T * k * 4);
    A((void**)&L.cache_w, T * k * 4);
    A((void**)&L.cache_norm, T * k * 4);
    A(&L.cache_h, T * k * D * es);
    if (c.n_shared) A(&L.shared_h, T * D * es);
    A((void**)&L.ema, T * E * 4);
    A((void**)&L.route_e, T * k * 4);
    A((void**)&L.route_w, T * k * 4);
    A((void**)&L.tau, E * 4);
    A((void**)&L.recompute, T * k);
    A((void**)&L.slot, T * k);
    A((void**)&L.matched, T * k);
    A((void**)&L.token_any, T);
    A((void**)&L.counts, G * 4);
    A((void**)&L.offsets, (G + 1) * 4);
    A((void**)&L.list, static_cast<size_t>(h->max_rows) * 4);
    A((void**)&L.stats, kStCount * 8);
    if (attn) {
      A(&L.attn_a, T * D * es);
      A(&L.attn_u, T * D * es);
    }
    if (ada) {
      A(&L.attn_m, T * D * es);
      if (c.keep_route_in) A(&L.route_m, T * D * es);
    }
    if (c.token_reuse_policy) A((void**)&L.cache_y, T * D * 4);
  }
  if (ada) {
    A(&h->ada_h, T * D * es);
    A((void**)&h->mod, static_cast<size_t>(c.n_layers) * mod_b_max * 6 * D * 4);
    A((void**)&h->ada_w, c.n_layers * sizeof(void*));
    A((void**)&h->ada_b, c.n_layers * sizeof(float*));
    if (ok) {
      std::vector<const void*> wp(c.n_layers);
      std::vector<const float*> bp(c.n_layers);
      for (int l = 0; l < c.n_layers; ++l) {
        wp[l] = layers[l].w_ada;
        bp[l] = layers[l].b_ada;
      }
      ok = cudaMemcpy(h->ada_w, wp.data(), c.n_layers * sizeof(void*), cudaMemcpyHostToDevice) == cudaSuccess &&
           cudaMemcpy(h->ada_b, bp.data(), c.n_layers * sizeof(float*), cudaMemcpyHostToDevice) == cudaSuccess;
    }
  }
  if (attn) {
    A(&h->qkv, T * 3 * D * es);
    A(&h->attn_o, T * D * es);
    A((void**)&h->attn_rows, T * 4);
    A((void**)&h->attn_n, 16);
    A((void**)&h->attn_samp, (T + 1) * 4);
    A((void**)&h->attn_inv, T * 4);
    A((void**)&h->attn_rowof, T * (k + c.n_shared) * 4);
  }
  const size_t nblk_router = (T + kRouterTokensPerBlock - 1) / kRouterTokensPerBlock;
  const size_t nblk_sel = (T + kSelectTokensPerBlock - 1) / kSelectTokensPerBlock;
  A((void**)&h->partials, nblk_router * E * 2 * 4);
  A((void**)&h->done, 2 * 4);
  A((void**)&h->block_counts, nblk_sel * G * 4);
  A((void**)&h->block_offsets, nblk_sel * G * 4);
  A(&h->xg, static_cast<size_t>(h->max_rows) * D * es);
  A(&h->hmid, static_cast<size_t>(h->max_rows) * F * es);
  if (!use_tc && !bf16) {
    // fp32: the second GEMM (few outputs, long K) in K splits, their partials
    // added in split order by a second pass; four splits while the workspace
    // stays within 512 MB.
    for (int sk = 4; sk > 1; sk /= 2) {
      if (static_cast<size_t>(sk) * h->max_rows * D * 4 <= (size_t(512) << 20)) {
        h->simt_split = sk;
        break;
      }
    }
    if (h->simt_split > 1) A((void**)&h->simt_partial, static_cast<size_t>(h->simt_split) * h->max_rows * D * 4);
  }
  if (use_tc) {
    A((void**)&h->tc_partial, tc_partial_bytes(h->n_sms));
    A((void**)&h->tc_sem, tc_split_units(h->n_sms) * sizeof(int));
    h->tc_dep_pairs_n = static_cast<int>(tc_dep_pairs(h->max_rows, h->G));
    A((void**)&h->tc_dep, static_cast<size_t>(h->tc_dep_pairs_n) * 2 * sizeof(int));
    A((void**)&h->tc_work, 2 * sizeof(int));
    // An AdaLN block forms its router input in its own kernel: the plain
    // preparation kernel, with the attention list built separately.
    h->prep = prep_plan(c.hidden, c.n_experts, c.top_k, c.max_tokens, h->n_sms, attn && !ada);
    if (h->prep.tokens_per_block) {
      const size_t nb = (T + h->prep.tokens_per_block - 1) / h->prep.tokens_per_block;
      h->prep_count_off = nb * E * 2;
      h->prep_words_n = h->prep_count_off + nb * (G + 1);
      A((void**)&h->prep_words, h->prep_words_n * 8);
    }
  }
  h->act.assign(c.n_layers, nullptr);
  for (int l = 1; l < c.n_layers && ok; ++l) A(&h->act[l], T * D * es);
  if (!ok) {
    free_all(h);
    delete h;
    return fail(nullptr, MOECA_ERR_OOM, "device allocation failed");
  }
  if ((ce = cudaHostAlloc((void**)&h->status_host, 4 * sizeof(int), cudaHostAllocMapped)) != cudaSuccess ||
      (ce = cudaHostGetDevicePointer((void**)&h->status_dev, h->status_host, 0)) != cudaSuccess) {
    cudaGetLastError();
    free_all(h);
    delete h;
    return fail(nullptr, MOECA_ERR_CUDA, std::string("status word: ") + cudaGetErrorString(ce));
  }
  std::memset(h->status_host, 0, 4 * sizeof(int));
  if (use_tc) {
    for (int l = 0; l < c.n_layers; ++l) {
      LayerBuf& L = h->layers[l];
      FfnArgs fa{};
      fa.G = h->G; fa.E = c.n_experts; fa.D = c.hidden; fa.F = c.ffn; fa.k = c.top_k; fa.T = c.max_tokens;
      fa.max_rows = h->max_rows;
      fa.xg = h->xg; fa.hmid = h->hmid;
      fa.w1 = L.w.w1; fa.w2 = L.w.w2; fa.ws1 = L.w.ws1; fa.ws2 = L.w.ws2;
      fa.tile_n = c.ffn_tile_n; fa.split_k = c.ffn_split_k;
      char err[256] = {0};
      L.tc = tc_plan_create(fa, h->n_sms, err, sizeof err);
      if (!L.tc) {
        free_all(h);
        delete h;
        return fail(nullptr, MOECA_ERR_CUDA, std::string("tensor-core plan: ") + err);
      }
    }
  }
  if ((ce = cudaDeviceSynchronize()) != cudaSuccess) {
    free_all(h);
    delete h;
    return fail(nullptr, MOECA_ERR_CUDA, cudaGetErrorString(ce));
  }
  *out = h;
  return MOECA_OK;
}

moeca_status moeca_step(moeca_handle* h, const void* x_in, void* x_out, const moeca_step_args* args,
                        void* stream) {
  if (!h) return fail(nullptr, MOECA_ERR_INVALID_ARG, "handle is NULL");
  if (!args) return fail(h, MOECA_ERR_INVALID_ARG, "args is NULL");
  const moeca_config& c = h->cfg;
  const int T = args->n_tokens;
  if (T < 0 || T > c.max_tokens) return fail(h, MOECA_ERR_INVALID_ARG, "n_tokens out of [0, max_tokens]");
  moeca_status st = check_device_status(h);
  if (st != MOECA_OK) return st;
  if (T == 0) return MOECA_OK;
  if (!x_in || !x_out) return fail(h, MOECA_ERR_INVALID_ARG, "x_in or x_out is NULL");
  const size_t xbytes = static_cast<size_t>(T) * c.hidden * h->es;
  if (overlaps(x_in, x_out, xbytes)) return fail(h, MOECA_ERR_INVALID_ARG, "x_in and x_out overlap");
  if (reinterpret_cast<uintptr_t>(x_in) % 16 || reinterpret_cast<uintptr_t>(x_out) % 16)
    return fail(h, MOECA_ERR_INVALID_ARG, "x_in and x_out must be 16-byte aligned");
  cudaSetDevice(h->device);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  bool all_valid = h->state_T == T;
  for (auto& L : h->layers) all_valid = all_valid && L.valid;
  const int N = c.refresh_period;
  const bool refresh = args->force_refresh || !all_valid || (N > 0 && args->step_index % N == 0);
  if (h->state_T != T) {
    // A new token count starts a new trajectory: the EMA positions restart.
    for (auto& L : h->layers) {
      cudaError_t e = cudaMemsetAsync(L.ema, 0, static_cast<size_t>(c.max_tokens) * c.n_experts * 4, s);
      if (e != cudaSuccess) return cuda_fail(h, e, "reset EMA");
      L.valid = false;
    }
  }
  const float tau0 = std::isnan(args->tau0_override) ? c.tau0 : args->tau0_override;
  const bool use_tc = h->bf16 && c.ffn_impl == MOECA_FFN_AUTO;
  const bool attn = c.n_heads > 0;
  const int seq = c.seq_len ? c.seq_len : T;
  if (attn && (T % seq || seq % 8))
    return fail(h, MOECA_ERR_INVALID_ARG, "n_tokens must be a multiple of seq_len, and seq_len of 8");
  // The tcgen05 attention core pays off once a CTA streams at least four
  // 128-key blocks; shorter samples go to the warp-level core.
  const bool use_attn_tc = c.attn_impl == 2 || (c.attn_impl == 0 && seq >= 512);
  const bool ada = c.adaln != 0;
  const int n_samp = T / seq;
  const size_t mod_ld = static_cast<size_t>(6) * c.hidden;
  if (ada && !args->cond) return fail(h, MOECA_ERR_INVALID_ARG, "an AdaLN stack needs cond");
  cudaError_t e = cudaSuccess;
  NvtxRange step_range("moeca_step");
  if (ada) {
    // Every layer's six modulation vectors per sample, from this step's c.
    AdaModArgs ma{};
    ma.L = c.n_layers; ma.B = n_samp; ma.D = c.hidden; ma.cond = args->cond;
    ma.w = h->ada_w; ma.b = h->ada_b; ma.out = h->mod;
    if ((e = timed(h, MOECA_K_ADALN, s, [&] { return launch_ada_mod(ma, h->n_sms, s); })) != cudaSuccess) {
      for (auto& L : h->layers) L.valid = false;
      return cuda_fail(h, e, "kernel launch");
    }
    h->mod_b = n_samp;
  }
  for (int l = 0; l < c.n_layers; ++l) {
    LayerBuf& L = h->layers[l];
    NvtxRange layer_range("layer");
    const void* in = l == 0 ? x_in : h->act[l];
    void* out = l + 1 == c.n_layers ? x_out : h->act[l + 1];
    const bool attn_full = attn && (refresh || c.attn_policy == 2);
    const bool attn_sync = attn && !attn_full && c.attn_policy == 0;
    // The MoE sub-layer's input: the layer input, u of a DiT-MoE block, or
    // m = LN-modulate(u) of an AdaLN block; its residual: the input or u.
    const void* moe_in = ada ? L.attn_m : (attn ? L.attn_u : in);
    const void* resid = attn ? L.attn_u : in;
    const float* mod_l = ada ? h->mod + static_cast<size_t>(l) * n_samp * mod_ld : nullptr;
    AdaLnArgs la{};
    la.T = T; la.D = c.hidden; la.seq = seq; la.eps = c.ln_eps; la.mod = mod_l;
    la.x = in; la.u = L.attn_u; la.status = h->status_dev;
    const size_t TD = static_cast<size_t>(T) * c.hidden;
    void* q_buf = h->qkv;
    void* k_buf = static_cast<char*>(h->qkv) + TD * h->es;
    void* vt_buf = static_cast<char*>(h->qkv) + 2 * TD * h->es;
    ProjArgs qa{};
    qa.A = ada ? h->ada_h : in; qa.a_rows = T; qa.B = L.w.w_qkv; qa.bias = L.w.b_qkv;
    qa.M = T; qa.N = 3 * c.hidden; qa.K = c.hidden; qa.mode = kProjQKV;
    qa.q_out = q_buf; qa.k_out = k_buf; qa.vt_out = vt_buf; qa.n_tok = T; qa.status = h->status_dev;
    AttnArgs aa{};
    aa.q = q_buf; aa.k = k_buf; aa.vt = vt_buf; aa.T = T; aa.D = c.hidden; aa.H = c.n_heads; aa.S = seq;
    aa.o = h->attn_o; aa.status = h->status_dev;
    ProjArgs oa{};
    oa.A = h->attn_o; oa.a_rows = T; oa.B = L.w.w_o; oa.bias = L.w.b_o;
    oa.M = T; oa.N = c.hidden; oa.K = c.hidden; oa.mode = kProjResidual;
    // Narrow tiles at moderate width: the recomputed rows are few and the
    // residual epilogue (x in; a, u and the FFN rows out) is latency-bound,
    // so more CTAs with two 32-column chunks each beat fewer wide ones.  At
    // D above 2048 the K loop dominates and narrow tiles would re-read the
    // operands four times over: the widest tile.
    oa.tile_n = c.hidden > 2048 ? 0 : 64;
    oa.n_tok = T; oa.x = in; oa.a_out = L.attn_a; oa.u_out = L.attn_u;
    if (ada) {
      oa.mode = kProjResidualGated;
      oa.gate = mod_l + 2 * c.hidden; oa.gate_ld = static_cast<int>(mod_ld); oa.seq = seq;
    }
    oa.row_stat = L.stats + kStAttnRows; oa.status = h->status_dev;
    if (attn_sync) {
      aa.rows = h->attn_rows; aa.sample_lo = h->attn_samp;
      qa.inv = h->attn_inv;
      oa.rows = h->attn_rows; oa.m_dev = h->attn_n;
    }
    if (attn_full) {
      // Every token's attention output, before the router sees u = x + a.
      if (ada) {
        AdaLnArgs ha = la;
        ha.h_out = h->ada_h;
        if ((e = timed(h, MOECA_K_ADALN, s, [&] { return launch_adaln_rows(ha, s); })) != cudaSuccess) break;
      }
      if ((e = timed(h, MOECA_K_QKV, s, [&] { return launch_proj_tc(qa, s); })) != cudaSuccess) break;
      if ((e = timed(h, MOECA_K_ATTN, s, [&] {
             return use_attn_tc ? launch_attn_tc(aa, s) : launch_attn_core(aa, s);
           })) != cudaSuccess) break;
      if ((e = timed(h, MOECA_K_OPROJ, s, [&] { return launch_proj_tc(oa, s); })) != cudaSuccess) break;
      if (ada) {
        AdaLnArgs mm = la;
        mm.m_out = L.attn_m; mm.m_copy = L.route_m;
        if ((e = timed(h, MOECA_K_ADALN, s, [&] { return launch_adaln_rows(mm, s); })) != cudaSuccess) break;
      }
    } else if (ada) {
      // u' = x + g_a a^{t0} and the router input m' for every token, and (sync
      // rule) the attention input h, in one pass over the rows.
      AdaLnArgs pa0 = la;
      pa0.a = L.attn_a; pa0.m_out = L.attn_m; pa0.m_copy = L.route_m;
      pa0.h_out = attn_sync ? h->ada_h : nullptr;
      if ((e = timed(h, MOECA_K_ADALN, s, [&] { return launch_adaln_rows(pa0, s); })) != cudaSuccess) break;
    } else if (attn && h->prep.tokens_per_block == 0) {
      // u' = x + a^{t0}: the router input, and the MoE input of every token
      // that keeps its cached attention (the fused preparation kernel forms
      // it itself while staging the rows).
      if ((e = timed(h, MOECA_K_ATTN_AUX, s, [&] {
             return launch_attn_residual(in, L.attn_a, L.attn_u, T, c.hidden, h->status_dev, s);
           })) != cudaSuccess)
        break;
    }
    // Under the sync rule the rows' inputs change after the decision: the
    // FFN rows are gathered once the attention update is done.
    const bool xg_gather = !(use_tc && kGemmGathersRows);  // the FFN reads gathered rows
    void* xg_now = !xg_gather || attn_sync ? nullptr : h->xg;

    const bool fused = h->prep.tokens_per_block != 0;
    RouterArgs ra{};
    ra.x = moe_in; ra.w_gate = L.w.w_gate; ra.b_gate = L.w.b_gate;
    ra.T = T; ra.D = c.hidden; ra.E = c.n_experts; ra.k = c.top_k;
    ra.renorm = c.renorm_topk; ra.beta = c.beta; ra.tau0 = tau0; ra.alpha = c.alpha;
    ra.entropy_norm = c.entropy_norm;
    ra.route_e = L.route_e; ra.route_w = L.route_w; ra.ema = L.ema;
    ra.partials = h->partials; ra.done = h->done; ra.tau = L.tau; ra.stats = L.stats;
    ra.status = h->status_dev;

    SelectArgs sa = select_args(h, L, T, refresh);

    CompactArgs ca{};
    ca.T = T; ca.k = c.top_k; ca.E = c.n_experts; ca.G = h->G; ca.D = c.hidden; ca.n_shared = c.n_shared;
    ca.refresh = refresh; ca.shared_policy = c.shared_policy;
    ca.route_e = L.route_e; ca.recompute = L.recompute; ca.slot = L.slot; ca.token_any = L.token_any;
    ca.block_offsets = h->block_offsets; ca.offsets = L.offsets; ca.list = L.list;
    ca.x = moe_in; ca.xg = xg_now; ca.status = h->status_dev;
    if (fused) {
      PrepArgs pa = prep_args_plain(h, L, moe_in, T, tau0, sa, xg_now);
      if (attn && !ada && !attn_full) {
        pa.x = in;
        pa.attn_a = L.attn_a;
        pa.u_out = L.attn_u;
      }
      if (attn_sync && !ada) {
        // The recomputing-token list comes out of the same compaction.
        pa.attn_list = 1;
        pa.attn_rows = h->attn_rows; pa.attn_n = h->attn_n; pa.attn_inv = h->attn_inv;
        pa.sample_lo = h->attn_samp; pa.seq = seq;
      }
      if (attn_sync && !ada && xg_gather) {
        // The rows of tokens that keep their attention are final now; the
        // output projection writes the others (row_of says where).
        pa.xg = h->xg;
        pa.gather_final_only = 1;
        pa.row_of = h->attn_rowof;
        oa.row_of = h->attn_rowof;
        oa.row_w = c.top_k + c.n_shared;
        oa.xg = h->xg;
      }
      if (++h->prep_epoch == 0) h->prep_epoch = 1;  // 0 marks words never written
      pa.epoch = pa.wait_epoch = h->prep_epoch;
      if (h->inject_stall) pa.wait_epoch = h->prep_epoch ^ 0x80000000u;  // a tag no launch writes
      if ((e = timed(h, MOECA_K_PREP, s, [&] { return launch_prep(pa, h->prep, s); })) != cudaSuccess) break;
    } else {
      if ((e = timed(h, MOECA_K_ROUTER, s, [&] { return launch_router(ra, h->bf16, s); })) != cudaSuccess) break;
      if ((e = timed(h, MOECA_K_SELECT, s, [&] { return launch_select(sa, s); })) != cudaSuccess) break;
      if ((e = timed(h, MOECA_K_COMPACT, s, [&] { return launch_compact(ca, h->bf16, s); })) != cudaSuccess) break;
    }
    if (attn_sync) {
      // Sec. 4.1: the tokens with a non-empty recompute set recompute their
      // attention output over all keys of their sample; their a and u rows
      // are replaced, then the FFN rows are gathered from u.
      if ((!fused || ada) && (e = timed(h, MOECA_K_ATTN_AUX, s, [&] {
                       return launch_attn_rows(L.token_any, T, seq, h->attn_rows, h->attn_n, h->attn_samp,
                                               h->attn_inv, s);
                     })) != cudaSuccess)
        break;
      if ((e = timed(h, MOECA_K_QKV, s, [&] { return launch_proj_tc(qa, s); })) != cudaSuccess) break;
      if ((e = timed(h, MOECA_K_ATTN, s, [&] {
             return use_attn_tc ? launch_attn_tc(aa, s) : launch_attn_core(aa, s);
           })) != cudaSuccess) break;
      if ((e = timed(h, MOECA_K_OPROJ, s, [&] { return launch_proj_tc(oa, s); })) != cudaSuccess) break;
      if (ada) {
        // The listed tokens' MoE input m from their new u.
        AdaLnArgs mm = la;
        mm.m_out = L.attn_m; mm.rows = h->attn_rows; mm.n_rows = h->attn_n;
        if ((e = timed(h, MOECA_K_ADALN, s, [&] { return launch_adaln_rows(mm, s); })) != cudaSuccess) break;
      }
      if (xg_gather && (!fused || ada)) {
        CompactArgs ga = ca;
        ga.xg = h->xg;
        if ((e = timed(h, MOECA_K_ATTN_AUX, s, [&] { return launch_gather(ga, h->bf16, s); })) != cudaSuccess)
          break;
      }
    }

    FfnArgs fa = ffn_args(h, L, T, moe_in);
    if (use_tc) {
      // Both GEMMs in one persistent launch: phase-2 tiles start as soon as
      // the phase-1 tiles of their rows are stored.
      e = timed(h, MOECA_K_FFN, s, [&] { return launch_ffn_tc(L.tc, fa, 0, s); });
    } else {
      for (int phase = 1; phase <= 2 && e == cudaSuccess; ++phase) {
        const int kind = phase == 1 ? MOECA_K_FFN1 : MOECA_K_FFN2;
        e = timed(h, kind, s, [&] {
          return use_tc ? launch_ffn_tc(L.tc, fa, phase, s) : launch_ffn_simt(fa, h->bf16, phase, s);
        });
      }
    }
    if (e != cudaSuccess) break;

    CombineArgs cb = combine_args(h, L, T, resid, out, refresh, use_tc);
    if (ada) {
      cb.gate = mod_l + 5 * c.hidden; cb.gate_ld = static_cast<int>(mod_ld); cb.seq = seq;
    }
    if ((e = timed(h, MOECA_K_COMBINE, s, [&] { return launch_combine(cb, h->bf16, s); })) != cudaSuccess) break;
    L.valid = true;
  }
  if (e != cudaSuccess) {
    for (auto& L : h->layers) L.valid = false;
    h->inject_stall = false;
    return cuda_fail(h, e, "kernel launch");
  }
  h->state_T = T;
  h->last_x_in = x_in;
  h->inject_stall = false;
  return MOECA_OK;
}

moeca_status moeca_step_host(moeca_handle* h, const void* x_in_host, void* x_out_host, const moeca_step_args* args,
                             void* stream) {
  if (!h) return fail(nullptr, MOECA_ERR_INVALID_ARG, "handle is NULL");
  if (!args) return fail(h, MOECA_ERR_INVALID_ARG, "args is NULL");
  const moeca_config& c = h->cfg;
  const int T = args->n_tokens;
  if (T < 0 || T > c.max_tokens) return fail(h, MOECA_ERR_INVALID_ARG, "n_tokens out of [0, max_tokens]");
  if (T == 0) return moeca_step(h, nullptr, nullptr, args, stream);
  if (!x_in_host || !x_out_host) return fail(h, MOECA_ERR_INVALID_ARG, "x_in_host or x_out_host is NULL");
  const bool ada = c.adaln != 0;
  if (ada && !args->cond) return fail(h, MOECA_ERR_INVALID_ARG, "an AdaLN stack needs cond");
  cudaSetDevice(h->device);
  auto& io = h->hio;
  cudaError_t e = cudaSuccess;
  if (!io.ready) {
    const size_t xb = static_cast<size_t>(c.max_tokens) * c.hidden * h->es;
    const size_t cb = ada ? static_cast<size_t>(std::max(1, c.seq_len ? c.max_tokens / c.seq_len : 1)) * c.hidden * 4 : 0;
    bool ok = true;
    for (int b = 0; b < 2 && ok; ++b) {
      ok = dev_alloc(h, &io.in[b], xb) && dev_alloc(h, &io.out[b], xb);
      if (ok && cb) ok = dev_alloc(h, reinterpret_cast<void**>(&io.cond[b]), cb);
    }
    if (!ok) return fail(h, MOECA_ERR_OOM, "host staging buffers");
    if ((e = cudaStreamCreateWithFlags(&io.up_stream, cudaStreamNonBlocking)) != cudaSuccess ||
        (e = cudaStreamCreateWithFlags(&io.back_stream, cudaStreamNonBlocking)) != cudaSuccess)
      return cuda_fail(h, e, "host copy streams");
    for (int b = 0; b < 2; ++b)
      if ((e = cudaEventCreateWithFlags(&io.up[b], cudaEventDisableTiming)) != cudaSuccess ||
          (e = cudaEventCreateWithFlags(&io.done[b], cudaEventDisableTiming)) != cudaSuccess ||
          (e = cudaEventCreateWithFlags(&io.back[b], cudaEventDisableTiming)) != cudaSuccess)
        return cuda_fail(h, e, "host copy events");
    io.ready = true;
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int b = static_cast<int>(io.calls & 1);
  const size_t xbytes = static_cast<size_t>(T) * c.hidden * h->es;
  const bool reused = io.calls >= 2;  // buffers b were used by the call before the last
  // Upload: staging input b is free once the step two calls back has run.
  if (reused && (e = cudaStreamWaitEvent(io.up_stream, io.done[b], 0)) != cudaSuccess) return cuda_fail(h, e, "wait");
  if ((e = cudaMemcpyAsync(io.in[b], x_in_host, xbytes, cudaMemcpyHostToDevice, io.up_stream)) != cudaSuccess)
    return cuda_fail(h, e, "upload");
  moeca_step_args a = *args;
  if (ada) {
    const int seq = c.seq_len ? c.seq_len : T;
    const size_t cbytes = static_cast<size_t>(T / seq) * c.hidden * 4;
    if ((e = cudaMemcpyAsync(io.cond[b], args->cond, cbytes, cudaMemcpyHostToDevice, io.up_stream)) != cudaSuccess)
      return cuda_fail(h, e, "upload cond");
    a.cond = io.cond[b];
  }
  if ((e = cudaEventRecord(io.up[b], io.up_stream)) != cudaSuccess) return cuda_fail(h, e, "record");
  // The step waits for its upload and for the read-back that last used output b.
  if ((e = cudaStreamWaitEvent(s, io.up[b], 0)) != cudaSuccess) return cuda_fail(h, e, "wait");
  if (reused && (e = cudaStreamWaitEvent(s, io.back[b], 0)) != cudaSuccess) return cuda_fail(h, e, "wait");
  moeca_status st = moeca_step(h, io.in[b], io.out[b], &a, stream);
  if (st != MOECA_OK) return st;
  if ((e = cudaEventRecord(io.done[b], s)) != cudaSuccess) return cuda_fail(h, e, "record");
  // Read-back once the step has run.
  if ((e = cudaStreamWaitEvent(io.back_stream, io.done[b], 0)) != cudaSuccess) return cuda_fail(h, e, "wait");
  if ((e = cudaMemcpyAsync(x_out_host, io.out[b], xbytes, cudaMemcpyDeviceToHost, io.back_stream)) != cudaSuccess)
    return cuda_fail(h, e, "read back");
  if ((e = cudaEventRecord(io.back[b], io.back_stream)) != cudaSuccess) return cuda_fail(h, e, "record");
  ++io.calls;
  return MOECA_OK;
}

moeca_status moeca_host_join(moeca_handle* h, void* stream) {
  if (!h) return fail(nullptr, MOECA_ERR_INVALID_ARG, "handle is NULL");
  auto& io = h->hio;
  if (!io.ready || io.calls == 0) return MOECA_OK;
  cudaSetDevice(h->device);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // The read-back stream runs the read-backs in call order: its last event covers all of them.
  const int last = static_cast<int>((io.calls - 1) & 1);
  cudaError_t e = cudaStreamWaitEvent(s, io.back[last], 0);
  if (e == cudaSuccess) e = cudaStreamWaitEvent(s, io.up[last], 0);
  return e == cudaSuccess ? MOECA_OK : cuda_fail(h, e, "join");
}

namespace {

// Layer l's routing and block partials (the fused preparation kernel, MODE 1)
// on layer input `in`, into the exchange buffer.
cudaError_t shard_route(moeca_handle* h, int l, const void* in, cudaStream_t s) {
  LayerBuf& L = h->layers[l];
  const SelectArgs sa = select_args(h, L, h->sh.T, h->sh.refresh);
  PrepArgs pa = prep_args_plain(h, L, in, h->sh.T, h->sh.tau0, sa, nullptr);
  pa.shard_send = h->shard_send;
  return timed(h, MOECA_K_PREP, s, [&] { return launch_prep_shard(pa, h->prep, 1, s); });
}

// Layer l from the gathered partials on: decisions and compaction (MODE 2),
// grouped FFN, combine.
cudaError_t shard_finish(moeca_handle* h, int l, const void* in, void* out, cudaStream_t s) {
  LayerBuf& L = h->layers[l];
  const int T = h->sh.T;
  const SelectArgs sa = select_args(h, L, T, h->sh.refresh);
  PrepArgs pa = prep_args_plain(h, L, in, T, h->sh.tau0, sa, h->xg);
  pa.shard_recv = h->shard_recv;
  pa.shard_blocks = h->sh.world * (T / h->prep.tokens_per_block);
  pa.shard_tokens = h->sh.total;
  if (++h->prep_epoch == 0) h->prep_epoch = 1;
  pa.epoch = pa.wait_epoch = h->prep_epoch;
  cudaError_t e = timed(h, MOECA_K_PREP, s, [&] { return launch_prep_shard(pa, h->prep, 2, s); });
  if (e != cudaSuccess) return e;
  FfnArgs fa = ffn_args(h, L, T, in);
  if ((e = timed(h, MOECA_K_FFN, s, [&] { return launch_ffn_tc(L.tc, fa, 0, s); })) != cudaSuccess) return e;
  const CombineArgs cb = combine_args(h, L, T, in, out, h->sh.refresh, true);
  return timed(h, MOECA_K_COMBINE, s, [&] { return launch_combine(cb, h->bf16, s); });
}

}  // namespace

moeca_status moeca_shard_exchange_bytes(moeca_handle* h, int32_t n_tokens, int64_t* bytes_per_rank) {
  if (!h || !bytes_per_rank) return fail(h, MOECA_ERR_INVALID_ARG, "NULL argument");
  const int TB = h->prep.tokens_per_block;
  if (!TB) return fail(h, MOECA_ERR_UNSUPPORTED, "no fused preparation kernel on this handle");
  if (n_tokens < 1 || n_tokens > h->cfg.max_tokens || n_tokens % TB)
    return fail(h, MOECA_ERR_INVALID_ARG, "n_tokens must be in [1, max_tokens] and a multiple of the block size");
  *bytes_per_rank = static_cast<int64_t>(n_tokens / TB) * h->cfg.n_experts * 2 * static_cast<int64_t>(sizeof(float));
  return MOECA_OK;
}

moeca_status moeca_shard_begin(moeca_handle* h, const void* x_in, void* x_out, const moeca_step_args* args,
                               const moeca_shard* shard, void* send, const void* recv, void* stream) {
  if (!h) return fail(nullptr, MOECA_ERR_INVALID_ARG, "handle is NULL");
  if (!args || !shard) return fail(h, MOECA_ERR_INVALID_ARG, "args or shard is NULL");
  const moeca_config& c = h->cfg;
  const int TB = h->prep.tokens_per_block;
  if (!TB || c.n_heads || !h->bf16 || c.ffn_impl != MOECA_FFN_AUTO || c.token_reuse_policy)
    return fail(h, MOECA_ERR_UNSUPPORTED,
                "token-sharded steps run the bf16 MoE layer stack on the fused preparation kernel "
                "(n_heads 0, tensor-core FFN, token_reuse_policy 0, a shape the fused kernel fits)");
  if (h->sh.active) return fail(h, MOECA_ERR_STATE, "a sharded step is in progress: call moeca_shard_next");
  const int T = args->n_tokens;
  if (T < 1 || T > c.max_tokens || T % TB)
    return fail(h, MOECA_ERR_INVALID_ARG, "n_tokens must be in [1, max_tokens] and a multiple of the block size");
  if (shard->world < 1 || shard->rank < 0 || shard->rank >= shard->world ||
      static_cast<long long>(shard->total_tokens) != static_cast<long long>(shard->world) * T)
    return fail(h, MOECA_ERR_INVALID_ARG, "0 <= rank < world and total_tokens = world x n_tokens");
  if (!send || !recv || reinterpret_cast<uintptr_t>(send) % 16 || reinterpret_cast<uintptr_t>(recv) % 16)
    return fail(h, MOECA_ERR_INVALID_ARG, "send and recv must be 16-byte aligned device buffers");
  moeca_status st = check_device_status(h);
  if (st != MOECA_OK) return st;
  if (!x_in || !x_out) return fail(h, MOECA_ERR_INVALID_ARG, "x_in or x_out is NULL");
  const size_t xbytes = static_cast<size_t>(T) * c.hidden * h->es;
  if (overlaps(x_in, x_out, xbytes)) return fail(h, MOECA_ERR_INVALID_ARG, "x_in and x_out overlap");
  if (reinterpret_cast<uintptr_t>(x_in) % 16 || reinterpret_cast<uintptr_t>(x_out) % 16)
    return fail(h, MOECA_ERR_INVALID_ARG, "x_in and x_out must be 16-byte aligned");
  cudaSetDevice(h->device);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  bool all_valid = h->state_T == T;
  for (auto& L : h->layers) all_valid = all_valid && L.valid;
  const int N = c.refresh_period;
  const bool refresh = args->force_refresh || !all_valid || (N > 0 && args->step_index % N == 0);
  if (h->state_T != T) {
    for (auto& L : h->layers) {
      cudaError_t e = cudaMemsetAsync(L.ema, 0, static_cast<size_t>(c.max_tokens) * c.n_experts * 4, s);
      if (e != cudaSuccess) return cuda_fail(h, e, "reset EMA");
      L.valid = false;
    }
  }
  h->shard_send = static_cast<float*>(send);
  h->shard_recv = static_cast<float*>(const_cast<void*>(recv));
  h->sh.layer = 0;
  h->sh.T = T;
  h->sh.world = shard->world;
  h->sh.total = shard->total_tokens;
  h->sh.refresh = refresh;
  h->sh.tau0 = std::isnan(args->tau0_override) ? c.tau0 : args->tau0_override;
  h->sh.x_in = x_in;
  h->sh.x_out = x_out;
  cudaError_t e = shard_route(h, 0, x_in, s);
  if (e != cudaSuccess) {
    for (auto& L : h->layers) L.valid = false;
    return cuda_fail(h, e, "kernel launch");
  }
  h->sh.active = true;
  return MOECA_OK;
}

moeca_status moeca_shard_next(moeca_handle* h, void* stream, int32_t* done) {
  if (!h || !done) return fail(h, MOECA_ERR_INVALID_ARG, "NULL argument");
  if (!h->sh.active) return fail(h, MOECA_ERR_STATE, "no sharded step in progress");
  cudaSetDevice(h->device);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int l = h->sh.layer, nL = h->cfg.n_layers;
  const void* in = l == 0 ? h->sh.x_in : h->act[l];
  void* out = l + 1 == nL ? h->sh.x_out : h->act[l + 1];
  NvtxRange range("moeca_shard_next");
  cudaError_t e = shard_finish(h, l, in, out, s);
  if (e == cudaSuccess) {
    h->layers[l].valid = true;
    if (l + 1 < nL) e = shard_route(h, l + 1, out, s);
  }
  if (e != cudaSuccess) {
    for (auto& L : h->layers) L.valid = false;
    h->sh.active = false;
    return cuda_fail(h, e, "kernel launch");
  }
  if (l + 1 < nL) {
    h->sh.layer = l + 1;
    *done = 0;
  } else {
    h->state_T = h->sh.T;
    h->last_x_in = h->sh.x_in;
    h->sh.active = false;
    *done = 1;
  }
  return MOECA_OK;
}

moeca_status moeca_get_stats(moeca_handle* h, int32_t layer, moeca_stats* out) {
  if (!h || !out) return fail(h, MOECA_ERR_INVALID_ARG, "NULL argument");
  const int L = h->cfg.n_layers;
  if (layer < -1 || layer >= L) return fail(h, MOECA_ERR_INVALID_ARG, "layer out of range");
  cudaSetDevice(h->device);
  cudaError_t e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return cuda_fail(h, e, "synchronize");
  std::memset(out, 0, sizeof *out);
  for (int l = 0; l < L; ++l) {
    if (layer >= 0 && l != layer) continue;
    unsigned long long v[kStCount];
    if ((e = cudaMemcpy(v, h->layers[l].stats, sizeof v, cudaMemcpyDeviceToHost)) != cudaSuccess)
      return cuda_fail(h, e, "read stats");
    out->layer_steps += v[kStLayerSteps];
    out->refresh_layer_steps += v[kStRefreshSteps];
    out->branches += v[kStBranches];
    out->cache_step_branches += v[kStCacheBranches];
    out->matched += v[kStMatched];
    out->recomputed += v[kStRecomputed];
    out->reused += v[kStReused];
    out->tokens_fully_reused += v[kStTokensFullyReused];
    out->shared_recomputed += v[kStSharedRecomputed];
    out->near_margin_route += v[kStNearRoute];
    out->near_margin_score += v[kStNearScore];
    out->attn_recomputed += v[kStAttnRows];
  }
  volatile int* st = h->status_host;
  out->device_status = st[0];
  out->device_detail = st[1];
  return out->device_status ? check_device_status(h) : MOECA_OK;
}

moeca_status moeca_reset_stats(moeca_handle* h) {
  if (!h) return fail(nullptr, MOECA_ERR_INVALID_ARG, "handle is NULL");
  cudaSetDevice(h->device);
  for (auto& L : h->layers) {
    cudaError_t e = cudaMemset(L.stats, 0, kStCount * 8);
    if (e != cudaSuccess) return cuda_fail(h, e, "reset stats");
  }
  return MOECA_OK;
}

moeca_status moeca_get_layer_state(moeca_handle* h, int32_t layer, const moeca_layer_state* dst,
                                   int32_t* n_tokens, void* stream) {
  if (!h || !dst) return fail(h, MOECA_ERR_INVALID_ARG, "NULL argument");
  if (layer < 0 || layer >= h->cfg.n_layers) return fail(h, MOECA_ERR_INVALID_ARG, "layer out of range");
  const LayerBuf& L = h->layers[layer];
  const size_t T = L.valid ? h->state_T : 0, k = h->cfg.top_k, D = h->cfg.hidden, E = h->cfg.n_experts;
  if (n_tokens) *n_tokens = static_cast<int32_t>(T);
  if (T == 0) return MOECA_OK;
  cudaSetDevice(h->device);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  struct { void* d; const void* s; size_t n; } cp[] = {
      {dst->cache_e, L.cache_e, T * k * 4},      {dst->cache_w, L.cache_w, T * k * 4},
      {dst->cache_norm, L.cache_norm, T * k * 4}, {dst->cache_h, L.cache_h, T * k * D * h->es},
      {dst->shared_h, L.shared_h, T * D * h->es}, {dst->ema, L.ema, T * E * 4},
      {dst->attn_a, L.attn_a, T * D * h->es},     {dst->cache_y, L.cache_y, T * D * 4}};
  for (auto& x : cp) {
    if (!x.d || !x.s) continue;
    cudaError_t e = cudaMemcpyAsync(x.d, x.s, x.n, cudaMemcpyDeviceToDevice, s);
    if (e != cudaSuccess) return cuda_fail(h, e, "copy layer state");
  }
  return MOECA_OK;
}

moeca_status moeca_set_layer_state(moeca_handle* h, int32_t layer, const moeca_layer_state* src,
                                   int32_t n_tokens, void* stream) {
  if (!h || !src) return fail(h, MOECA_ERR_INVALID_ARG, "NULL argument");
  if (layer < 0 || layer >= h->cfg.n_layers) return fail(h, MOECA_ERR_INVALID_ARG, "layer out of range");
  if (n_tokens < 1 || n_tokens > h->cfg.max_tokens) return fail(h, MOECA_ERR_INVALID_ARG, "n_tokens out of range");
  if (!src->cache_e || !src->cache_w || !src->cache_norm || !src->cache_h || !src->ema ||
      (h->cfg.n_shared && !src->shared_h) || (h->cfg.n_heads && !src->attn_a) ||
      (h->cfg.token_reuse_policy && !src->cache_y))
    return fail(h, MOECA_ERR_INVALID_ARG, "every state buffer is required");
  LayerBuf& L = h->layers[layer];
  const size_t T = n_tokens, k = h->cfg.top_k, D = h->cfg.hidden, E = h->cfg.n_experts;
  cudaSetDevice(h->device);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  struct { void* d; const void* s; size_t n; } cp[] = {
      {L.cache_e, src->cache_e, T * k * 4},      {L.cache_w, src->cache_w, T * k * 4},
      {L.cache_norm, src->cache_norm, T * k * 4}, {L.cache_h, src->cache_h, T * k * D * h->es},
      {L.shared_h, src->shared_h, T * D * h->es}, {L.ema, src->ema, T * E * 4},
      {L.attn_a, src->attn_a, T * D * h->es},     {L.cache_y, src->cache_y, T * D * 4}};
  for (auto& x : cp) {
    if (!x.d || !x.s) continue;
    cudaError_t e = cudaMemcpyAsync(x.d, x.s, x.n, cudaMemcpyDeviceToDevice, s);
    if (e != cudaSuccess) return cuda_fail(h, e, "load layer state");
  }
  if (h->state_T != n_tokens) {
    for (auto& other : h->layers) other.valid = false;
    h->state_T = n_tokens;
  }
  L.valid = true;
  return MOECA_OK;
}

moeca_status moeca_get_layer_trace(moeca_handle* h, int32_t layer, const moeca_layer_trace* dst,
                                   void* stream) {
  if (!h || !dst) return fail(h, MOECA_ERR_INVALID_ARG, "NULL argument");
  if (layer < 0 || layer >= h->cfg.n_layers) return fail(h, MOECA_ERR_INVALID_ARG, "layer out of range");
  const LayerBuf& L = h->layers[layer];
  const size_t T = h->state_T, k = h->cfg.top_k, D = h->cfg.hidden, E = h->cfg.n_experts, G = h->G;
  if (T == 0) return fail(h, MOECA_ERR_STATE, "no step has run");
  cudaSetDevice(h->device);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const void* in = layer == 0 ? h->last_x_in : h->act[layer];
  const void* moe_in = h->cfg.adaln ? L.attn_m : (h->cfg.n_heads ? L.attn_u : in);
  const size_t mod_n = static_cast<size_t>(h->mod_b) * 6 * D;
  struct { void* d; const void* s; size_t n; } cp[] = {
      {dst->route_e, L.route_e, T * k * 4}, {dst->route_w, L.route_w, T * k * 4},
      {dst->tau, L.tau, E * 4},             {dst->recompute, L.recompute, T * k},
      {dst->slot, L.slot, T * k},           {dst->matched, L.matched, T * k},
      {dst->token_any, L.token_any, T},     {dst->counts, L.counts, G * 4},
      {dst->offsets, L.offsets, (G + 1) * 4},
      {dst->list, L.list, T * (k + h->cfg.n_shared) * 4},
      {dst->layer_in, moe_in, T * D * h->es},
      {dst->block_in, h->cfg.n_heads ? in : nullptr, T * D * h->es},
      {dst->route_in, L.route_m, T * D * h->es},
      {dst->resid, h->cfg.n_heads ? L.attn_u : in, T * D * h->es},
      {dst->mod, h->mod ? h->mod + static_cast<size_t>(layer) * mod_n : nullptr, mod_n * 4}};
  for (auto& x : cp) {
    if (!x.d || !x.s) continue;
    cudaError_t e = cudaMemcpyAsync(x.d, x.s, x.n, cudaMemcpyDeviceToDevice, s);
    if (e != cudaSuccess) return cuda_fail(h, e, "copy layer trace");
  }
  return MOECA_OK;
}

moeca_status moeca_reset(moeca_handle* h) {
  if (!h) return fail(nullptr, MOECA_ERR_INVALID_ARG, "handle is NULL");
  cudaSetDevice(h->device);
  {
    // Let every kernel of earlier steps finish before the counters and the
    // device status are cleared.
    cudaError_t e = cudaDeviceSynchronize();
    if (e != cudaSuccess) return cuda_fail(h, e, "synchronise before reset");
    h->status_host[0] = 0;
    h->status_host[1] = 0;
  }
  if (h->prep_words) {
    cudaError_t e = cudaMemset(h->prep_words, 0, h->prep_words_n * 8);
    if (e != cudaSuccess) return cuda_fail(h, e, "reset exchange words");
    h->prep_epoch = 0;
  }
  // Counters that kernels leave at zero, unless a launch was cut short.
  if (h->tc_dep) {
    cudaError_t e = cudaMemset(h->tc_dep, 0, static_cast<size_t>(h->tc_dep_pairs_n) * 2 * sizeof(int));
    if (e == cudaSuccess) e = cudaMemset(h->tc_sem, 0, tc_split_units(h->n_sms) * sizeof(int));
    if (e == cudaSuccess) e = cudaMemset(h->tc_work, 0, 2 * sizeof(int));
    if (e != cudaSuccess) return cuda_fail(h, e, "reset GEMM counters");
  }
  for (auto& L : h->layers) {
    L.valid = false;
    cudaError_t e = cudaMemset(L.ema, 0, static_cast<size_t>(h->cfg.max_tokens) * h->cfg.n_experts * 4);
    if (e != cudaSuccess) return cuda_fail(h, e, "reset EMA");
  }
  h->state_T = 0;
  h->sh.active = false;
  return MOECA_OK;
}

moeca_status moeca_inject_fault(moeca_handle* h, int32_t kind) {
  if (!h) return fail(nullptr, MOECA_ERR_INVALID_ARG, "handle is NULL");
  if (kind != MOECA_FAULT_BARRIER_STALL) return fail(h, MOECA_ERR_INVALID_ARG, "unknown fault kind");
  if (h->prep.tokens_per_block == 0) return fail(h, MOECA_ERR_UNSUPPORTED, "no fused preparation kernel on this handle");
  h->inject_stall = true;
  return MOECA_OK;
}

moeca_status moeca_set_kernel_timing(moeca_handle* h, int32_t enable) {
  if (!h) return fail(nullptr, MOECA_ERR_INVALID_ARG, "handle is NULL");
  h->timing = enable != 0;
  return MOECA_OK;
}

moeca_status moeca_get_kernel_times(moeca_handle* h, moeca_kernel_times* out, int32_t reset) {
  if (!h || !out) return fail(h, MOECA_ERR_INVALID_ARG, "NULL argument");
  cudaSetDevice(h->device);
  for (auto& pt : h->pending) {
    cudaError_t e = cudaEventSynchronize(pt.stop);
    if (e != cudaSuccess) return cuda_fail(h, e, "event synchronize");
    float ms = 0.f;
    cudaEventElapsedTime(&ms, pt.start, pt.stop);
    h->total_ms[pt.kind] += ms;
    h->launches[pt.kind] += 1;
    h->event_pool.push_back(pt.start);
    h->event_pool.push_back(pt.stop);
  }
  h->pending.clear();
  for (int i = 0; i < MOECA_K_COUNT; ++i) {
    out->total_ms[i] = h->total_ms[i];
    out->launches[i] = h->launches[i];
    if (reset) {
      h->total_ms[i] = 0.0;
      h->launches[i] = 0;
    }
  }
  return MOECA_OK;
}

moeca_status moeca_ddpm_schedule(int32_t n_steps, int32_t n_train, double beta_start, double beta_end,
                                 int32_t* t, double* alpha, double* alpha_bar, double* beta) {
  if (n_steps < 2 || n_steps > n_train || !(beta_start > 0.0 && beta_start <= beta_end && beta_end < 1.0))
    return fail(nullptr, MOECA_ERR_INVALID_ARG, "2 <= n_steps <= n_train and 0 < beta_start <= beta_end < 1");
  // Training schedule: linear betas, abar the running product of 1 - beta.
  std::vector<double> abar(n_train);
  double prod = 1.0;
  for (int s = 0; s < n_train; ++s) {
    const double b = n_train == 1 ? beta_start : beta_start + (beta_end - beta_start) * s / (n_train - 1);
    prod *= 1.0 - b;
    abar[s] = prod;
  }
  double prev = 1.0;
  for (int j = 0; j < n_steps; ++j) {
    const int ts = static_cast<int>(std::floor(static_cast<double>(j) * (n_train - 1) / (n_steps - 1) + 0.5));
    const double ab = abar[ts];
    const double al = ab / prev;
    if (t) t[j] = ts;
    if (alpha) alpha[j] = al;
    if (alpha_bar) alpha_bar[j] = ab;
    if (beta) beta[j] = 1.0 - al;
    prev = ab;
  }
  return MOECA_OK;
}

moeca_status moeca_ddpm_step(const moeca_ddpm_args* a, void* stream) {
  if (!a || !a->x_t || !a->eps || !a->x_prev) return fail(nullptr, MOECA_ERR_INVALID_ARG, "NULL argument");
  if (a->n < 0 || a->n % 8) return fail(nullptr, MOECA_ERR_INVALID_ARG, "n must be a non-negative multiple of 8");
  if (a->eps_dtype != MOECA_F32 && a->eps_dtype != MOECA_BF16) return fail(nullptr, MOECA_ERR_INVALID_ARG, "eps_dtype");
  if (!(a->alpha > 0.0 && a->alpha <= 1.0) || !(a->alpha_bar >= 0.0 && a->alpha_bar < 1.0) || !(a->sigma >= 0.0))
    return fail(nullptr, MOECA_ERR_INVALID_ARG, "0 < alpha <= 1, 0 <= alpha_bar < 1, sigma >= 0");
  if (a->sigma > 0.0 && !a->z) return fail(nullptr, MOECA_ERR_INVALID_ARG, "z is NULL with sigma > 0");
  const void* ps[] = {a->x_t, a->eps, a->z, a->x_prev, a->x_next};
  for (const void* p : ps)
    if (reinterpret_cast<uintptr_t>(p) % 16) return fail(nullptr, MOECA_ERR_INVALID_ARG, "pointers must be 16-byte aligned");
  DdpmArgs d{};
  d.n = a->n;
  d.bf16 = a->eps_dtype == MOECA_BF16;
  d.c1 = static_cast<float>((1.0 - a->alpha) / std::sqrt(1.0 - a->alpha_bar));
  d.inv_sqrt_alpha = static_cast<float>(1.0 / std::sqrt(a->alpha));
  d.sigma = static_cast<float>(a->sigma);
  d.x_t = a->x_t; d.eps = a->eps; d.z = a->sigma > 0.0 ? a->z : nullptr;
  d.x_prev = a->x_prev; d.x_next = a->x_next;
  cudaError_t e = launch_ddpm(d, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return fail(nullptr, MOECA_ERR_CUDA, std::string("ddpm step: ") + cudaGetErrorString(e));
  return MOECA_OK;
}

moeca_status moeca_destroy(moeca_handle* h) {
  if (!h) return MOECA_OK;
  cudaSetDevice(h->device);
  cudaDeviceSynchronize();
  free_all(h);
  delete h;
  return MOECA_OK;
}

}  // extern "C"
