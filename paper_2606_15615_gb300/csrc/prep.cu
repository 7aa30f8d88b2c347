// Fused per-layer preparation of the branch-cached MoE layer, one launch
// (programmatic dependent launch, every block co-resident) with two
// grid-wide exchanges:
//
//   A  router (Eq. 7): gate logits on the tensor cores (mma.sync m16n8k16,
//      bf16 in, fp32 accumulate; the warps of a 16-token group split D) from
//      the block's token rows and the gate matrix staged in shared memory by
//      bulk async copies; fp32 softmax and top-k with ties to the lower
//      expert id; the EMA statistic (Eq. 10) and the block's entropy partial
//      sums, published; then the threshold-free half of each token's
//      decision (matching, slots, scores; Sec. 4.2, Eq. 9).
//   -- exchange 1: every block reads all blocks' partials --
//   B  every block reduces the partials in block order to the same
//      thresholds tau_e (Eq. 11-12), finishes its tokens' decisions and
//      publishes its recomputed rows per expert group.
//   -- exchange 2: every block reads all blocks' row counts --
//   C  every block forms the group offsets and its own prefix, writes its
//      rows into the per-group lists (ascending token order) and gathers
//      their inputs for the grouped FFN.
//
// An exchange is data-carrying: each published value is a 64-bit word whose
// high half is the launch's epoch (a number the host never reuses before a
// reset), stored and loaded with relaxed GPU-scope accesses (each word is
// single-copy atomic).  A reader polls the words it needs until every one
// carries the epoch, so a value and its readiness arrive in the same load:
// no fence, no arrival counter, one round trip.  The poll is bounded by one
// second of %globaltimer; on timeout it records MOECA's timeout status and
// the block skips its later phases.
//
// The results are those of router_kernel + select_kernel + compact_kernel,
// which remain the path for fp32, for shapes whose staging does not fit in
// shared memory, and for grids that cannot be co-resident.
#include "common.cuh"
#include "kernels.h"
#include "select_token.cuh"

// This file is compiled twice: plain (the MoE layer alone) and, from
// prep_attn.cu with MOECA_PREP_ATTN 1, for DiT-MoE blocks.  The block's work
// (u = x + a^{t0}, the FFN-row map, the recomputing-token list) exists only
// in the second build, so the MoE path's code -- phases run once per launch
// and on the critical path -- carries none of it.
#ifndef MOECA_PREP_ATTN
#define MOECA_PREP_ATTN 0
#endif
#ifndef MOECA_PREP_SHARD
#define MOECA_PREP_SHARD 0
#endif

namespace moeca {
namespace {
constexpr bool kAttn = MOECA_PREP_ATTN != 0;

constexpr int kThreads = 128;
constexpr int kMaxGroups = kMaxExperts + 1;
constexpr unsigned long long kBarrierNs = 1000000000ull;

template <int G>
__device__ __forceinline__ float grp_max(float v) {
#pragma unroll
  for (int o = G / 2; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
template <int G>
__device__ __forceinline__ float grp_sum(float v) {
#pragma unroll
  for (int o = G / 2; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Tagged words of the grid-wide exchanges: payload in the low 32 bits, the
// launch's epoch in the high 32.
__device__ __forceinline__ unsigned long long tag_word(uint32_t payload, unsigned epoch) {
  return (static_cast<unsigned long long>(epoch) << 32) | payload;
}
__device__ __forceinline__ void st_word(unsigned long long* p, unsigned long long v) {
  asm volatile("st.relaxed.gpu.global.b64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}
__device__ __forceinline__ unsigned long long ld_word(const unsigned long long* p) {
  unsigned long long v;
  asm volatile("ld.relaxed.gpu.global.b64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}

// Read n tagged words p[idx(0)] .. p[idx(n - 1)] and hand their payloads to
// f(j, payload) in order j = 0..n-1.  Words are fetched kB at a time; while
// any word of a batch still carries another epoch, the batch's stale words
// are fetched again (one round trip per retry).  Returns false once
// `deadline` (%globaltimer) has passed.
template <int kB, typename Idx, typename F>
__device__ __forceinline__ bool read_tagged(const unsigned long long* p, int n, Idx idx, unsigned epoch,
                                            unsigned long long deadline, F&& f) {
  for (int j0 = 0; j0 < n; j0 += kB) {
    unsigned long long v[kB];
#pragma unroll
    for (int u = 0; u < kB; ++u) v[u] = 0ull;  // epoch 0 is never used: every word starts stale
    for (;;) {
#pragma unroll
      for (int u = 0; u < kB; ++u)
        if (j0 + u < n && static_cast<unsigned>(v[u] >> 32) != epoch) v[u] = ld_word(p + idx(j0 + u));
      bool all = true;
#pragma unroll
      for (int u = 0; u < kB; ++u) all &= j0 + u >= n || static_cast<unsigned>(v[u] >> 32) == epoch;
      if (all) break;
      if (globaltimer() > deadline) return false;
    }
#pragma unroll
    for (int u = 0; u < kB; ++u)
      if (j0 + u < n) f(j0 + u, static_cast<uint32_t>(v[u]));
  }
  return true;
}

// TB tokens per block (16 or 32); EPAD experts padded to a multiple of 8.
// Bytes of the region holding the partial logits of phase A, one
// [TB][EPAD + 1] table per warp of a 16-token group (each sums its own range
// of D), rounded up to 16.
__host__ __device__ constexpr int prep_wpg(int TB) { return 4 / (TB / 16); }
__host__ __device__ constexpr size_t prep_region_bytes(int TB, int EPAD) {
  return (static_cast<size_t>(prep_wpg(TB)) * TB * (EPAD + 1) * 4 + 15) / 16 * 16;
}

// DiT-MoE block work kept out of line, so the MoE-only path's code (phases
// run once per launch, on the critical path) is what it is without it.
// Bulk copies of the block's cached attention rows a^{t0} (thread 0).
static __device__ __noinline__ void issue_attn_rows(const PrepArgs& a, __nv_bfloat16* s_a, int ldw, int tok0,
                                                    int ntok, uint32_t row_bytes, uint32_t bar) {
  const __nv_bfloat16* ar = static_cast<const __nv_bfloat16*>(a.attn_a);
  for (int q = 0; q < ntok; ++q)
    bulk_g2s(smem_u32(s_a + q * ldw), ar + static_cast<size_t>(tok0 + q) * a.D, row_bytes, bar);
}

// u = x + a^{t0} (rounded to bf16) in place of the staged x rows, and to u_out.
static __device__ __noinline__ void form_u(const PrepArgs& a, __nv_bfloat16* s_x, const __nv_bfloat16* s_a, int ldw,
                                           int tok0, int ntok, int t) {
  __nv_bfloat16* u_out = static_cast<__nv_bfloat16*>(a.u_out);
  const int nv = a.D / 8;
  for (int idx = t; idx < ntok * nv; idx += kThreads) {
    const int q = idx / nv, c = idx % nv;
    uint4* xs = reinterpret_cast<uint4*>(s_x + q * ldw) + c;
    float xv[8], av[8];
    unpack_vec(*xs, xv, static_cast<__nv_bfloat16*>(nullptr));
    unpack_vec(*(reinterpret_cast<const uint4*>(s_a + q * ldw) + c), av, static_cast<__nv_bfloat16*>(nullptr));
#pragma unroll
    for (int j = 0; j < 8; ++j) xv[j] += av[j];
    uint4 uv;
    __nv_bfloat162* uh = reinterpret_cast<__nv_bfloat162*>(&uv);
#pragma unroll
    for (int j = 0; j < 4; ++j) uh[j] = __floats2bfloat162_rn(xv[2 * j], xv[2 * j + 1]);
    *xs = uv;
    reinterpret_cast<uint4*>(u_out + static_cast<size_t>(tok0 + q) * a.D)[c] = uv;
  }
}

// One lane's token (warp 0 of phase C): its FFN-row map entries (the list
// positions of its recomputed branches, -1 elsewhere) and its place in the
// recomputing-token list.  `pos[p]` are the positions the list loop wrote.
static __device__ __noinline__ void attn_bookkeeping(const PrepArgs& a, int i, int lane, int ntok, bool any,
                                                     const int* pos, int shared_pos, int list_pos) {
  if (lane >= ntok) return;  // 16-token blocks: lanes 16-31 hold the next block's tokens
  if (a.row_of) {
    const int W = a.sel.k + a.n_shared;
    int32_t* row_of = a.row_of + static_cast<size_t>(i) * W;
    for (int p = 0; p < a.sel.k; ++p) row_of[p] = pos[p];
    if (a.n_shared) row_of[a.sel.k] = shared_pos;
  }
  if (a.attn_list) {
    if (any) a.attn_rows[list_pos] = i;
    a.attn_inv[i] = any ? list_pos : -1;
    if (i % a.seq == 0) a.sample_lo[i / a.seq] = list_pos;
  }
}

// MODE 0: the whole preparation of a layer (the default).  A token-sharded
// stack (each rank holds a block-aligned slice of the batch) runs it in two
// launches around an all-gather of the entropy partials, Eq. 11's per-expert
// sums being the only coupling between tokens: MODE 1 routes its blocks'
// tokens and writes the block partials (plain floats) for the exchange;
// MODE 2 reads every rank's partials, in the global block order MODE 0 uses,
// and decides and compacts.
template <int TB, int EPAD, int KMAX, int MODE>
__global__ void __launch_bounds__(kThreads) prep_kernel(PrepArgs a) {
  constexpr int G = kThreads / TB;       // lanes per token in the routing epilogue (4 or 8)
  constexpr int EPL = EPAD / G;          // experts per lane (>= 1)
  constexpr int NTILE = EPAD / 8;        // mma n-tiles
  constexpr int TOKG = TB / 16;          // 16-token mma groups
  constexpr int WPG = 4 / TOKG;          // warps per token group
  static_assert(EPL >= 1 && EPL * G == EPAD, "experts per lane");
  extern __shared__ __align__(128) uint8_t dyn[];
  __shared__ float sm_S[TB * EPAD];
  __shared__ float sm_U[TB * EPAD];
  __shared__ float sm_rs[kThreads][2];
  __shared__ float sm_tau[kMaxExperts];
  __shared__ float sm_H[kMaxExperts];
  __shared__ int sm_live[kMaxExperts];
  __shared__ float sm_lo, sm_hi;
  __shared__ int sm_near;
  // Groups: E routed, the shared expert, and (DiT-MoE block) the list of
  // tokens that recompute their attention.
  __shared__ unsigned sm_bal[kMaxGroups + 1];
  __shared__ int sm_pre[kMaxGroups + 1];
  __shared__ int sm_tot[kMaxGroups + 1];
  __shared__ int sm_off[kMaxGroups + 2];
  __shared__ int sm_rows[TB * (KMAX + 1)][2];
  __shared__ bool sm_any[kAttn ? TB : 1];
  __shared__ int sm_nrows;
  __shared__ int sm_fail;
  __shared__ __align__(8) uint64_t sm_bar;
  // Per-token inputs of the decision, fetched at the start and kept here.
  __shared__ int32_t sm_re[TB * KMAX];
  __shared__ float sm_rw[TB * KMAX];
  __shared__ int32_t sm_ce[TB * KMAX];
  __shared__ float sm_cw[TB * KMAX];
  __shared__ float sm_cn[TB * KMAX];
  __shared__ float sm_ema[TB * EPAD];

  const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
  const int E = a.E, k = a.k, D = a.D, T = a.T;
  const int ldw = D + 8;  // padded row, in bf16
  __nv_bfloat16* s_w = reinterpret_cast<__nv_bfloat16*>(dyn);
  __nv_bfloat16* s_x = s_w + EPAD * ldw;
  float* s_logit = reinterpret_cast<float*>(s_x + TB * ldw);  // [WPG][TB][EPAD + 1]
  const int tok0 = blockIdx.x * TB;
  const int ntok = min(TB, T - tok0);
  // DiT-MoE block on a cache step: the cached attention rows, after the
  // logits region.
  const bool add_a = kAttn && a.attn_a != nullptr;
  __nv_bfloat16* s_a = reinterpret_cast<__nv_bfloat16*>(reinterpret_cast<uint8_t*>(s_logit) +
                                                        prep_region_bytes(TB, EPAD));

  // ---- A0: stage gate rows and token rows ----
  // Before the programmatic-dependency wait: everything that the previous
  // kernel (the layer below's combine) does not write.  The gate matrix is a
  // weight; the cached metadata and the EMA rows were last written by this
  // layer's own kernels one step earlier, which completed before the
  // previous kernel could start.
  if (t == 0) {
    sm_near = 0;
    sm_nrows = 0;
    sm_fail = 0;
    mbar_init(smem_u32(&sm_bar), 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  const uint32_t bar = smem_u32(&sm_bar);
  const uint32_t row_bytes = static_cast<uint32_t>(D) * 2;
  constexpr bool kRoute = MODE != 2;  // MODE 2 reads the routing MODE 1 wrote
  // The copies are issued by the lanes of warp 0 (one row each), after lane
  // 0's expect-tx, which carries the barrier's only arrival.
  if (t == 0) mbar_expect_tx(bar, row_bytes * ((kRoute ? E : 0) + ntok + (add_a ? ntok : 0)));
  if (warp == 0) {
    __syncwarp();
    const __nv_bfloat16* wg = static_cast<const __nv_bfloat16*>(a.w_gate);
    if (kRoute)
      for (int e = lane; e < E; e += 32) bulk_g2s(smem_u32(s_w + e * ldw), wg + static_cast<size_t>(e) * D, row_bytes, bar);
    if constexpr (kAttn) {
      if (add_a && lane == 0) issue_attn_rows(a, s_a, ldw, tok0, ntok, row_bytes, bar);  // written on an earlier step
    }
  }
  // Prefetch what later phases read: cached metadata and EMA rows.
  {
    const size_t cb = static_cast<size_t>(tok0) * k;
    if (!a.sel.refresh)
      for (int idx = t; idx < ntok * k; idx += kThreads) {
        sm_ce[idx] = a.sel.cache_e[cb + idx];
        sm_cw[idx] = a.sel.cache_w[cb + idx];
        sm_cn[idx] = a.sel.cache_norm[cb + idx];
      }
    const size_t eb = static_cast<size_t>(tok0) * E;
    if (kRoute)
      for (int idx = t; idx < ntok * E; idx += kThreads) sm_ema[(idx / E) * EPAD + idx % E] = a.ema[eb + idx];
  }
  // Zero the padding rows the tensor cores read (experts past E, tokens past T).
  for (int idx = t; kRoute && idx < (EPAD - E) * (D / 8); idx += kThreads) {
    const int r = E + idx / (D / 8), c = idx % (D / 8);
    reinterpret_cast<uint4*>(s_w + r * ldw)[c] = make_uint4(0, 0, 0, 0);
  }
  for (int idx = t; idx < (TB - ntok) * (D / 8); idx += kThreads) {
    const int r = ntok + idx / (D / 8), c = idx % (D / 8);
    reinterpret_cast<uint4*>(s_x + r * ldw)[c] = make_uint4(0, 0, 0, 0);
  }
  pdl_entry();
  if (warp == 0) {
    const __nv_bfloat16* x = static_cast<const __nv_bfloat16*>(a.x);
    for (int q = lane; q < ntok; q += 32)
      bulk_g2s(smem_u32(s_x + q * ldw), x + static_cast<size_t>(tok0 + q) * D, row_bytes, bar);
  }
  if (!mbar_wait_for(bar, 0, kBarrierNs) && t == 0) report_status(a.status, kStatusWaitTimeout, 610);
  __syncthreads();
  // The grouped GEMM after this kernel reads the routed W1 first, expert by
  // expert.  HBM is nearly idle while the routing, the exchanges and the
  // decisions run, so the blocks bring its head into L2 now (a hint, issued
  // once the block's own rows have landed so as not to delay them).
  if (warp == 0 && a.l2_pf_bytes) l2_prefetch_share(a.l2_pf, a.l2_pf_bytes, blockIdx.x, gridDim.x, lane);
  if constexpr (kAttn) {
    if (add_a) {
      // u = x + a^{t0}: the router input, the rows the FFN gathers, and the
      // residual; written out for the kernels after this one.
      form_u(a, s_x, s_a, ldw, tok0, ntok, t);
      __syncthreads();
    }
  }

  if constexpr (!kRoute) {
    // The routing of the block's tokens, written by MODE 1.
    for (int idx = t; idx < ntok * k; idx += kThreads) {
      sm_re[idx] = a.route_e[static_cast<size_t>(tok0) * k + idx];
      sm_rw[idx] = a.route_w[static_cast<size_t>(tok0) * k + idx];
    }
    __syncthreads();
  } else {
  // ---- A1: logits on the tensor cores ----
  // The WPG warps of a 16-token group each take a contiguous range of the
  // D / 16 k-steps and every n-tile over it, with two interleaved
  // accumulator chains and the next step's fragments loaded ahead; each
  // warp's partial logits go to its own table, added in range order below.
  {
    const int tg = warp / WPG, h = warp % WPG;
    const int KS = D / 16;
    const int ks0 = h * KS / WPG, ks1 = (h + 1) * KS / WPG;
    float acc[2][NTILE][4];
#pragma unroll
    for (int c = 0; c < 2; ++c)
#pragma unroll
      for (int j = 0; j < NTILE; ++j) acc[c][j][0] = acc[c][j][1] = acc[c][j][2] = acc[c][j][3] = 0.f;
    if (tg < TOKG) {
      const uint32_t a_addr = smem_u32(s_x + (tg * 16 + (lane & 15)) * ldw + (lane >> 4) * 8);
      const int bl = lane & 15;
      uint32_t b_addr[NTILE];
#pragma unroll
      for (int j = 0; j < NTILE; ++j) b_addr[j] = smem_u32(s_w + (j * 8 + (bl & 7)) * ldw + (bl >> 3) * 8);
      uint32_t A[4], B[NTILE][2];
      auto load = [&](int ks, uint32_t* Ar, uint32_t (*Br)[2]) {
        ldsm_x4(a_addr + ks * 32, Ar[0], Ar[1], Ar[2], Ar[3]);
#pragma unroll
        for (int j = 0; j < NTILE; ++j) ldsm_x2(b_addr[j] + ks * 32, Br[j][0], Br[j][1]);
      };
      if (ks0 < ks1) load(ks0, A, B);
      for (int ks = ks0; ks < ks1; ks += 2) {
        uint32_t A1[4], B1[NTILE][2];
        const bool two = ks + 1 < ks1;
        if (two) load(ks + 1, A1, B1);
#pragma unroll
        for (int j = 0; j < NTILE; ++j) mma_16816(acc[0][j], A[0], A[1], A[2], A[3], B[j][0], B[j][1]);
        if (two) {
          if (ks + 2 < ks1) load(ks + 2, A, B);
#pragma unroll
          for (int j = 0; j < NTILE; ++j) mma_16816(acc[1][j], A1[0], A1[1], A1[2], A1[3], B1[j][0], B1[j][1]);
        }
      }
      const int g = lane >> 2, c2 = (lane & 3) * 2;
      float* tab = s_logit + h * TB * (EPAD + 1);
#pragma unroll
      for (int j = 0; j < NTILE; ++j) {
        const int r0 = tg * 16 + g, e0 = j * 8 + c2;
        tab[r0 * (EPAD + 1) + e0] = acc[0][j][0] + acc[1][j][0];
        tab[r0 * (EPAD + 1) + e0 + 1] = acc[0][j][1] + acc[1][j][1];
        tab[(r0 + 8) * (EPAD + 1) + e0] = acc[0][j][2] + acc[1][j][2];
        tab[(r0 + 8) * (EPAD + 1) + e0 + 1] = acc[0][j][3] + acc[1][j][3];
      }
    }
  }
  __syncthreads();

  // ---- A2: softmax, top-k, EMA, entropy terms (G lanes per token) ----
  {
    const int tok = t / G, g = t % G;
    const int i = tok0 + tok;
    const bool valid = tok < ntok;
    float zl[EPL];
    float lmax = -INFINITY, labs = 0.f;
#pragma unroll
    for (int j = 0; j < EPL; ++j) {
      const int e = g + G * j;
      if (e < E) {
        float z = 0.f;
#pragma unroll
        for (int hh = 0; hh < WPG; ++hh) z += s_logit[(hh * TB + tok) * (EPAD + 1) + e];
        zl[j] = z + (a.b_gate ? a.b_gate[e] : 0.f);
        lmax = fmaxf(lmax, zl[j]);
        labs = fmaxf(labs, fabsf(zl[j]));
      } else {
        zl[j] = -INFINITY;
      }
    }
    const float m = grp_max<G>(lmax);
    const float zabs = grp_max<G>(labs);
    float lsum = 0.f;
#pragma unroll
    for (int j = 0; j < EPL; ++j)
      if (g + G * j < E) lsum += expf(zl[j] - m);
    const float denom = grp_sum<G>(lsum);
    const int ranks = (k + 1 < E) ? k + 1 : E;
    unsigned taken = 0u;
    unsigned long long topk_mask = 0ull;
    int sel_e[KMAX + 1];
    float sel_z[KMAX + 1];
#pragma unroll
    for (int r = 0; r < KMAX + 1; ++r) {
      sel_e[r] = 0;
      sel_z[r] = 0.f;
      if (r < ranks) {
        float bv = -INFINITY;
        int be = 0x7fffffff;
#pragma unroll
        for (int j = 0; j < EPL; ++j) {
          const int e = g + G * j;
          if (e < E && !((taken >> j) & 1u) && (zl[j] > bv || (zl[j] == bv && e < be))) {
            bv = zl[j];
            be = e;
          }
        }
#pragma unroll
        for (int o = G / 2; o > 0; o >>= 1) {
          const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
          const int oe = __shfl_xor_sync(0xffffffffu, be, o);
          if (ov > bv || (ov == bv && oe < be)) {
            bv = ov;
            be = oe;
          }
        }
        if (be < E && be % G == g) taken |= 1u << (be / G);
        sel_e[r] = be;
        sel_z[r] = bv;
        if (r < k && be < E) topk_mask |= 1ull << be;
      }
    }
    if (valid) {
      float wsum = 0.f, w[KMAX];
#pragma unroll
      for (int p = 0; p < KMAX; ++p) {
        w[p] = 0.f;
        if (p < k) {
          w[p] = expf(sel_z[p] - m) / denom;
          wsum += w[p];
        }
      }
      bool near = false;
#pragma unroll
      for (int p = 0; p < KMAX; ++p)
        if (p + 1 < ranks && (sel_z[p] - sel_z[p + 1]) < 1e-5f * zabs) near = true;
      if (g == 0 && near) atomicAdd(&sm_near, 1);
#pragma unroll
      for (int p = 0; p < KMAX; ++p) {
        if (p < k && p % G == g) {
          const float wp = a.renorm ? w[p] / wsum : w[p];
          a.route_e[static_cast<size_t>(i) * k + p] = sel_e[p];
          a.route_w[static_cast<size_t>(i) * k + p] = wp;
          sm_re[tok * k + p] = sel_e[p];
          sm_rw[tok * k + p] = wp;
        }
      }
    }
#pragma unroll
    for (int j = 0; j < EPL; ++j) {
      const int e = g + G * j;
      float c = 0.f, u = 0.f;
      if (valid && e < E) {
        const float ind = ((topk_mask >> e) & 1ull) ? 1.f : 0.f;
        c = a.beta * sm_ema[tok * EPAD + e] + (1.f - a.beta) * ind;
        a.ema[static_cast<size_t>(i) * E + e] = c;
        if (c > 0.f) u = c * logf(c);
      }
      sm_S[tok * EPAD + e] = c;
      sm_U[tok * EPAD + e] = u;
    }
  }
  __syncthreads();
  }  // kRoute
  const unsigned epoch = a.epoch;
  if constexpr (kRoute) {
    // Block partials per expert: J interleaved runs over the block's tokens,
    // added in run order, then published.
    const int J = kThreads / E;
    const int e = t % E, jr = t / E;
    float S = 0.f, U = 0.f;
    if (jr < J)
      for (int q = jr; q < TB; q += J) {
        S += sm_S[q * EPAD + e];
        U += sm_U[q * EPAD + e];
      }
    sm_rs[t][0] = S;
    sm_rs[t][1] = U;
    __syncthreads();
    if (t < E) {
      float Ss = 0.f, Us = 0.f;
      for (int q = 0; q < J; ++q) {
        Ss += sm_rs[q * E + t][0];
        Us += sm_rs[q * E + t][1];
      }
      if constexpr (MODE == 1) {
        reinterpret_cast<float2*>(a.shard_send)[static_cast<size_t>(blockIdx.x) * E + t] = make_float2(Ss, Us);
      } else {
        unsigned long long* pw = a.part_words + (static_cast<size_t>(blockIdx.x) * E + t) * 2;
        st_word(pw, tag_word(__float_as_uint(Ss), epoch));
        st_word(pw + 1, tag_word(__float_as_uint(Us), epoch));
      }
    }
    if (t == 0 && sm_near) atomicAdd(a.stats + kStNearRoute, static_cast<unsigned long long>(sm_near));
  }
  if constexpr (MODE == 1) return;  // the exchange and the rest run in MODE 2

  // The threshold-free half of the decisions (warp 0, one token per lane),
  // while the other blocks publish their partials.
  TokenPrepT<KMAX> tp;
  if (warp == 0) {
    const bool valid = lane < ntok;
    const int q = valid ? lane * k : 0;
    prepare_token(a.sel, tok0 + lane, valid, sm_re + q, sm_rw + q, sm_ce + q, sm_cw + q, sm_cn + q, tp);
  }

  // ---- exchange 1, B: thresholds from every block's partials (same order in every block) ----
  __syncthreads();  // sm_rs is rewritten below: the block-partial reads above are done
  {
    const int J = kThreads / E;
    const int e = t % E, j = t / E;
    const int nb = MODE == 2 ? a.shard_blocks : static_cast<int>(gridDim.x);
    float S = 0.f, U = 0.f;
    bool ok = true;
    if (MODE == 2 && j < J) {
      // Every rank's blocks, gathered in rank order = global block order.
      const float2* part = reinterpret_cast<const float2*>(a.shard_recv);
      for (int b = j; b < nb; b += J) {
        const float2 v = __ldcg(part + static_cast<size_t>(b) * E + e);
        S += v.x;
        U += v.y;
      }
    } else if (j < J) {
      const int n = 2 * ((nb - j + J - 1) / J);  // (S, U) of blocks j, j + J, ...
      ok = read_tagged<8>(
          a.part_words, n, [&](int q) { return (static_cast<size_t>(j + (q >> 1) * J) * E + e) * 2 + (q & 1); },
          a.wait_epoch, globaltimer() + kBarrierNs, [&](int q, uint32_t v) {
            if (q & 1) U += __uint_as_float(v);
            else S += __uint_as_float(v);
          });
    }
    if (!ok) {
      report_status(a.status, kStatusWaitTimeout, 600);
      sm_fail = 1;
    }
    sm_rs[t][0] = S;
    sm_rs[t][1] = U;
    __syncthreads();
    if (sm_fail) return;
    if (t < E) {
      float Ss = 0.f, Us = 0.f;
      for (int jj = 0; jj < J; ++jj) {
        Ss += sm_rs[jj * E + t][0];
        Us += sm_rs[jj * E + t][1];
      }
      sm_live[t] = Ss > 0.f;
      sm_H[t] = Ss > 0.f ? logf(Ss) - Us / Ss : 0.f;
    }
    __syncthreads();
    if (t == 0 && a.entropy_norm != 0) {  // min-max normalisation only
      float lo = 0.f, hi = 0.f;
      bool any = false;
      for (int ee = 0; ee < E; ++ee) {
        if (!sm_live[ee]) continue;
        if (!any || sm_H[ee] < lo) lo = sm_H[ee];
        if (!any || sm_H[ee] > hi) hi = sm_H[ee];
        any = true;
      }
      sm_lo = lo;
      sm_hi = hi;
    }
    __syncthreads();
    if (t < E) {
      float hb = 0.5f;
      if (sm_live[t]) {
        if (a.entropy_norm == 0) {
          const int Te = MODE == 2 ? a.shard_tokens : T;  // every rank's tokens (Eq. 11's i)
          if (Te > 1) hb = fminf(1.f, fmaxf(0.f, sm_H[t] / logf(static_cast<float>(Te))));
        } else if (sm_hi > sm_lo) {
          hb = (sm_H[t] - sm_lo) / (sm_hi - sm_lo);
        }
      }
      const float tau = a.tau0 * (1.0f + a.alpha * (2.0f * hb - 1.0f));
      sm_tau[t] = tau;
      if (blockIdx.x == 0) a.tau[t] = tau;
    }
    __syncthreads();
  }

  // ---- B: finish the block's decisions (warp 0), publish its rows per group ----
  const int GG = a.G + ((kAttn && a.attn_list) ? 1 : 0);  // the attention list is group G, after the FFN groups
  TokenDecisionT<KMAX> d;
  if (warp == 0) {
    const bool valid = lane < ntok;
    finish_token(a.sel, tok0 + lane, tp, sm_tau, d);
    int n_full = (valid && !d.bad && !d.any) ? 1 : 0;
    // The groups this lane's token has a row in: its recomputed experts, the
    // shared expert, and (DiT-MoE block) the list of recomputing tokens.
    uint32_t gm[3] = {0u, 0u, 0u};
#pragma unroll
    for (int p = 0; p < KMAX; ++p)
      if (d.rec[p]) gm[d.e[p] >> 5] |= 1u << (d.e[p] & 31);
    if (d.shared_row) gm[E >> 5] |= 1u << (E & 31);
    if ((kAttn && a.attn_list) && valid && d.any) gm[a.G >> 5] |= 1u << (a.G & 31);
    for (int g = 0; g < GG; ++g) {
      const unsigned b = __ballot_sync(0xffffffffu, (gm[g >> 5] >> (g & 31)) & 1u);
      if (lane == (g & 31)) sm_bal[g] = b;
    }
    __syncwarp();
    for (int g = lane; g < GG; g += 32)
      st_word(a.count_words + static_cast<size_t>(blockIdx.x) * GG + g, tag_word(__popc(sm_bal[g]), epoch));
    const int c_matched = warp_sum_i(d.n_matched), c_rec = warp_sum_i(d.n_rec), c_near = warp_sum_i(d.n_near);
    const int c_full = warp_sum_i(n_full), c_shared = warp_sum_i(d.shared_row ? 1 : 0);
    if (lane == 0) {
      unsigned long long* st = a.stats;
      atomicAdd(st + kStRecomputed, static_cast<unsigned long long>(c_rec));
      atomicAdd(st + kStReused, static_cast<unsigned long long>(ntok * k - c_rec));
      if (c_shared) atomicAdd(st + kStSharedRecomputed, static_cast<unsigned long long>(c_shared));
      if (!a.sel.refresh) {
        atomicAdd(st + kStMatched, static_cast<unsigned long long>(c_matched));
        atomicAdd(st + kStTokensFullyReused, static_cast<unsigned long long>(c_full));
        if (c_near) atomicAdd(st + kStNearScore, static_cast<unsigned long long>(c_near));
      }
      if (blockIdx.x == 0) {
        const unsigned long long br = static_cast<unsigned long long>(T) * k;
        atomicAdd(st + kStLayerSteps, 1ull);
        atomicAdd(st + kStBranches, br);
        if (a.sel.refresh) atomicAdd(st + kStRefreshSteps, 1ull);
        else atomicAdd(st + kStCacheBranches, br);
      }
    }
  }

  // ---- exchange 2, C: group offsets, this block's prefix, row lists and row gather ----
  {
    const int nb = gridDim.x;
    // Per group: rows of the blocks before this one and of all blocks.  Each
    // group's blocks are split over kThreads / GG threads (block ranges),
    // whose parts are then added in range order.
    {
      const int R = kThreads / GG;
      const int g = t % GG, j = t / GG;
      int pre = 0, tot = 0;
      bool ok = true;
      if (j < R) {
        const int b0 = j * nb / R, b1 = (j + 1) * nb / R;
        const int me = static_cast<int>(blockIdx.x);
        ok = read_tagged<8>(
            a.count_words, b1 - b0, [&](int q) { return static_cast<size_t>(b0 + q) * GG + g; }, a.wait_epoch,
            globaltimer() + kBarrierNs, [&](int q, uint32_t v) {
              const int c = static_cast<int>(v);
              if (b0 + q < me) pre += c;
              tot += c;
            });
      }
      if (!ok) {
        report_status(a.status, kStatusWaitTimeout, 601);
        sm_fail = 1;
      }
      sm_rs[t][0] = __int_as_float(pre);
      sm_rs[t][1] = __int_as_float(tot);
      __syncthreads();
      if (sm_fail) return;
      for (int gg = t; gg < GG; gg += kThreads) {
        int p2 = 0, t2 = 0;
        for (int jj = 0; jj < R; ++jj) {
          p2 += __float_as_int(sm_rs[jj * GG + gg][0]);
          t2 += __float_as_int(sm_rs[jj * GG + gg][1]);
        }
        sm_pre[gg] = p2;
        sm_tot[gg] = t2;
      }
    }
    __syncthreads();
    if (warp == 0) {
      // Exclusive scan of the group totals into offsets, 32 groups at a time.
      int carry = 0;
      for (int g0 = 0; g0 < GG; g0 += 32) {
        const int g = g0 + lane;
        const int v = g < GG ? sm_tot[g] : 0;
        int incl = v;
#pragma unroll
        for (int dd = 1; dd < 32; dd <<= 1) {
          const int u = __shfl_up_sync(0xffffffffu, incl, dd);
          if (lane >= dd) incl += u;
        }
        if (g < GG) sm_off[g] = carry + incl - v;
        carry += __shfl_sync(0xffffffffu, incl, 31);
      }
      if (lane == 0) sm_off[GG] = carry;
    }
    __syncthreads();
    if (blockIdx.x == 0) {
      for (int g = t; g < a.G; g += kThreads) a.counts[g] = sm_tot[g];
      for (int g = t; g <= a.G; g += kThreads) a.offsets[g] = sm_off[g];
      if (kAttn && a.attn_list && t == 0) {
        *a.attn_n = sm_tot[a.G];
        a.sample_lo[T / a.seq] = sm_tot[a.G];
      }
    }
    if (warp == 0) {
      const int i = tok0 + lane;
      const unsigned lt = (1u << lane) - 1u;
      const bool track = kAttn && a.row_of != nullptr;  // DiT-MoE block, sync rule: record the FFN rows
      int pos_of[KMAX];
      int shared_pos = -1;
      // This lane's slots in the block's row table: after the rows of lower lanes.
      int nr = d.shared_row ? 1 : 0;
#pragma unroll
      for (int p = 0; p < KMAX; ++p) nr += d.rec[p] ? 1 : 0;
      int r = nr;
#pragma unroll
      for (int dd = 1; dd < 32; dd <<= 1) {
        const int u = __shfl_up_sync(0xffffffffu, r, dd);
        if (lane >= dd) r += u;
      }
      if (lane == 31) sm_nrows = r;
      r -= nr;
#pragma unroll
      for (int p = 0; p < KMAX; ++p) {
        if (track) pos_of[p] = -1;
        if (d.rec[p]) {
          const int g = d.e[p];
          const int pos = sm_off[g] + sm_pre[g] + __popc(sm_bal[g] & lt);
          a.list[pos] = i * k + d.sl[p];
          if (track) pos_of[p] = pos;
          sm_rows[r][0] = pos;
          sm_rows[r][1] = i;
          ++r;
        }
      }
      if (d.shared_row) {
        const int pos = sm_off[E] + sm_pre[E] + __popc(sm_bal[E] & lt);
        a.list[pos] = i;
        shared_pos = pos;
        sm_rows[r][0] = pos;
        sm_rows[r][1] = i;
      }
      if constexpr (kAttn) {
        if (lane < TB) sm_any[lane] = d.any;
        if (a.row_of || a.attn_list) {
          const int list_pos = a.attn_list ? sm_pre[a.G] + __popc(sm_bal[a.G] & lt) : 0;
          attn_bookkeeping(a, i, lane, ntok, d.any, pos_of, shared_pos, list_pos);
        }
      }
    }
    __syncthreads();
    // Gather the rows' inputs from the token rows staged in phase A (unless
    // the caller gathers them later: xg null).
    const int nv = D / 8;
    uint4* xg = static_cast<uint4*>(a.xg);
    const int n = xg ? sm_nrows : 0;
    for (int r = warp; r < n; r += kThreads / 32) {
      // Under the sync rule the rows of a token with recomputed branches are
      // written by the attention output projection (the FFN-row map).
      if constexpr (kAttn) {
        if (a.gather_final_only && sm_any[sm_rows[r][1] - tok0]) continue;
      }
      const uint4* src = reinterpret_cast<const uint4*>(s_x + (sm_rows[r][1] - tok0) * ldw);
      uint4* dst = xg + static_cast<size_t>(sm_rows[r][0]) * nv;
      for (int c = lane; c < nv; c += 32) dst[c] = src[c];
    }
  }
}

template <int TB, int EPAD>
size_t prep_smem(int D, bool attn) {
  const size_t ldw = static_cast<size_t>(D) + 8;
  const size_t rows = (EPAD + TB) * ldw * 2;                        // gate rows, token rows
  const size_t a_rows = attn ? TB * ldw * 2 : 0;                    // cached attention rows
  return rows + prep_region_bytes(TB, EPAD) + a_rows;
}

template <int TB, int EPAD, int KMAX, int MODE = 0>
cudaError_t prep_launch(const PrepArgs& a, int n_blocks, size_t smem, cudaStream_t s) {
  cudaError_t e =
      set_dyn_smem_on_device(reinterpret_cast<const void*>(prep_kernel<TB, EPAD, KMAX, MODE>), kPrepSmemMax);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(n_blocks);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  // A programmatic dependent launch, like every kernel of the step: the
  // blocks start while the previous kernel drains and wait in
  // griddepcontrol.wait.  (A cooperative launch would not start early.)  The
  // grid barriers need every block resident: the plan keeps the grid within
  // one block per SM's occupancy, the kernels before it never wait on it,
  // and the kernel after it is launched only once every block has passed
  // the wait, so all blocks are resident by the first barrier; the barrier
  // waits are bounded regardless.
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, prep_kernel<TB, EPAD, KMAX, MODE>, a);
}

template <int TB, int EPAD, int KMAX>
int prep_occupancy(size_t smem) {
  if (set_dyn_smem_on_device(reinterpret_cast<const void*>(prep_kernel<TB, EPAD, KMAX, 0>), kPrepSmemMax) !=
      cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  int n = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, prep_kernel<TB, EPAD, KMAX, 0>, kThreads, smem) !=
      cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return n;
}

// Dispatch on (TB, EPAD, KMAX) at run time.
template <typename F>
auto with_shape(int TB, int epad, int kmax, F&& f) {
#define MOECA_PREP_CASE(tb, ep, km) \
  if (TB == tb && epad == ep && kmax == km) return f.template operator()<tb, ep, km>();
#define MOECA_PREP_K(tb, ep) MOECA_PREP_CASE(tb, ep, 2) MOECA_PREP_CASE(tb, ep, 4) MOECA_PREP_CASE(tb, ep, 8)
  MOECA_PREP_K(32, 8) MOECA_PREP_K(32, 16) MOECA_PREP_K(32, 24) MOECA_PREP_K(32, 32)
  MOECA_PREP_K(16, 8) MOECA_PREP_K(16, 16) MOECA_PREP_K(16, 24) MOECA_PREP_K(16, 32)
  MOECA_PREP_K(16, 40) MOECA_PREP_K(16, 48) MOECA_PREP_K(16, 56) MOECA_PREP_K(16, 64)
#undef MOECA_PREP_K
#undef MOECA_PREP_CASE
  return f.template operator()<0, 0, 0>();
}

int kmax_of(int k) { return k <= 2 ? 2 : (k <= 4 ? 4 : 8); }

}  // namespace

#if MOECA_PREP_SHARD
// The token-sharded launches (MODE 1, MODE 2) of the plain build, compiled in
// their own translation unit (prep_shard.cu) beside the plain one.
cudaError_t launch_prep_shard(const PrepArgs& a, const PrepShape& p, int mode, cudaStream_t s) {
  const int nb = (a.T + p.tokens_per_block - 1) / p.tokens_per_block;
  return with_shape(p.tokens_per_block, p.epad, p.kmax, [&]<int tb, int ep, int kk>() -> cudaError_t {
    if constexpr (tb == 0) return cudaErrorInvalidValue;
    else return mode == 1 ? prep_launch<tb, ep, kk, 1>(a, nb, p.smem, s) : prep_launch<tb, ep, kk, 2>(a, nb, p.smem, s);
  });
}
#else
#if MOECA_PREP_ATTN
PrepShape prep_plan_attn(int D, int E, int k, int max_tokens, int n_sms) {
  const bool attn = true;
#else
PrepShape prep_plan_plain(int D, int E, int k, int max_tokens, int n_sms) {
  const bool attn = false;
#endif
  PrepShape p{0, 0, 0, 0};
  if (D % 16 || E < 1 || E > kMaxExperts || k < 1 || k > kMaxTopK) return p;
  const int epad = (E + 7) / 8 * 8;
  const int km = kmax_of(k);
  for (int TB : {32, 16}) {
    if (TB == 32 && epad > 32) continue;  // keeps 32-token blocks' per-lane expert arrays short
    const int nb = (max_tokens + TB - 1) / TB;
    const size_t smem = with_shape(TB, epad, km, [&]<int tb, int ep, int kk>() -> size_t {
      if constexpr (tb == 0) return 0;
      else return prep_smem<tb, ep>(D, attn);
    });
    if (smem == 0 || smem > kPrepSmemMax) continue;
    const int occ = with_shape(TB, epad, km, [&]<int tb, int ep, int kk>() -> int {
      if constexpr (tb == 0) return 0;
      else return prep_occupancy<tb, ep, kk>(smem);
    });
    if (occ <= 0 || static_cast<long long>(occ) * n_sms < nb) continue;
    p.tokens_per_block = TB;
    p.epad = epad;
    p.kmax = km;
    p.smem = smem;
    p.attn = attn;
    return p;
  }
  return p;
}

#if MOECA_PREP_ATTN
cudaError_t launch_prep_attn(const PrepArgs& a, const PrepShape& p, cudaStream_t s) {
#else
cudaError_t launch_prep_plain(const PrepArgs& a, const PrepShape& p, cudaStream_t s) {
#endif
  const int nb = (a.T + p.tokens_per_block - 1) / p.tokens_per_block;
  return with_shape(p.tokens_per_block, p.epad, p.kmax, [&]<int tb, int ep, int kk>() -> cudaError_t {
    if constexpr (tb == 0) return cudaErrorInvalidValue;
    else return prep_launch<tb, ep, kk>(a, nb, p.smem, s);
  });
}

#if !MOECA_PREP_ATTN
PrepShape prep_plan(int D, int E, int k, int max_tokens, int n_sms, bool attn) {
  return attn ? prep_plan_attn(D, E, k, max_tokens, n_sms) : prep_plan_plain(D, E, k, max_tokens, n_sms);
}

cudaError_t launch_prep(const PrepArgs& a, const PrepShape& p, cudaStream_t s) {
  return p.attn ? launch_prep_attn(a, p, s) : launch_prep_plain(a, p, s);
}
#endif

#endif  // MOECA_PREP_SHARD

}  // namespace moeca
