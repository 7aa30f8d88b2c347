// Branch selection and compaction of the branch-cached MoE layer.
//
// select_kernel, one token per thread (Sec. 4.2):
//   * match each routed branch p against the token's cached branches by
//     expert id; an unmatched branch is always recomputed;
//   * score a matched branch  s = w_p + lambda1 |w_p - w_q^{t0}|
//     + lambda2 ||h_q|| / sum_j ||h_j||   (Eq. 9)  and recompute iff s > tau_e;
//   * matched branches keep their cache slot q(p); unmatched ones take the
//     slots whose expert is no longer routed, ascending p -> ascending q;
//     on a full-computation step every branch is recomputed with slot = p;
//   * write the new cache metadata, token_any = (R_i non-empty, Sec. 4.1) and
//     per-block counts of recomputed rows per expert group (warp ballots).
// The last block scans the per-block counts into per-group row offsets.
//
// compact_kernel, same token blocks: ranks each recomputed row inside its
// group in ascending token order (ballot + popc prefix) and writes the row
// list (token * k + slot for routed experts, token for the shared expert).
// gather_kernel then copies every listed row's layer input into a
// contiguous buffer for the GEMMs, one warp per row over the whole list.
#include "common.cuh"
#include "kernels.h"
#include "select_token.cuh"

namespace moeca {
namespace {

constexpr int kThreads = kSelectTokensPerBlock;
constexpr int kWarps = kThreads / 32;
constexpr int kMaxGroups = kMaxExperts + 1;

// KMAX >= k bounds the per-token loops at compile time.
template <int KMAX>
__global__ void __launch_bounds__(kThreads) select_kernel(SelectArgs a) {
  pdl_entry();
  const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
  const int i = blockIdx.x * kThreads + t;
  const bool valid = i < a.T;
  const int k = a.k, E = a.E, G = a.G;
  TokenDecisionT<KMAX> d;
  const size_t b0 = static_cast<size_t>(valid ? i : 0) * a.k;
  decide_token<KMAX>(a, i, valid, a.route_e + b0, a.route_w + b0, a.cache_e + b0, a.cache_w + b0, a.cache_norm + b0, d);
  const int* e = d.e;
  const bool* rec = d.rec;
  const bool any = d.any, bad = d.bad, shared_row = d.shared_row;
  const int n_matched = d.n_matched, n_rec = d.n_rec, n_near = d.n_near;

  // Rows per (warp, group) by ballot, then per block.
  __shared__ int sm_wc[kWarps][kMaxGroups];
  for (int g = 0; g < G; ++g) {
    bool has = false;
    if (g < E) {
#pragma unroll
      for (int p = 0; p < KMAX; ++p) has |= (rec[p] && e[p] == g);
    } else {
      has = shared_row;
    }
    const unsigned b = __ballot_sync(0xffffffffu, has);
    if (lane == 0) sm_wc[warp][g] = __popc(b);
  }
  // Branch counters.
  const int c_matched = warp_sum_i(n_matched);
  const int c_rec = warp_sum_i(n_rec);
  const int c_near = warp_sum_i(n_near);
  const int c_full = warp_sum_i(valid && !bad && !any ? 1 : 0);
  const int c_shared = warp_sum_i(shared_row ? 1 : 0);
  __shared__ int sm_c[kWarps][5];
  if (lane == 0) {
    sm_c[warp][0] = c_matched;
    sm_c[warp][1] = c_rec;
    sm_c[warp][2] = c_near;
    sm_c[warp][3] = c_full;
    sm_c[warp][4] = c_shared;
  }
  __syncthreads();
  for (int g = t; g < G; g += kThreads) {
    int s = 0;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) s += sm_wc[w][g];
    a.block_counts[static_cast<size_t>(blockIdx.x) * G + g] = s;
  }
  if (t == 0) {
    int tot[5] = {0, 0, 0, 0, 0};
    for (int w = 0; w < kWarps; ++w)
      for (int j = 0; j < 5; ++j) tot[j] += sm_c[w][j];
    const int nb = min(kThreads, a.T - static_cast<int>(blockIdx.x) * kThreads);
    unsigned long long* st = a.stats;
    atomicAdd(st + kStRecomputed, static_cast<unsigned long long>(tot[1]));
    atomicAdd(st + kStReused, static_cast<unsigned long long>(nb * k - tot[1]));
    if (tot[4]) atomicAdd(st + kStSharedRecomputed, static_cast<unsigned long long>(tot[4]));
    if (!a.refresh) {
      atomicAdd(st + kStMatched, static_cast<unsigned long long>(tot[0]));
      atomicAdd(st + kStTokensFullyReused, static_cast<unsigned long long>(tot[3]));
      if (tot[2]) atomicAdd(st + kStNearScore, static_cast<unsigned long long>(tot[2]));
    }
    if (blockIdx.x == 0) {
      const unsigned long long br = static_cast<unsigned long long>(a.T) * k;
      atomicAdd(st + kStLayerSteps, 1ull);
      atomicAdd(st + kStBranches, br);
      if (a.refresh) atomicAdd(st + kStRefreshSteps, 1ull);
      else atomicAdd(st + kStCacheBranches, br);
    }
  }
  // The last block turns per-block counts into offsets.
  __threadfence();
  __syncthreads();
  __shared__ unsigned ticket;
  if (t == 0) ticket = atomicAdd(a.done, 1u);
  __syncthreads();
  if (ticket != gridDim.x - 1) return;
  __threadfence();
  // Chunks of 16 blocks: every thread loads counts in parallel, then one
  // thread per group scans the chunk in block order.
  __shared__ int sm_tot[kMaxGroups];
  __shared__ int sm_chunk[16][kMaxGroups];
  for (int g = t; g < G; g += kThreads) sm_tot[g] = 0;
  for (unsigned b0 = 0; b0 < gridDim.x; b0 += 16) {
    const int nb = min(16u, gridDim.x - b0);
    __syncthreads();
    for (int idx = t; idx < nb * G; idx += kThreads)
      sm_chunk[idx / G][idx % G] = __ldcg(a.block_counts + static_cast<size_t>(b0 + idx / G) * G + idx % G);
    __syncthreads();
    for (int g = t; g < G; g += kThreads) {
      int run = sm_tot[g];
      for (int j = 0; j < nb; ++j) {
        a.block_offsets[static_cast<size_t>(b0 + j) * G + g] = run;
        run += sm_chunk[j][g];
      }
      sm_tot[g] = run;
    }
  }
  __syncthreads();
  for (int g = t; g < G; g += kThreads) a.counts[g] = sm_tot[g];
  if (t == 0) {
    int off = 0;
    for (int g = 0; g < G; ++g) {
      a.offsets[g] = off;
      off += sm_tot[g];
    }
    a.offsets[G] = off;
    *a.done = 0u;
  }
}

template <typename TI, int KMAX>
__global__ void __launch_bounds__(kThreads) compact_kernel(CompactArgs a) {
  pdl_entry();
  const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
  const int i = blockIdx.x * kThreads + t;
  const bool valid = i < a.T;
  const int k = a.k, E = a.E, G = a.G;
  int e[KMAX], sl[KMAX];
  bool rec[KMAX];
  bool any = false;
#pragma unroll
  for (int p = 0; p < KMAX; ++p) {
    e[p] = -1;
    sl[p] = 0;
    rec[p] = false;
    if (valid && p < k) {
      const size_t b = static_cast<size_t>(i) * k + p;
      rec[p] = a.recompute[b] != 0;
      e[p] = a.route_e[b];
      sl[p] = a.slot[b];
      if (e[p] < 0 || e[p] >= E) rec[p] = false;  // flagged by select
    }
  }
  if (valid) any = a.token_any[i] != 0;
  const bool shared_row = valid && a.n_shared && (a.refresh || a.shared_policy || any);

  __shared__ unsigned sm_bal[kWarps][kMaxGroups];
  __shared__ int sm_pre[kWarps][kMaxGroups];
  for (int g = 0; g < G; ++g) {
    bool has = false;
    if (g < E) {
#pragma unroll
      for (int p = 0; p < KMAX; ++p) has |= (rec[p] && e[p] == g);
    } else {
      has = shared_row;
    }
    const unsigned b = __ballot_sync(0xffffffffu, has);
    if (lane == 0) sm_bal[warp][g] = b;
  }
  __syncthreads();
  for (int g = t; g < G; g += kThreads) {
    int run = a.offsets[g] + a.block_offsets[static_cast<size_t>(blockIdx.x) * G + g];
#pragma unroll
    for (int w = 0; w < kWarps; ++w) {
      sm_pre[w][g] = run;
      run += __popc(sm_bal[w][g]);
    }
  }
  __syncthreads();
  const unsigned lt = (1u << lane) - 1u;
#pragma unroll
  for (int p = 0; p < KMAX; ++p) {
    if (rec[p]) {
      const int g = e[p];
      const int pos = sm_pre[warp][g] + __popc(sm_bal[warp][g] & lt);
      a.list[pos] = i * k + sl[p];
    }
  }
  if (shared_row) {
    const int pos = sm_pre[warp][E] + __popc(sm_bal[warp][E] & lt);
    a.list[pos] = i;
  }
}

// Gather of every listed row's layer input into the group-contiguous buffer
// the GEMMs read: one warp per row over the whole list (rows of group g are
// [offsets[g], offsets[g + 1])), 16-byte vectors.  A list entry is
// token * k + slot for a routed group and the token for the shared group.
template <typename TI>
__global__ void __launch_bounds__(256) gather_kernel(CompactArgs a) {
  pdl_entry();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = a.G, E = a.E;
  __shared__ int off_sm[kMaxGroups + 1];  // group offsets, read once
  for (int g = threadIdx.x; g <= G; g += blockDim.x) off_sm[g] = a.offsets[g];
  __syncthreads();
  const int rows = off_sm[G];
  const int nv = a.D * static_cast<int>(sizeof(TI)) / 16;
  const uint4* x = static_cast<const uint4*>(a.x);
  uint4* xg = static_cast<uint4*>(a.xg);
  for (int r = blockIdx.x * 8 + warp; r < rows; r += gridDim.x * 8) {
    // Group of row r: the last g with offsets[g] <= r (G <= 65: a short search).
    int lo = 0, hi = G - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (off_sm[mid] <= r) lo = mid;
      else hi = mid - 1;
    }
    const int ent = a.list[r];
    const int tok = lo < E ? ent / a.k : ent;
    if (tok < 0 || tok >= a.T) {
      if (lane == 0) report_status(a.status, kStatusBadIndex, 5100000 + r);
      continue;
    }
    const uint4* src = x + static_cast<size_t>(tok) * nv;
    uint4* dst = xg + static_cast<size_t>(r) * nv;
    for (int c = lane; c < nv; c += 32) dst[c] = src[c];
  }
}

}  // namespace

cudaError_t launch_select(const SelectArgs& a, cudaStream_t s) {
  const int grid = (a.T + kThreads - 1) / kThreads;
  if (a.k <= 2) return launch_pdl(select_kernel<2>, dim3(grid), dim3(kThreads), 0, s, a);
  if (a.k <= 4) return launch_pdl(select_kernel<4>, dim3(grid), dim3(kThreads), 0, s, a);
  return launch_pdl(select_kernel<kMaxTopK>, dim3(grid), dim3(kThreads), 0, s, a);
}

cudaError_t launch_compact(const CompactArgs& a, bool bf16, cudaStream_t s) {
  const int grid = (a.T + kThreads - 1) / kThreads;
  auto run = [&](auto kern) { return launch_pdl(kern, dim3(grid), dim3(kThreads), 0, s, a); };
  cudaError_t e;
  if (bf16) e = a.k <= 2 ? run(compact_kernel<__nv_bfloat16, 2>) : a.k <= 4 ? run(compact_kernel<__nv_bfloat16, 4>)
                                                                            : run(compact_kernel<__nv_bfloat16, kMaxTopK>);
  else e = a.k <= 2 ? run(compact_kernel<float, 2>) : a.k <= 4 ? run(compact_kernel<float, 4>)
                                                             : run(compact_kernel<float, kMaxTopK>);
  if (e != cudaSuccess || a.xg == nullptr) return e;
  // The row gather runs over the whole list, one warp per row.
  const int rows = a.T * (a.k + a.n_shared);
  const int ggrid = (rows + 7) / 8;
  return bf16 ? launch_pdl(gather_kernel<__nv_bfloat16>, dim3(ggrid), dim3(256), 0, s, a)
              : launch_pdl(gather_kernel<float>, dim3(ggrid), dim3(256), 0, s, a);
}

cudaError_t launch_gather(const CompactArgs& a, bool bf16, cudaStream_t s) {
  const int rows = a.T * (a.k + a.n_shared);
  const int ggrid = (rows + 7) / 8;
  return bf16 ? launch_pdl(gather_kernel<__nv_bfloat16>, dim3(ggrid), dim3(256), 0, s, a)
              : launch_pdl(gather_kernel<float>, dim3(ggrid), dim3(256), 0, s, a);
}

}  // namespace moeca
