// Combine of fresh and cached branch outputs (Eq. 8) with the residual of
// Eq. 5 / Eq. 6, and the cached-norm refresh that Eq. 9's o reads next step.
//
// One warp per token, 16-byte vectors over D:
//   y_i = sum_{p=1..k} w_{i,p}^t cache_h[i, slot(p)]  (+ shared_h[i])
//   out_i = x_i + y_i            (fp32 accumulation in p order, rounded once)
//   cache_norm[i, q] = ||cache_h[i, q]||_2 for every slot q (slot is a
//   permutation of 0..k-1, so the k rows read are all of the token's slots).
#include "common.cuh"
#include "kernels.h"

namespace moeca {
namespace {

constexpr int kWarps = 8;

// CG 16-byte chunks per lane are in flight at once (all k cache rows, the
// shared row and x loaded before any arithmetic).
template <typename TI, int KMAX, int CG>
__global__ void __launch_bounds__(kWarps * 32) combine_kernel(CombineArgs a) {
  constexpr int V = Elem<TI>::kVec;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int i = blockIdx.x * kWarps + warp;
  if (i >= a.T) return;
  const int k = a.k, D = a.D, nvec = D / V;
  const TI* x = static_cast<const TI*>(a.x) + static_cast<size_t>(i) * D;
  TI* out = static_cast<TI*>(a.out) + static_cast<size_t>(i) * D;
  const TI* ch = static_cast<const TI*>(a.cache_h) + static_cast<size_t>(i) * k * D;
  const TI* sh = a.shared_h ? static_cast<const TI*>(a.shared_h) + static_cast<size_t>(i) * D : nullptr;
  float w[KMAX];
  int q[KMAX];
  bool bad = false;
#pragma unroll
  for (int p = 0; p < KMAX; ++p) {
    w[p] = 0.f;
    q[p] = 0;
    if (p < k) {
      w[p] = a.route_w[static_cast<size_t>(i) * k + p];
      q[p] = a.slot[static_cast<size_t>(i) * k + p];
      if (q[p] < 0 || q[p] >= k) bad = true;
    }
  }
  if (bad) {
    if (lane == 0) report_status(a.status, kStatusBadIndex, 3000000 + i);
    return;
  }
  float ss[KMAX];
#pragma unroll
  for (int p = 0; p < KMAX; ++p) ss[p] = 0.f;
  for (int c0 = 0; c0 < nvec; c0 += 32 * CG) {
    float h[CG][KMAX][V], xs[CG][V], hs[CG][V];
#pragma unroll
    for (int g = 0; g < CG; ++g) {
      const int c = c0 + g * 32 + lane;
      if (c < nvec) {
#pragma unroll
        for (int p = 0; p < KMAX; ++p)
          if (p < k) load_vec(ch + static_cast<size_t>(q[p]) * D + c * V, h[g][p]);
        load_vec(x + c * V, xs[g]);
        if (sh) load_vec(sh + c * V, hs[g]);
      }
    }
#pragma unroll
    for (int g = 0; g < CG; ++g) {
      const int c = c0 + g * 32 + lane;
      if (c < nvec) {
        float y[V];
#pragma unroll
        for (int j = 0; j < V; ++j) y[j] = 0.f;
#pragma unroll
        for (int p = 0; p < KMAX; ++p) {
          if (p < k) {
#pragma unroll
            for (int j = 0; j < V; ++j) {
              y[j] = fmaf(w[p], h[g][p][j], y[j]);
              ss[p] = fmaf(h[g][p][j], h[g][p][j], ss[p]);
            }
          }
        }
        if (sh) {
#pragma unroll
          for (int j = 0; j < V; ++j) y[j] += hs[g][j];
        }
#pragma unroll
        for (int j = 0; j < V; ++j) xs[g][j] += y[j];
        store_vec(out + c * V, xs[g]);
      }
    }
  }
#pragma unroll
  for (int p = 0; p < KMAX; ++p) {
    if (p < k) {
      const float s2 = warp_sum(ss[p]);
      if (lane == 0) a.cache_norm[static_cast<size_t>(i) * k + q[p]] = sqrtf(s2);
    }
  }
}

template <typename TI>
void launch_t(const CombineArgs& a, cudaStream_t s) {
  const int grid = (a.T + kWarps - 1) / kWarps;
  if (a.k <= 2) combine_kernel<TI, 2, 4><<<grid, kWarps * 32, 0, s>>>(a);
  else if (a.k <= 4) combine_kernel<TI, 4, 2><<<grid, kWarps * 32, 0, s>>>(a);
  else combine_kernel<TI, 8, 1><<<grid, kWarps * 32, 0, s>>>(a);
}

}  // namespace

cudaError_t launch_combine(const CombineArgs& a, bool bf16, cudaStream_t s) {
  if (bf16) launch_t<__nv_bfloat16>(a, s);
  else launch_t<float>(a, s);
  return cudaGetLastError();
}

}  // namespace moeca
