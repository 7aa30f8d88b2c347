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

template <typename TI>
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
  float w[kMaxTopK];
  int q[kMaxTopK];
  bool bad = false;
#pragma unroll
  for (int p = 0; p < kMaxTopK; ++p) {
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
  float ss[kMaxTopK];
#pragma unroll
  for (int p = 0; p < kMaxTopK; ++p) ss[p] = 0.f;
  for (int c = lane; c < nvec; c += 32) {
    float y[V];
#pragma unroll
    for (int j = 0; j < V; ++j) y[j] = 0.f;
#pragma unroll
    for (int p = 0; p < kMaxTopK; ++p) {
      if (p < k) {
        float h[V];
        load_vec(ch + static_cast<size_t>(q[p]) * D + c * V, h);
#pragma unroll
        for (int j = 0; j < V; ++j) {
          y[j] = fmaf(w[p], h[j], y[j]);
          ss[p] = fmaf(h[j], h[j], ss[p]);
        }
      }
    }
    if (sh) {
      float h[V];
      load_vec(sh + c * V, h);
#pragma unroll
      for (int j = 0; j < V; ++j) y[j] += h[j];
    }
    float xv[V];
    load_vec(x + c * V, xv);
#pragma unroll
    for (int j = 0; j < V; ++j) xv[j] += y[j];
    store_vec(out + c * V, xv);
  }
#pragma unroll
  for (int p = 0; p < kMaxTopK; ++p) {
    if (p < k) {
      const float s = warp_sum(ss[p]);
      if (lane == 0) a.cache_norm[static_cast<size_t>(i) * k + q[p]] = sqrtf(s);
    }
  }
}

}  // namespace

cudaError_t launch_combine(const CombineArgs& a, bool bf16, cudaStream_t s) {
  const int grid = (a.T + kWarps - 1) / kWarps;
  if (bf16) combine_kernel<__nv_bfloat16><<<grid, kWarps * 32, 0, s>>>(a);
  else combine_kernel<float><<<grid, kWarps * 32, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace moeca
