// Combine of fresh and cached branch outputs (Eq. 8) with the residual of
// Eq. 5 / Eq. 6, and the cached-norm refresh that Eq. 9's o reads next step.
//
// One warp per token, 16-byte vectors over D:
//   y_i = sum_{p=1..k} w_{i,p}^t cache_h[i, slot(p)]  (+ shared_h[i])
//   out_i = x_i + y_i            (fp32 accumulation in p order, rounded once)
//   out_i = x_i + g_i * y_i      in an AdaLN block (g the sample's MoE gate, Sec. 3)
//   cache_norm[i, q] = ||cache_h[i, q]||_2 for every slot q (slot is a
//   permutation of 0..k-1, so the k rows read are all of the token's slots).
// Under the token-level reading of Sec. 4.1 (token_reuse_policy 1) every
// computing token also stores its y in fp32, and on a cache step a token
// whose recompute set is empty takes y from there instead (its cache rows
// and norms are unchanged, so they are not read).
#include "common.cuh"
#include "kernels.h"

namespace moeca {
namespace {

constexpr int kWarps = 8;

// CG 16-byte chunks per lane are in flight at once (all k cache rows, the
// shared row and x loaded before any arithmetic).
template <typename TI, int KMAX, int CG, bool GATED, bool YC>
__global__ void __launch_bounds__(kWarps * 32) combine_kernel(CombineArgs a) {
  constexpr int V = Elem<TI>::kVec;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int i = blockIdx.x * kWarps + warp;
  if (i >= a.T) {
    pdl_entry();
    return;
  }
  if (a.rearm && blockIdx.x == 0 && threadIdx.x == 0) {
    // The grouped GEMM before this kernel has ended: re-arm its ticket.
    pdl_entry();
    *a.rearm = 0;
  }
  const int k = a.k, D = a.D, nvec = D / V;
  const TI* x = static_cast<const TI*>(a.x) + static_cast<size_t>(i) * D;
  TI* out = static_cast<TI*>(a.out) + static_cast<size_t>(i) * D;
  const TI* ch = static_cast<const TI*>(a.cache_h) + static_cast<size_t>(i) * k * D;
  const TI* sh = a.shared_h ? static_cast<const TI*>(a.shared_h) + static_cast<size_t>(i) * D : nullptr;
  const float* gr = GATED ? a.gate + static_cast<size_t>(i / a.seq) * a.gate_ld : nullptr;
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
  // The gate weights, slots and layer input come from earlier kernels than
  // the one before (prep, the layer below's combine); only the cache rows
  // (and shared rows) are the previous kernel's output.  Load the first
  // input chunks, then wait.
  const uint4* x4 = reinterpret_cast<const uint4*>(x);
  uint4 x_first[CG];
#pragma unroll
  for (int g = 0; g < CG; ++g) {
    const int c = g * 32 + lane;
    if (c < nvec) x_first[g] = x4[c];
  }
  // token_any comes from the preparation kernel, which completed before the
  // previous kernel passed its own dependency wait.
  const bool copy_tok = YC && a.copy_y && !a.token_any[i];
  pdl_entry();
  if (bad) {
    if (lane == 0) report_status(a.status, kStatusBadIndex, 3000000 + i);
    return;
  }
  if constexpr (YC) {
    if (copy_tok) {
      // Sec. 4.1, token level: y = y^{t0}, read back in fp32.
      const float4* yc = reinterpret_cast<const float4*>(a.cache_y + static_cast<size_t>(i) * D);
      for (int c = lane; c < nvec; c += 32) {
        float xs[V], y[V];
#pragma unroll
        for (int j = 0; j < V / 4; ++j) {
          const float4 v = yc[static_cast<size_t>(c) * (V / 4) + j];
          y[4 * j] = v.x; y[4 * j + 1] = v.y; y[4 * j + 2] = v.z; y[4 * j + 3] = v.w;
        }
        unpack_vec(x4[c], xs, static_cast<TI*>(nullptr));
        if constexpr (GATED) {
#pragma unroll
          for (int j = 0; j < V; ++j) xs[j] = fmaf(gr[c * V + j], y[j], xs[j]);
        } else {
#pragma unroll
          for (int j = 0; j < V; ++j) xs[j] += y[j];
        }
        store_vec(out + c * V, xs);
      }
      return;
    }
  }
  float ss[KMAX];
#pragma unroll
  for (int p = 0; p < KMAX; ++p) ss[p] = 0.f;
  // Raw 16-byte vectors stay packed in registers until used.
  const uint4* ch4 = reinterpret_cast<const uint4*>(ch);
  const uint4* sh4 = reinterpret_cast<const uint4*>(sh);
  for (int c0 = 0; c0 < nvec; c0 += 32 * CG) {
    uint4 h[CG][KMAX], xr[CG], hr[CG];
    float4 gq[GATED ? CG : 1][V / 4];  // AdaLN gate values of the chunks, loaded with the rows
#pragma unroll
    for (int g = 0; g < CG; ++g) {
      const int c = c0 + g * 32 + lane;
      if (c < nvec) {
#pragma unroll
        for (int p = 0; p < KMAX; ++p)
          if (p < k) h[g][p] = ch4[static_cast<size_t>(q[p]) * nvec + c];
        xr[g] = c0 == 0 ? x_first[g] : x4[c];
        if (sh) hr[g] = sh4[c];
        if constexpr (GATED) {
#pragma unroll
          for (int j = 0; j < V / 4; ++j) gq[g][j] = __ldg(reinterpret_cast<const float4*>(gr + c * V) + j);
        }
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
            float hv[V];
            unpack_vec(h[g][p], hv, static_cast<TI*>(nullptr));
#pragma unroll
            for (int j = 0; j < V; ++j) {
              y[j] = fmaf(w[p], hv[j], y[j]);
              ss[p] = fmaf(hv[j], hv[j], ss[p]);
            }
          }
        }
        if (sh) {
          float hv[V];
          unpack_vec(hr[g], hv, static_cast<TI*>(nullptr));
#pragma unroll
          for (int j = 0; j < V; ++j) y[j] += hv[j];
        }
        if constexpr (YC) {
          float4* yo = reinterpret_cast<float4*>(a.cache_y + static_cast<size_t>(i) * D) + static_cast<size_t>(c) * (V / 4);
#pragma unroll
          for (int j = 0; j < V / 4; ++j) yo[j] = make_float4(y[4 * j], y[4 * j + 1], y[4 * j + 2], y[4 * j + 3]);
        }
        float xs[V];
        unpack_vec(xr[g], xs, static_cast<TI*>(nullptr));
        if constexpr (GATED) {
          const float* gv = reinterpret_cast<const float*>(gq[g]);
#pragma unroll
          for (int j = 0; j < V; ++j) xs[j] = fmaf(gv[j], y[j], xs[j]);
        } else {
#pragma unroll
          for (int j = 0; j < V; ++j) xs[j] += y[j];
        }
        store_vec(out + c * V, xs);
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

template <typename TI, bool GATED, bool YC>
void launch_t(const CombineArgs& a, cudaStream_t s) {
  const int grid = (a.T + kWarps - 1) / kWarps;
  // The gated form holds the gate values with the rows: half the chunks in flight keeps it near 128 registers.
  if (a.k <= 2) launch_pdl(combine_kernel<TI, 2, GATED ? 2 : 4, GATED, YC>, dim3(grid), dim3(kWarps * 32), 0, s, a);
  else if (a.k <= 4) launch_pdl(combine_kernel<TI, 4, 2, GATED, YC>, dim3(grid), dim3(kWarps * 32), 0, s, a);
  else launch_pdl(combine_kernel<TI, 8, 1, GATED, YC>, dim3(grid), dim3(kWarps * 32), 0, s, a);
}

template <bool YC>
void launch_y(const CombineArgs& a, bool bf16, cudaStream_t s) {
  if (bf16 && a.gate) launch_t<__nv_bfloat16, true, YC>(a, s);
  else if (bf16) launch_t<__nv_bfloat16, false, YC>(a, s);
  else launch_t<float, false, YC>(a, s);
}

}  // namespace

cudaError_t launch_combine(const CombineArgs& a, bool bf16, cudaStream_t s) {
  if (a.gate && !bf16) return cudaErrorInvalidValue;  // AdaLN blocks are bf16 only
  if (a.cache_y && (!a.token_any || reinterpret_cast<uintptr_t>(a.cache_y) % 16)) return cudaErrorInvalidValue;
  if (a.cache_y) launch_y<true>(a, bf16, s);
  else launch_y<false>(a, bf16, s);
  return cudaGetLastError();
}

}  // namespace moeca
