// Router of the branch-cached MoE layer.
//
// Per token i (a group of up to 8 lanes): gate logits z = x_i W_g^T (+ b)
// with fp32 accumulation, softmax over the E experts, top-k by descending logit with
// ties to the lower expert id, optional renormalisation of the k weights
// (Eq. 7).  The same pass updates the EMA statistic
//   C_{e,i} <- beta C_{e,i} + (1 - beta) 1[e in B_i]        (Eq. 10)
// and accumulates per block S_e = sum_i C_{e,i} and U_e = sum_i C ln C, from
// which the last block to finish derives the spatial entropy
//   H_e = ln S_e - U_e / S_e  (= -sum_i P ln P with P = C / S, Eq. 11),
// its normalisation and the expert threshold tau_e (Eq. 12).
#include <mutex>
#include <type_traits>

#include "common.cuh"
#include "kernels.h"
#include "moeca.h"

namespace moeca {
namespace {


// Bit-exact group reductions over the G lanes of one token (G divides 32).
template <int G>
__device__ __forceinline__ float group_max(float v) {
#pragma unroll
  for (int o = G / 2; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
template <int G>
__device__ __forceinline__ float group_sum(float v) {
#pragma unroll
  for (int o = G / 2; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// One token per group of G lanes (G = min(E, 8) rounded down to a power of
// two); lane g of a group owns experts e = g + G j, j < EPL.  One thread
// stages the block's token rows and the gate matrix into shared memory with
// bulk async copies completing on one mbarrier (rows padded by 16 bytes, so
// the tokens of a warp and the G experts of a group hit different banks);
// shapes too large for shared memory read the same data through L1 / L2.
// Each lane accumulates its logits over D in fp32; softmax and top-k run as
// shuffles inside the group.
//
// bf16 with both staged: the logits come from the tensor cores instead
// (mma.sync m16n8k16, bf16 in, fp32 accumulate over D in order): 16-token
// groups by 8-expert tiles, the gate rows zero-padded to a multiple of 8,
// into a shared logit table the lanes then read.
template <typename TI, int G, int EPL, int NT>
__global__ void __launch_bounds__(NT) router_kernel(RouterArgs a, int stage_x, int stage_wg) {
  constexpr int V = Elem<TI>::kVec;
  constexpr int TB = NT / G;                  // tokens per block
  constexpr int EMAXB = G * EPL;              // experts covered by a group
  constexpr int kThreads = NT;
  constexpr bool kTensor = std::is_same_v<TI, __nv_bfloat16> && TB % 16 == 0 && TB / 16 <= NT / 32;
  // 32-token blocks for wide gates (256 threads): the logit table and the
  // entropy terms take the gate rows' shared memory once the tensor cores
  // are done with it, so the gate matrix and 32 token rows fit beside each
  // other (the host launches this form only with both staged).
  constexpr bool kAlias = kTensor && NT == 256;
  extern __shared__ uint4 sm_dyn[];           // [EPAD][rowv + 1] gate rows, [TB][rowv + 1] token rows, logits
  __shared__ float sm_S_st[kAlias ? 1 : TB * EMAXB];
  __shared__ float sm_U_st[kAlias ? 1 : TB * EMAXB];
  float* sm_S = sm_S_st;
  float* sm_U = sm_U_st;
  __shared__ int sm_near;
  __shared__ __align__(8) uint64_t sm_bar;
  const int t = threadIdx.x;
  const int g = t % G, tok = t / G;
  const int E = a.E, k = a.k;
  const int rowv = a.D / V, pstride = rowv + 1;
  const int i = blockIdx.x * TB + tok;
  const bool valid = i < a.T;
  const int ntok = min(TB, a.T - static_cast<int>(blockIdx.x) * TB);
  // Loaded before the dependency wait: the gate bias (a weight) and this
  // token's EMA values (this layer's state, last written one step earlier by
  // this kernel, which completed before the previous kernel could start).
  float bias_pre[EPL], ema_pre[EPL];
#pragma unroll
  for (int j = 0; j < EPL; ++j) {
    const int e = g + G * j;
    bias_pre[j] = (e < E && a.b_gate) ? a.b_gate[e] : 0.f;
    ema_pre[j] = (valid && e < E) ? a.ema[static_cast<size_t>(i) * E + e] : 0.f;
  }
  pdl_entry();
  const uint4* wsrc = static_cast<const uint4*>(a.w_gate);
  int wstride = rowv;
  const uint4* xsrc = static_cast<const uint4*>(a.x) + static_cast<size_t>(i) * rowv;
  const int epad = (E + 7) / 8 * 8;
  uint4* sm_wg = sm_dyn;
  uint4* sm_x = sm_dyn + (stage_wg ? epad * pstride : 0);
  const bool tensor = kTensor && stage_x && stage_wg;
  float* sm_logit = kAlias ? reinterpret_cast<float*>(sm_wg)
                           : reinterpret_cast<float*>(sm_x + TB * pstride);  // [TB][epad + 1], tensor path
  if constexpr (kAlias) {
    sm_S = sm_logit + TB * (epad + 1);
    sm_U = sm_S + TB * EMAXB;
  }
  if (t == 0) {
    sm_near = 0;
    if (stage_wg || stage_x) {
      mbar_init(smem_u32(&sm_bar), 1);
      asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
  }
  __syncthreads();
  if (stage_wg || stage_x) {
    const uint32_t bar = smem_u32(&sm_bar);
    const uint32_t row_bytes = static_cast<uint32_t>(rowv) * 16;
    // Lane 0's expect-tx carries the barrier's only arrival; the lanes of
    // warp 0 then issue one row copy each.
    if (t == 0) mbar_expect_tx(bar, row_bytes * ((stage_wg ? E : 0) + (stage_x ? ntok : 0)));
    if (t < 32) {
      __syncwarp();
      if (stage_wg)
        for (int e = t; e < E; e += 32) bulk_g2s(smem_u32(sm_wg + e * pstride), wsrc + e * rowv, row_bytes, bar);
      if (stage_x)
        for (int q = t; q < ntok; q += 32)
          bulk_g2s(smem_u32(sm_x + q * pstride),
                   static_cast<const uint4*>(a.x) + static_cast<size_t>(blockIdx.x * TB + q) * rowv, row_bytes, bar);
    }
    if (tensor) {
      // Zero the padding rows the tensor cores read: gate rows past E, token rows past ntok.
      for (int idx = t; idx < (epad - E) * rowv; idx += kThreads)
        sm_wg[(E + idx / rowv) * pstride + idx % rowv] = make_uint4(0, 0, 0, 0);
      for (int idx = t; idx < (TB - ntok) * rowv; idx += kThreads)
        sm_x[(ntok + idx / rowv) * pstride + idx % rowv] = make_uint4(0, 0, 0, 0);
    }
    if (!mbar_wait_for(bar, 0, 1000000000ull) && t == 0) report_status(a.status, kStatusWaitTimeout, 500);
    if (tensor) __syncthreads();
    if (stage_wg) {
      wsrc = sm_wg;
      wstride = pstride;
    }
    if (stage_x) xsrc = sm_x + tok * pstride;
  }
  float z[EPL];
#pragma unroll
  for (int j = 0; j < EPL; ++j) z[j] = 0.f;
  if constexpr (kTensor) {
    if (tensor) {
      constexpr int NW = NT / 32, TOKG = TB / 16, WPG = NW / TOKG;
      const int warp = t >> 5, lane = t & 31;
      const int ntile = epad / 8, ldw = pstride * 8;  // row stride in bf16
      const int tg = warp / WPG;
      const __nv_bfloat16* xb = reinterpret_cast<const __nv_bfloat16*>(sm_x);
      const __nv_bfloat16* wb = reinterpret_cast<const __nv_bfloat16*>(sm_wg);
      const uint32_t a_addr = smem_u32(xb + (tg * 16 + (lane & 15)) * ldw + (lane >> 4) * 8);
      const int bl = lane & 15;
      if constexpr (kAlias) {
        // Every warp's n-tiles stay in registers until all warps are done
        // reading the gate rows; then the table overwrites them.
        constexpr int NTW = (kMaxExperts / 8 + WPG - 1) / WPG;
        float acc[NTW][4];
#pragma unroll
        for (int q = 0; q < NTW; ++q) {
          acc[q][0] = acc[q][1] = acc[q][2] = acc[q][3] = 0.f;
          const int nt = warp % WPG + q * WPG;
          if (nt < ntile) {
            const uint32_t b_addr = smem_u32(wb + (nt * 8 + (bl & 7)) * ldw + (bl >> 3) * 8);
            for (int k0 = 0; k0 < a.D; k0 += 16) {
              uint32_t a0, a1, a2, a3, b0, b1;
              ldsm_x4(a_addr + k0 * 2, a0, a1, a2, a3);
              ldsm_x2(b_addr + k0 * 2, b0, b1);
              mma_16816(acc[q], a0, a1, a2, a3, b0, b1);
            }
          }
        }
        __syncthreads();
#pragma unroll
        for (int q = 0; q < NTW; ++q) {
          const int nt = warp % WPG + q * WPG;
          if (nt < ntile) {
            const int r0 = tg * 16 + (lane >> 2), e0 = nt * 8 + (lane & 3) * 2;
            sm_logit[r0 * (epad + 1) + e0] = acc[q][0];
            sm_logit[r0 * (epad + 1) + e0 + 1] = acc[q][1];
            sm_logit[(r0 + 8) * (epad + 1) + e0] = acc[q][2];
            sm_logit[(r0 + 8) * (epad + 1) + e0 + 1] = acc[q][3];
          }
        }
      } else {
        for (int nt = warp % WPG; nt < ntile; nt += WPG) {
          float acc[4] = {0.f, 0.f, 0.f, 0.f};
          const uint32_t b_addr = smem_u32(wb + (nt * 8 + (bl & 7)) * ldw + (bl >> 3) * 8);
          for (int k0 = 0; k0 < a.D; k0 += 16) {
            uint32_t a0, a1, a2, a3, b0, b1;
            ldsm_x4(a_addr + k0 * 2, a0, a1, a2, a3);
            ldsm_x2(b_addr + k0 * 2, b0, b1);
            mma_16816(acc, a0, a1, a2, a3, b0, b1);
          }
          const int r0 = tg * 16 + (lane >> 2), e0 = nt * 8 + (lane & 3) * 2;
          sm_logit[r0 * (epad + 1) + e0] = acc[0];
          sm_logit[r0 * (epad + 1) + e0 + 1] = acc[1];
          sm_logit[(r0 + 8) * (epad + 1) + e0] = acc[2];
          sm_logit[(r0 + 8) * (epad + 1) + e0 + 1] = acc[3];
        }
      }
      __syncthreads();
#pragma unroll
      for (int j = 0; j < EPL; ++j) {
        const int e = g + G * j;
        if (e < E) z[j] = sm_logit[tok * (epad + 1) + e];
      }
    }
  }
  if (valid && !tensor) {
#pragma unroll 2
    for (int c = 0; c < rowv; ++c) {
      float xv[V];
      unpack_vec(xsrc[c], xv, static_cast<TI*>(nullptr));
#pragma unroll
      for (int j = 0; j < EPL; ++j) {
        const int e = g + G * j;
        if (e < E) {
          float wv[V];
          unpack_vec(wsrc[e * wstride + c], wv, static_cast<TI*>(nullptr));
#pragma unroll
          for (int q = 0; q < V; ++q) z[j] = fmaf(xv[q], wv[q], z[j]);
        }
      }
    }
  }
// Logits of experts this lane does not own (e >= E) are -inf.
  float zl[EPL];
  float lmax = -INFINITY, labs = 0.f;
#pragma unroll
  for (int j = 0; j < EPL; ++j) {
    const int e = g + G * j;
    if (e < E) {
      zl[j] = z[j] + bias_pre[j];
      lmax = fmaxf(lmax, zl[j]);
      labs = fmaxf(labs, fabsf(zl[j]));
    } else {
      zl[j] = -INFINITY;
    }
  }
  const float m = group_max<G>(lmax);
  const float zabs = group_max<G>(labs);
  float lsum = 0.f;
#pragma unroll
  for (int j = 0; j < EPL; ++j)
    if (g + G * j < E) lsum += expf(zl[j] - m);
  const float denom = group_sum<G>(lsum);
  // Top-(k+1): repeated group argmax, ties to the lower expert id.
  const int ranks = (k + 1 < E) ? k + 1 : E;
  unsigned taken = 0u;
  unsigned long long topk_mask = 0ull;
  int sel_e[kMaxTopK + 1];
  float sel_z[kMaxTopK + 1];
#pragma unroll
  for (int r = 0; r < kMaxTopK + 1; ++r) {
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
    float wsum = 0.f, w[kMaxTopK];
#pragma unroll
    for (int p = 0; p < kMaxTopK; ++p) {
      w[p] = 0.f;
      if (p < k) {
        w[p] = expf(sel_z[p] - m) / denom;
        wsum += w[p];
      }
    }
    bool near = false;
#pragma unroll
    for (int p = 0; p < kMaxTopK; ++p)
      if (p + 1 < ranks && (sel_z[p] - sel_z[p + 1]) < 1e-5f * zabs) near = true;
    if (g == 0 && near) atomicAdd(&sm_near, 1);
#pragma unroll
    for (int p = 0; p < kMaxTopK; ++p) {
      if (p < k && p % G == g) {
        a.route_e[static_cast<size_t>(i) * k + p] = sel_e[p];
        a.route_w[static_cast<size_t>(i) * k + p] = a.renorm ? w[p] / wsum : w[p];
      }
    }
  }
  // EMA statistic (Eq. 10) and this token's entropy terms.
#pragma unroll
  for (int j = 0; j < EPL; ++j) {
    const int e = g + G * j;
    if (e < EMAXB) {
      float c = 0.f, u = 0.f;
      if (valid && e < E) {
        const float ind = ((topk_mask >> e) & 1ull) ? 1.f : 0.f;
        c = a.beta * ema_pre[j] + (1.f - a.beta) * ind;
        a.ema[static_cast<size_t>(i) * E + e] = c;
        if (c > 0.f) u = c * logf(c);
      }
      sm_S[tok * EMAXB + e] = c;
      sm_U[tok * EMAXB + e] = u;
    }
  }
  __syncthreads();
  // Block partials per expert, summed over the block's tokens in token order
  // split into J interleaved runs that are added in run order.
  __shared__ float sm_rs[kThreads][2];
  {
    const int J = kThreads / E;
    const int e = t % E, jr = t / E;
    float S = 0.f, U = 0.f;
    if (jr < J)
      for (int q = jr; q < TB; q += J) {
        S += sm_S[q * EMAXB + e];
        U += sm_U[q * EMAXB + e];
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
      a.partials[(static_cast<size_t>(blockIdx.x) * E + t) * 2 + 0] = Ss;
      a.partials[(static_cast<size_t>(blockIdx.x) * E + t) * 2 + 1] = Us;
    }
  }
  if (t == 0 && sm_near) atomicAdd(a.stats + kStNearRoute, static_cast<unsigned long long>(sm_near));
  // The last block to arrive reduces all partials in block order.
  __threadfence();
  __syncthreads();
  __shared__ unsigned ticket;
  if (t == 0) ticket = atomicAdd(a.done, 1u);
  __syncthreads();
  if (ticket != gridDim.x - 1) return;
  __threadfence();
  // Thread t sums blocks j, j + J, j + 2J, ... of expert e = t % E (J runs per
  // expert, loads independent); the J sums are then added in j order.  fp32
  // throughout: FP64 is slow on this part and the sums need no more.
  __shared__ float sm_H[kMaxExperts];
  __shared__ int sm_live[kMaxExperts];
  __shared__ float sm_lo, sm_hi;
  __shared__ float sm_red[kThreads][2];
  {
    const int J = kThreads / E;
    const int e = t % E, j = t / E;
    float S = 0.f, U = 0.f;
    if (j < J) {
      // 32 loads in flight per thread, then added in block order.
      const float2* part = reinterpret_cast<const float2*>(a.partials);
      for (unsigned b0 = j; b0 < gridDim.x; b0 += 32u * J) {
        float2 v[32];
#pragma unroll
        for (int u = 0; u < 32; ++u) {
          const unsigned b = b0 + u * J;
          v[u] = b < gridDim.x ? __ldcg(part + static_cast<size_t>(b) * E + e) : make_float2(0.f, 0.f);
        }
#pragma unroll
        for (int u = 0; u < 32; ++u) {
          S += v[u].x;
          U += v[u].y;
        }
      }
    }
    sm_red[t][0] = S;
    sm_red[t][1] = U;
    __syncthreads();
    if (t < E) {
      float Ss = 0.f, Us = 0.f;
      for (int jj = 0; jj < J; ++jj) {
        Ss += sm_red[jj * E + t][0];
        Us += sm_red[jj * E + t][1];
      }
      sm_live[t] = Ss > 0.f;
      sm_H[t] = Ss > 0.f ? logf(Ss) - Us / Ss : 0.f;
    }
  }
  __syncthreads();
  if (t < 32) {
    // Range of the live experts' entropies (min and max are exact in any order).
    float lo = INFINITY, hi = -INFINITY;
    for (int e = t; e < E; e += 32) {
      if (!sm_live[e]) continue;
      lo = fminf(lo, sm_H[e]);
      hi = fmaxf(hi, sm_H[e]);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, o));
      hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, o));
    }
    if (t == 0) {
      const bool any = lo <= hi;
      sm_lo = any ? lo : 0.f;
      sm_hi = any ? hi : 0.f;
      *a.done = 0u;
    }
  }
  __syncthreads();
  if (t < E) {
    float hb = 0.5f;
    if (sm_live[t]) {
      if (a.entropy_norm == 0) {
        if (a.T > 1) hb = fminf(1.f, fmaxf(0.f, sm_H[t] / logf(static_cast<float>(a.T))));
      } else if (sm_hi > sm_lo) {
        hb = (sm_H[t] - sm_lo) / (sm_hi - sm_lo);
      }
    }
    a.tau[t] = a.tau0 * (1.0f + a.alpha * (2.0f * hb - 1.0f));
  }
}

// The padded gate matrix, and the block's token rows when they also fit, go
// to shared memory; otherwise lanes read them through L1 / L2.  The staging
// cap is what the 227 KB per-block limit leaves beside the kernel's static
// shared memory.
constexpr size_t kSmemPerBlock = 227 * 1024;

template <typename TI, int G, int EPL, int NT>
cudaError_t launch_g(const RouterArgs& a, cudaStream_t s) {
  constexpr int TB = NT / G;
  constexpr bool kAlias = std::is_same_v<TI, __nv_bfloat16> && NT == 256;
  // The staging cap depends on the kernel's static shared memory only; the
  // attribute that allows it is set on every device the process uses.
  cudaFuncAttributes attr;
  cudaError_t e = cudaFuncGetAttributes(&attr, router_kernel<TI, G, EPL, NT>);
  if (e != cudaSuccess) return e;
  const size_t cap = kSmemPerBlock - attr.sharedSizeBytes - 1024;
  e = set_dyn_smem_on_device(reinterpret_cast<const void*>(router_kernel<TI, G, EPL, NT>), static_cast<int>(cap));
  if (e != cudaSuccess) return e;
  const int grid = (a.T + TB - 1) / TB;
  const size_t row = static_cast<size_t>(a.D / Elem<TI>::kVec + 1) * 16;
  const size_t epad = (a.E + 7) / 8 * 8;
  const size_t wg_bytes = epad * row, x_bytes = TB * row, logit_bytes = TB * (epad + 1) * 4;
  if constexpr (kAlias) {
    // The logit table and the entropy terms must fit in the gate rows' space,
    // and both the gate rows and the token rows must be staged.
    const size_t alias_bytes = logit_bytes + 2 * static_cast<size_t>(TB) * G * EPL * 4;
    if (wg_bytes + x_bytes > cap || alias_bytes > wg_bytes) return cudaErrorNotSupported;
    return launch_pdl(router_kernel<TI, G, EPL, NT>, dim3(grid), dim3(NT), wg_bytes + x_bytes, s, a, 1, 1);
  }
  const int stage_wg = wg_bytes <= cap;
  const int stage_x = stage_wg && wg_bytes + x_bytes + logit_bytes <= cap;
  const size_t smem = (stage_wg ? wg_bytes : 0) + (stage_x ? x_bytes + logit_bytes : 0);
  return launch_pdl(router_kernel<TI, G, EPL, NT>, dim3(grid), dim3(NT), smem, s, a, stage_x, stage_wg);
}

template <typename TI>
cudaError_t launch_t(const RouterArgs& a, cudaStream_t s) {
  const int E = a.E;
  if (E == 1) return launch_g<TI, 1, 1, 128>(a, s);
  if (E <= 3) return launch_g<TI, 2, 2, 128>(a, s);
  if (E <= 7) return launch_g<TI, 4, 2, 128>(a, s);
  if (E <= 8) return launch_g<TI, 8, 1, 128>(a, s);
  if (E <= 16) return launch_g<TI, 8, 2, 128>(a, s);
  // 16 tokens per block for wide gates, so the token rows and the logit
  // table fit beside the staged gate matrix (the tensor-core path).
  if (E <= 32) return launch_g<TI, 8, 4, 128>(a, s);
  if constexpr (std::is_same_v<TI, __nv_bfloat16>) {
    // 32-token blocks (one wave of 128 blocks at 4096 tokens) when the gate
    // matrix and the token rows fit in shared memory together.
    const cudaError_t e = launch_g<TI, 8, 8, 256>(a, s);
    if (e != cudaErrorNotSupported) return e;
  }
  return launch_g<TI, 8, 8, 128>(a, s);
}

}  // namespace

cudaError_t launch_router(const RouterArgs& a, bool bf16, cudaStream_t s) {
  return bf16 ? launch_t<__nv_bfloat16>(a, s) : launch_t<float>(a, s);
}

}  // namespace moeca

// ---------------------------------------------------------------------------
// Allocation-free router call (moeca_route_noalloc).
//
// For callers that may not allocate device memory.  The router kernel above
// needs scratch for its per-block entropy partial sums, its last-block ticket
// and a near-tie counter; here that scratch is one array compiled into the
// library instead of a workspace from moeca_create.  Host code must not pass
// g_route_scratch itself to a kernel (on the host that name is only a stand-in
// for the device array): its device address, per device, comes from
// cudaGetSymbolAddress on the first call made with that device current.
// ---------------------------------------------------------------------------
namespace moeca {
namespace {

constexpr size_t kScratchHeader = 256;      // ticket at 0, counters at 64
constexpr size_t kScratchPartials = 32768;  // float2 (sum C, sum C ln C) per (block, expert)
constexpr size_t kScratchBytes = kScratchHeader + kScratchPartials * sizeof(float2);
constexpr int kScratchDevices = 64;

static __device__ __align__(256) unsigned char g_route_scratch[kScratchBytes];

std::mutex g_scratch_mu;
void* g_scratch_addr[kScratchDevices] = {};

}  // namespace

}  // namespace moeca

extern "C" moeca_status moeca_route_noalloc(const moeca_route_args* r, void* stream) {
  using namespace moeca;
  if (!r || !r->x || !r->w_gate || !r->ema || !r->route_e || !r->route_w || !r->tau) return MOECA_ERR_INVALID_ARG;
  const bool bf16 = r->dtype == MOECA_BF16;
  if (r->dtype != MOECA_BF16 && r->dtype != MOECA_F32) return MOECA_ERR_INVALID_ARG;
  if (r->n_tokens < 1 || r->hidden < 1 || r->hidden % (bf16 ? 8 : 4) || r->n_experts < 1 ||
      r->n_experts > kMaxExperts || r->top_k < 1 || r->top_k > kMaxTopK || r->top_k > r->n_experts)
    return MOECA_ERR_INVALID_ARG;
  if (!(r->beta >= 0.f && r->beta < 1.f) || !(r->alpha >= 0.f && r->alpha < 1.f) || r->tau0 != r->tau0)
    return MOECA_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(r->x) % 16 || reinterpret_cast<uintptr_t>(r->w_gate) % 16)
    return MOECA_ERR_INVALID_ARG;
  const size_t blocks = (static_cast<size_t>(r->n_tokens) + kRouterTokensPerBlock - 1) / kRouterTokensPerBlock;
  if (blocks * static_cast<size_t>(r->n_experts) > kScratchPartials) return MOECA_ERR_UNSUPPORTED;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return MOECA_ERR_CUDA;
  }
  if (dev < 0 || dev >= kScratchDevices) return MOECA_ERR_UNSUPPORTED;
  void* base = nullptr;
  {
    std::lock_guard<std::mutex> lock(g_scratch_mu);
    if (!g_scratch_addr[dev]) {
      void* p = nullptr;
      if (cudaGetSymbolAddress(&p, g_route_scratch) != cudaSuccess || !p) {
        cudaGetLastError();
        return MOECA_ERR_CUDA;
      }
      g_scratch_addr[dev] = p;
    }
    base = g_scratch_addr[dev];
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // The ticket and the counters must start at zero; the partials are written
  // by every block before the last block reads them.
  if (cudaMemsetAsync(base, 0, kScratchHeader, s) != cudaSuccess) {
    cudaGetLastError();
    return MOECA_ERR_CUDA;
  }
  RouterArgs a{};
  a.x = r->x;
  a.w_gate = r->w_gate;
  a.b_gate = r->b_gate;
  a.T = r->n_tokens;
  a.D = r->hidden;
  a.E = r->n_experts;
  a.k = r->top_k;
  a.renorm = r->renorm_topk;
  a.beta = r->beta;
  a.tau0 = r->tau0;
  a.alpha = r->alpha;
  a.entropy_norm = r->entropy_norm;
  a.route_e = r->route_e;
  a.route_w = r->route_w;
  a.ema = r->ema;
  a.partials = reinterpret_cast<float*>(static_cast<unsigned char*>(base) + kScratchHeader);
  a.done = static_cast<unsigned*>(base);
  a.tau = r->tau;
  a.stats = reinterpret_cast<unsigned long long*>(static_cast<unsigned char*>(base) + 64);
  if (launch_router(a, bf16, s) != cudaSuccess) {
    cudaGetLastError();
    return MOECA_ERR_CUDA;
  }
  return MOECA_OK;
}
