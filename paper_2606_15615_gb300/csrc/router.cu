// Router of the branch-cached MoE layer.
//
// Per token i (one warp): gate logits z = x_i W_g^T (+ b) with fp32
// accumulation, softmax over the E experts, top-k by descending logit with
// ties to the lower expert id, optional renormalisation of the k weights
// (Eq. 7).  The same pass updates the EMA statistic
//   C_{e,i} <- beta C_{e,i} + (1 - beta) 1[e in B_i]        (Eq. 10)
// and accumulates per block S_e = sum_i C_{e,i} and U_e = sum_i C ln C, from
// which the last block to finish derives the spatial entropy
//   H_e = ln S_e - U_e / S_e  (= -sum_i P ln P with P = C / S, Eq. 11),
// its normalisation and the expert threshold tau_e (Eq. 12).
#include <mutex>

#include "common.cuh"
#include "kernels.h"
#include "moeca.h"

namespace moeca {
namespace {

constexpr int kWarps = 8;
constexpr int kTokensPerWarp = kRouterTokensPerBlock / kWarps;

template <typename TI, int EMAX>
__global__ void __launch_bounds__(kWarps * 32) router_kernel(RouterArgs a) {
  constexpr int V = Elem<TI>::kVec;
  constexpr int EPL = (EMAX + 31) / 32;  // EMA experts per lane
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const TI* __restrict__ x = static_cast<const TI*>(a.x);
  const TI* __restrict__ wg = static_cast<const TI*>(a.w_gate);
  const int E = a.E, k = a.k, nvec = a.D / V;

  __shared__ float sm_S[kWarps][EMAX];
  __shared__ float sm_U[kWarps][EMAX];
  __shared__ int sm_near[kWarps];

  float accS[EPL], accU[EPL];
#pragma unroll
  for (int j = 0; j < EPL; ++j) accS[j] = accU[j] = 0.f;
  int near_count = 0;

  for (int tt = 0; tt < kTokensPerWarp; ++tt) {
    const int i = blockIdx.x * kRouterTokensPerBlock + warp * kTokensPerWarp + tt;
    if (i >= a.T) break;  // warp-uniform
    float z[EMAX];
#pragma unroll
    for (int e = 0; e < EMAX; ++e) z[e] = 0.f;
    const TI* xr = x + static_cast<size_t>(i) * a.D;
    for (int c = lane; c < nvec; c += 32) {
      float xv[V];
      load_vec(xr + c * V, xv);
#pragma unroll
      for (int e = 0; e < EMAX; ++e) {
        if (e < E) {
          float wv[V];
          load_vec(wg + static_cast<size_t>(e) * a.D + c * V, wv);
#pragma unroll
          for (int j = 0; j < V; ++j) z[e] = fmaf(xv[j], wv[j], z[e]);
        }
      }
    }
#pragma unroll
    for (int e = 0; e < EMAX; ++e) {
      if (e < E) {
        z[e] = warp_sum(z[e]);
        if (a.b_gate) z[e] += a.b_gate[e];
      }
    }
    // Top-(k+1) by repeated argmax (every lane holds every logit).
    unsigned long long taken = 0ull, topk_mask = 0ull;
    int sel[kMaxTopK];
    float selz[kMaxTopK + 1];
    const int ranks = (k + 1 < E) ? k + 1 : E;
    float zabs = 0.f;
#pragma unroll
    for (int e = 0; e < EMAX; ++e)
      if (e < E) zabs = fmaxf(zabs, fabsf(z[e]));
#pragma unroll
    for (int p = 0; p < kMaxTopK + 1; ++p) {
      if (p < ranks) {
        int be = -1;
        float best = 0.f;
#pragma unroll
        for (int e = 0; e < EMAX; ++e) {
          if (e < E && !((taken >> e) & 1ull) && (be < 0 || z[e] > best)) {
            best = z[e];
            be = e;
          }
        }
        taken |= 1ull << be;
        selz[p] = best;
        if (p < k) {
          sel[p] = be;
          topk_mask |= 1ull << be;
        }
      }
    }
    // Softmax over all E from the top logit, then the k weights.
    const float m = selz[0];
    float denom = 0.f;
#pragma unroll
    for (int e = 0; e < EMAX; ++e)
      if (e < E) denom += expf(z[e] - m);
    float w[kMaxTopK];
    float wsum = 0.f;
#pragma unroll
    for (int p = 0; p < kMaxTopK; ++p) {
      if (p < k) {
        w[p] = expf(selz[p] - m) / denom;
        wsum += w[p];
      }
    }
    bool near = false;
#pragma unroll
    for (int p = 0; p < kMaxTopK; ++p)
      if (p + 1 < ranks && (selz[p] - selz[p + 1]) < 1e-5f * zabs) near = true;
    if (lane == 0 && near) ++near_count;
#pragma unroll
    for (int p = 0; p < kMaxTopK; ++p) {
      if (p < k && lane == p) {
        a.route_e[static_cast<size_t>(i) * k + p] = sel[p];
        a.route_w[static_cast<size_t>(i) * k + p] = a.renorm ? w[p] / wsum : w[p];
      }
    }
    // EMA statistic and entropy partial sums.
#pragma unroll
    for (int j = 0; j < EPL; ++j) {
      const int e = lane + 32 * j;
      if (e < E) {
        float* cp = a.ema + static_cast<size_t>(i) * E + e;
        const float ind = ((topk_mask >> e) & 1ull) ? 1.f : 0.f;
        const float c = a.beta * (*cp) + (1.f - a.beta) * ind;
        *cp = c;
        accS[j] += c;
        if (c > 0.f) accU[j] += c * logf(c);
      }
    }
  }
#pragma unroll
  for (int j = 0; j < EPL; ++j) {
    const int e = lane + 32 * j;
    if (e < EMAX) {
      sm_S[warp][e] = accS[j];
      sm_U[warp][e] = accU[j];
    }
  }
  if (lane == 0) sm_near[warp] = near_count;
  __syncthreads();
  const int t = threadIdx.x;
  if (t < E) {
    float S = 0.f, U = 0.f;
#pragma unroll
    for (int w8 = 0; w8 < kWarps; ++w8) {
      S += sm_S[w8][t];
      U += sm_U[w8][t];
    }
    a.partials[(static_cast<size_t>(blockIdx.x) * E + t) * 2 + 0] = S;
    a.partials[(static_cast<size_t>(blockIdx.x) * E + t) * 2 + 1] = U;
  }
  if (t == 0) {
    int n = 0;
    for (int w8 = 0; w8 < kWarps; ++w8) n += sm_near[w8];
    if (n) atomicAdd(a.stats + kStNearRoute, static_cast<unsigned long long>(n));
  }
  // The last block to arrive reduces all partials in block order.
  __threadfence();
  __syncthreads();
  __shared__ unsigned ticket;
  if (t == 0) ticket = atomicAdd(a.done, 1u);
  __syncthreads();
  if (ticket != gridDim.x - 1) return;
  __threadfence();
  // Thread t sums blocks j, j + J, j + 2J, ... of expert e = t % E (J = 256 / E
  // lanes per expert, loads independent); the J sums are then added in j order.
  __shared__ double sm_H[EMAX];
  __shared__ int sm_live[EMAX];
  __shared__ double sm_lo, sm_hi;
  __shared__ double sm_red[kWarps * 32][2];
  {
    const int J = (kWarps * 32) / E;
    const int e = t % E, j = t / E;
    double S = 0.0, U = 0.0;
    if (j < J) {
      const float2* part = reinterpret_cast<const float2*>(a.partials);
#pragma unroll 4
      for (unsigned b = j; b < gridDim.x; b += J) {
        const float2 v = __ldcg(part + static_cast<size_t>(b) * E + e);
        S += static_cast<double>(v.x);
        U += static_cast<double>(v.y);
      }
    }
    sm_red[t][0] = S;
    sm_red[t][1] = U;
    __syncthreads();
    if (t < E) {
      double Ss = 0.0, Us = 0.0;
      for (int jj = 0; jj < J; ++jj) {
        Ss += sm_red[jj * E + t][0];
        Us += sm_red[jj * E + t][1];
      }
      sm_live[t] = Ss > 0.0;
      sm_H[t] = Ss > 0.0 ? log(Ss) - Us / Ss : 0.0;
    }
  }
  __syncthreads();
  if (t == 0) {
    double lo = 0.0, hi = 0.0;
    bool any = false;
    for (int e = 0; e < E; ++e) {
      if (!sm_live[e]) continue;
      if (!any || sm_H[e] < lo) lo = sm_H[e];
      if (!any || sm_H[e] > hi) hi = sm_H[e];
      any = true;
    }
    sm_lo = lo;
    sm_hi = hi;
    *a.done = 0u;
  }
  __syncthreads();
  if (t < E) {
    double hb = 0.5;
    if (sm_live[t]) {
      if (a.entropy_norm == 0) {
        if (a.T > 1) hb = fmin(1.0, fmax(0.0, sm_H[t] / log(static_cast<double>(a.T))));
      } else if (sm_hi > sm_lo) {
        hb = (sm_H[t] - sm_lo) / (sm_hi - sm_lo);
      }
    }
    a.tau[t] = a.tau0 * (1.0f + a.alpha * (2.0f * static_cast<float>(hb) - 1.0f));
  }
}

template <typename TI>
cudaError_t launch_t(const RouterArgs& a, cudaStream_t s) {
  const int grid = (a.T + kRouterTokensPerBlock - 1) / kRouterTokensPerBlock;
  const dim3 block(kWarps * 32);
  if (a.E <= 8) router_kernel<TI, 8><<<grid, block, 0, s>>>(a);
  else if (a.E <= 16) router_kernel<TI, 16><<<grid, block, 0, s>>>(a);
  else if (a.E <= 32) router_kernel<TI, 32><<<grid, block, 0, s>>>(a);
  else router_kernel<TI, 64><<<grid, block, 0, s>>>(a);
  return cudaGetLastError();
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
