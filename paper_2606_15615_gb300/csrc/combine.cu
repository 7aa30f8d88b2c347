// Combine of fresh and cached branch outputs (Eq. 8) with the residual of
// Eq. 5 / Eq. 6, and the cached-norm refresh that Eq. 9's o reads next step.
//
// Two forms: a direct one (combine_kernel, the default: one warp per token,
// 16-byte vectors over D) and a staged one (combine_staged_kernel, below):
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
// shared row and x loaded before any arithmetic).  MINB is the launch's
// minimum of resident blocks per SM (see direct_min_blocks).
template <typename TI, int KMAX, int CG, bool GATED, bool YC, int MINB>
__global__ void __launch_bounds__(kWarps * 32, MINB) combine_kernel(CombineArgs a) {
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
  // A token whose branches are all reused (its shared row too) reads nothing
  // the grouped GEMM before this kernel writes, so it does not wait for it.
  if (!(a.early && !a.token_any[i])) pdl_entry();
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

// Staged form: each warp walks its tokens i = w, w + W, ...
// (w its global warp index, W the grid's warps) and stages a token's rows in
// shared memory with bulk copies, lane 0 issuing them onto one mbarrier per
// buffer: the token's k cache rows (one contiguous [k, D] block; slot is a
// permutation of 0..k-1, so these are all the rows Eq. 8 and the norms read),
// its shared-expert row and its residual row.  Two buffers per warp: the next
// token's rows are in flight while this one is combined, so every warp keeps
// a whole token's bytes in flight and no lane waits on more than one round
// trip per token.  Arithmetic and its order are those of combine_kernel.
constexpr int kStagedWarps = 4;

template <typename TI>
__host__ __device__ inline size_t staged_buf_bytes(int k, int n_shared, int D) {
  return (static_cast<size_t>(k + n_shared + 1) * D * sizeof(TI) + 127) / 128 * 128;
}

template <typename TI, int KMAX, bool GATED>
__global__ void __launch_bounds__(kStagedWarps * 32) combine_staged_kernel(CombineArgs a) {
  constexpr int V = Elem<TI>::kVec;
  extern __shared__ __align__(128) uint8_t dyn[];
  __shared__ __align__(8) uint64_t bars[kStagedWarps][2];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int k = a.k, D = a.D, nvec = D / V, T = a.T;
  const bool has_sh = a.shared_h != nullptr;
  const size_t row_bytes = static_cast<size_t>(D) * sizeof(TI);
  const size_t buf_bytes = staged_buf_bytes<TI>(k, has_sh ? 1 : 0, D);
  uint8_t* wbuf = dyn + static_cast<size_t>(warp) * 2 * buf_bytes;
  const uint32_t bar0 = smem_u32(&bars[warp][0]), bar1 = smem_u32(&bars[warp][1]);
  const int nw = gridDim.x * kStagedWarps;
  int i = blockIdx.x * kStagedWarps + warp;
  if (lane == 0) {
    mbar_init(bar0, 1);
    mbar_init(bar1, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncwarp();
  const TI* ch = static_cast<const TI*>(a.cache_h);
  const TI* sh = static_cast<const TI*>(a.shared_h);
  const TI* xin = static_cast<const TI*>(a.x);
  const uint32_t tx = static_cast<uint32_t>(row_bytes) * (k + (has_sh ? 1 : 0) + 1);
  // Lane 0 stages token t into buffer b; the residual row (an earlier
  // kernel's output) may go before the dependency wait, the cache and shared
  // rows (the previous kernel's output) only after it.
  auto issue_rows = [&](int t, int b) {
    const uint32_t dst = smem_u32(wbuf + b * buf_bytes), bar = b ? bar1 : bar0;
    bulk_g2s(dst, ch + static_cast<size_t>(t) * k * D, static_cast<uint32_t>(row_bytes) * k, bar);
    if (has_sh) bulk_g2s(dst + static_cast<uint32_t>(row_bytes) * k, sh + static_cast<size_t>(t) * D,
                         static_cast<uint32_t>(row_bytes), bar);
  };
  auto issue_x = [&](int t, int b) {
    const uint32_t dst = smem_u32(wbuf + b * buf_bytes), bar = b ? bar1 : bar0;
    mbar_expect_tx(bar, tx);
    bulk_g2s(dst + static_cast<uint32_t>(row_bytes) * (k + (has_sh ? 1 : 0)), xin + static_cast<size_t>(t) * D,
             static_cast<uint32_t>(row_bytes), bar);
  };
  if (lane == 0 && i < T) issue_x(i, 0);
  pdl_entry();
  if (a.rearm && blockIdx.x == 0 && threadIdx.x == 0) *a.rearm = 0;  // the grouped GEMM before has ended
  if (lane == 0 && i < T) issue_rows(i, 0);
  uint32_t phase = 0u;  // bit b: parity of buffer b's next completion
  for (int b = 0; i < T; i += nw, b ^= 1) {
    const int nx = i + nw;
    if (lane == 0 && nx < T) {
      issue_x(nx, b ^ 1);
      issue_rows(nx, b ^ 1);
    }
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
    const bool ok = mbar_wait_for(b ? bar1 : bar0, (phase >> b) & 1u, 1000000000ull);
    phase ^= 1u << b;
    if (!ok) {
      // The copies never completed: record it, let the next token's copies
      // (if issued) land before this warp leaves its shared memory, stop.
      if (lane == 0) {
        report_status(a.status, kStatusWaitTimeout, 3100000 + i);
        if (nx < T) mbar_wait_for(b ? bar0 : bar1, (phase >> (b ^ 1)) & 1u, 1000000000ull);
      }
      __syncwarp();
      return;
    }
    if (bad) {
      if (lane == 0) report_status(a.status, kStatusBadIndex, 3000000 + i);
      __syncwarp();
      continue;
    }
    const uint8_t* buf = wbuf + b * buf_bytes;
    const uint4* hrow = reinterpret_cast<const uint4*>(buf);
    const uint4* srow = reinterpret_cast<const uint4*>(buf + row_bytes * k);
    const uint4* xrow = reinterpret_cast<const uint4*>(buf + row_bytes * (k + (has_sh ? 1 : 0)));
    const float* gr = GATED ? a.gate + static_cast<size_t>(i / a.seq) * a.gate_ld : nullptr;
    TI* out = static_cast<TI*>(a.out) + static_cast<size_t>(i) * D;
    float ss[KMAX];
#pragma unroll
    for (int p = 0; p < KMAX; ++p) ss[p] = 0.f;
    for (int c = lane; c < nvec; c += 32) {
      float y[V];
#pragma unroll
      for (int j = 0; j < V; ++j) y[j] = 0.f;
#pragma unroll
      for (int p = 0; p < KMAX; ++p) {
        if (p < k) {
          float hv[V];
          unpack_vec(hrow[static_cast<size_t>(q[p]) * nvec + c], hv, static_cast<TI*>(nullptr));
#pragma unroll
          for (int j = 0; j < V; ++j) {
            y[j] = fmaf(w[p], hv[j], y[j]);
            ss[p] = fmaf(hv[j], hv[j], ss[p]);
          }
        }
      }
      if (has_sh) {
        float hv[V];
        unpack_vec(srow[c], hv, static_cast<TI*>(nullptr));
#pragma unroll
        for (int j = 0; j < V; ++j) y[j] += hv[j];
      }
      float xs[V];
      unpack_vec(xrow[c], xs, static_cast<TI*>(nullptr));
      if constexpr (GATED) {
        float gv[V];
#pragma unroll
        for (int j = 0; j < V / 4; ++j) {
          const float4 g4 = __ldg(reinterpret_cast<const float4*>(gr + c * V) + j);
          gv[4 * j] = g4.x; gv[4 * j + 1] = g4.y; gv[4 * j + 2] = g4.z; gv[4 * j + 3] = g4.w;
        }
#pragma unroll
        for (int j = 0; j < V; ++j) xs[j] = fmaf(gv[j], y[j], xs[j]);
      } else {
#pragma unroll
        for (int j = 0; j < V; ++j) xs[j] += y[j];
      }
      store_vec(out + c * V, xs);
    }
#pragma unroll
    for (int p = 0; p < KMAX; ++p) {
      if (p < k) {
        const float s2 = warp_sum(ss[p]);
        if (lane == 0) a.cache_norm[static_cast<size_t>(i) * k + q[p]] = sqrtf(s2);
      }
    }
    __syncwarp();  // every lane is done with buffer b before lane 0 refills it
  }
}

template <typename TI, bool GATED>
cudaError_t launch_staged(const CombineArgs& a, cudaStream_t s) {
  const size_t smem = static_cast<size_t>(kStagedWarps) * 2 * staged_buf_bytes<TI>(a.k, a.shared_h ? 1 : 0, a.D);
  auto run = [&](auto kern) -> cudaError_t {
    cudaError_t e = set_dyn_smem_on_device(reinterpret_cast<const void*>(kern), static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    int per_sm = 0;
    if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kStagedWarps * 32, smem)) != cudaSuccess)
      return e;
    long long grid = (a.T + kStagedWarps - 1) / kStagedWarps;
    const long long cap = static_cast<long long>(a.n_sms > 0 ? a.n_sms : 1) * (per_sm > 0 ? per_sm : 1);
    if (grid > cap) grid = cap;
    return launch_pdl(kern, dim3(static_cast<unsigned>(grid)), dim3(kStagedWarps * 32), smem, s, a);
  };
  if (a.k <= 2) return run(combine_staged_kernel<TI, 2, GATED>);
  if (a.k <= 4) return run(combine_staged_kernel<TI, 4, GATED>);
  return run(combine_staged_kernel<TI, 8, GATED>);
}

// Resident blocks per SM that the direct form asks of the compiler, with one
// 16-byte chunk per row and lane in flight.  Top-2 tokens fit four blocks
// (64 registers a thread): every token of a 4096-token batch is then in
// flight at once, which measured 37.5 -> 20.8 us per launch at D 2560 with a
// shared expert against two blocks with four chunks in flight.  Top-4 takes
// three, top-8 two (with the AdaLN gate values one block fewer, and fp32 top-8
// one): under a tighter cap the compiler spills, or moves row loads next to
// their use, one round trip each (top-8 at D 1152: 25 us per launch with two
// blocks, 30 to 60 us with three in the spill-free variants tried).
template <typename TI, int KMAX, bool GATED>
constexpr int direct_min_blocks() {
  return KMAX <= 2 ? (GATED ? 3 : 4) : KMAX <= 4 ? (GATED ? 2 : 3) : sizeof(TI) == 4 ? 1 : 2;
}

template <typename TI, bool GATED, bool YC>
void launch_t(const CombineArgs& a, cudaStream_t s) {
  const int grid = (a.T + kWarps - 1) / kWarps;
  if (a.k <= 2)
    launch_pdl(combine_kernel<TI, 2, 1, GATED, YC, direct_min_blocks<TI, 2, GATED>()>, dim3(grid), dim3(kWarps * 32), 0, s, a);
  else if (a.k <= 4)
    launch_pdl(combine_kernel<TI, 4, 1, GATED, YC, direct_min_blocks<TI, 4, GATED>()>, dim3(grid), dim3(kWarps * 32), 0, s, a);
  else
    launch_pdl(combine_kernel<TI, 8, 1, GATED, YC, direct_min_blocks<TI, 8, GATED>()>, dim3(grid), dim3(kWarps * 32), 0, s, a);
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
  if (a.T <= 0) return cudaSuccess;
  // The direct form by default: inside the launch pipeline it measured the
  // shorter step (12-layer D 768: 0.7785 -> 0.774 ms; 28-layer D 1152: 4.150
  // -> 4.108 ms) although the staged form is the faster launch when timed
  // alone at D 768 (8.5 vs 10.4 us).  The staged form, on request, while a
  // warp's two buffers take at most 24 KB, so that two blocks (8 warps) fit
  // an SM: with larger tokens (D 2560 with a shared expert, top-8 at D 1152:
  // about 41 KB a warp) a block of 4 warps per SM measured slower than the
  // direct form (31 vs 26 us, 40 vs 27 us per launch).  The 16-byte alignment
  // of every staged row holds for D a multiple of the vector width.  The
  // token-level reading of Sec. 4.1 (cache_y) keeps the direct form.
  const size_t per_warp = 2 * (bf16 ? staged_buf_bytes<__nv_bfloat16>(a.k, a.shared_h ? 1 : 0, a.D)
                                    : staged_buf_bytes<float>(a.k, a.shared_h ? 1 : 0, a.D));
  if (!a.cache_y && !a.direct && per_warp <= 24 * 1024 && reinterpret_cast<uintptr_t>(a.x) % 16 == 0) {
    if (bf16 && a.gate) return launch_staged<__nv_bfloat16, true>(a, s);
    if (bf16) return launch_staged<__nv_bfloat16, false>(a, s);
    return launch_staged<float, false>(a, s);
  }
  if (a.cache_y) launch_y<true>(a, bf16, s);
  else launch_y<false>(a, bf16, s);
  return cudaGetLastError();
}

}  // namespace moeca
