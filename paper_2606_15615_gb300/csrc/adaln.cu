// AdaLN modulation of a DiT-MoE block (Sec. 3: each sub-layer f enters the
// residual stream as x + AdaLN o f(x)) and the reverse-diffusion update of the
// sampler (Eq. 1).
//
// ada_mod_kernel      the six modulation vectors of every block for every
//                     sample, SiLU(c) W_ada^T + b_ada, all layers in one launch
//                     at the start of a step (HBM-bound: it streams W_ada once)
// adaln_rows_kernel   per token row: layer normalisation over D and the
//                     modulation, the gated attention residual u = x + g a,
//                     and the MoE input m; one warp per row, the row in
//                     registers
// ddpm_kernel         x_{t-1} = (x_t - c1 eps) / sqrt(alpha_t) + sigma_t z
#include "common.cuh"
#include "kernels.h"

namespace moeca {
namespace {

constexpr int kModWarps = 8;
constexpr int kModB = 8;  // samples accumulated per pass over the weight rows
constexpr int kModR = 4;  // weight rows per warp pass: each staged SiLU(c) load feeds kModR rows

__global__ void __launch_bounds__(kModWarps * 32) ada_mod_kernel(AdaModArgs a) {
  extern __shared__ __align__(16) float s_c[];  // [B, D] SiLU(c)
  const int D = a.D, B = a.B;
  // The previous step's last kernels still read `out` (the gates), and the
  // caller may have written cond with a kernel: wait first.
  pdl_entry();
  for (int i = threadIdx.x; i < B * D; i += blockDim.x) {
    const float z = a.cond[i];
    s_c[i] = z / (1.f + expf(-z));
  }
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int per_layer = 6 * D;                   // a multiple of kModR (D is a multiple of 64)
  const long long n_groups = static_cast<long long>(a.L) * (per_layer / kModR);
  const int nvec = D / 8;
  for (long long g = static_cast<long long>(blockIdx.x) * kModWarps + warp; g < n_groups;
       g += static_cast<long long>(gridDim.x) * kModWarps) {
    const long long r0 = g * kModR;              // kModR rows of one layer
    const int l = static_cast<int>(r0 / per_layer);
    const int j0 = static_cast<int>(r0 - static_cast<long long>(l) * per_layer);
    const uint4* wrow = reinterpret_cast<const uint4*>(a.w[l]) + static_cast<size_t>(j0) * nvec;
    const float* bl = a.b[l];
    float* out = a.out + static_cast<size_t>(l) * B * per_layer + j0;
    for (int b0 = 0; b0 < B; b0 += kModB) {
      float acc[kModR][kModB];
#pragma unroll
      for (int r = 0; r < kModR; ++r)
#pragma unroll
        for (int q = 0; q < kModB; ++q) acc[r][q] = 0.f;
#pragma unroll 2
      for (int c = lane; c < nvec; c += 32) {
        float wf[kModR][8];
#pragma unroll
        for (int r = 0; r < kModR; ++r)
          unpack_vec(__ldg(wrow + static_cast<size_t>(r) * nvec + c), wf[r], static_cast<__nv_bfloat16*>(nullptr));
#pragma unroll
        for (int q = 0; q < kModB; ++q) {
          if (b0 + q < B) {
            const float4* cp = reinterpret_cast<const float4*>(s_c + static_cast<size_t>(b0 + q) * D + 8 * c);
            const float4 c0 = cp[0], c1 = cp[1];
            const float cv[8] = {c0.x, c0.y, c0.z, c0.w, c1.x, c1.y, c1.z, c1.w};
#pragma unroll
            for (int r = 0; r < kModR; ++r) {
              float s = acc[r][q];
#pragma unroll
              for (int e = 0; e < 8; ++e) s = fmaf(wf[r][e], cv[e], s);
              acc[r][q] = s;
            }
          }
        }
      }
#pragma unroll
      for (int r = 0; r < kModR; ++r) {
        const float bias = bl ? bl[j0 + r] : 0.f;
#pragma unroll
        for (int q = 0; q < kModB; ++q) {
          const float v = warp_sum(acc[r][q]);
          if (lane == 0 && b0 + q < B) out[static_cast<size_t>(b0 + q) * per_layer + r] = v + bias;
        }
      }
    }
  }
}

constexpr int kLnWarps = 8;
constexpr int kLnChunks = kAdaLnMaxD / 256;  // 16-byte chunks per lane

// Eight floats from global or shared memory (a generic pointer: the row
// pass reads the modulation vectors from either).
__device__ __forceinline__ void load8(const float* p, float* v) {
  const float4 a = reinterpret_cast<const float4*>(p)[0];
  const float4 b = reinterpret_cast<const float4*>(p)[1];
  v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}

__device__ __forceinline__ void load8f(const float* p, float* v) {
  const float4 a = __ldg(reinterpret_cast<const float4*>(p));
  const float4 b = __ldg(reinterpret_cast<const float4*>(p) + 1);
  v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}

// Plain (coherent) loads, for a buffer the same kernel writes: the read-only
// path above requires the data to stay unchanged for the kernel's duration.
__device__ __forceinline__ void load8f_rw(const float* p, float* v) {
  const float4 a = reinterpret_cast<const float4*>(p)[0];
  const float4 b = reinterpret_cast<const float4*>(p)[1];
  v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}

__device__ __forceinline__ uint4 pack8(const float* f) {
  uint4 v;
  __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&v);
#pragma unroll
  for (int q = 0; q < 4; ++q) h[q] = __floats2bfloat162_rn(f[2 * q], f[2 * q + 1]);
  return v;
}

// Mean and 1 / sqrt(var + eps) of the row held as bf16 chunks (chunk c = lane + 32 q),
// two passes over the registers.
__device__ __forceinline__ void row_stats(const uint4* v, int nvec, int lane, int D, float eps, float& mean,
                                          float& rstd) {
  float s = 0.f;
#pragma unroll
  for (int q = 0; q < kLnChunks; ++q) {
    if (lane + 32 * q < nvec) {
      float f[8];
      unpack_vec(v[q], f, static_cast<__nv_bfloat16*>(nullptr));
#pragma unroll
      for (int j = 0; j < 8; ++j) s += f[j];
    }
  }
  mean = warp_sum(s) / static_cast<float>(D);
  float ss = 0.f;
#pragma unroll
  for (int q = 0; q < kLnChunks; ++q) {
    if (lane + 32 * q < nvec) {
      float f[8];
      unpack_vec(v[q], f, static_cast<__nv_bfloat16*>(nullptr));
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const float d = f[j] - mean;
        ss = fmaf(d, d, ss);
      }
    }
  }
  rstd = rsqrtf(warp_sum(ss) / static_cast<float>(D) + eps);
}

// dst = bf16((v - mean) rstd (1 + scale) + shift), chunk by chunk.
__device__ __forceinline__ void store_modulated(const uint4* v, int nvec, int lane, float mean, float rstd,
                                                const float* shift, const float* scale, __nv_bfloat16* dst,
                                                __nv_bfloat16* dst2) {
#pragma unroll
  for (int q = 0; q < kLnChunks; ++q) {
    const int c = lane + 32 * q;
    if (c < nvec) {
      float f[8], sh[8], sc[8];
      unpack_vec(v[q], f, static_cast<__nv_bfloat16*>(nullptr));
      load8(shift + 8 * c, sh);
      load8(scale + 8 * c, sc);
#pragma unroll
      for (int j = 0; j < 8; ++j) f[j] = fmaf((f[j] - mean) * rstd, 1.f + sc[j], sh[j]);
      const uint4 o = pack8(f);
      reinterpret_cast<uint4*>(dst)[c] = o;
      if (dst2) reinterpret_cast<uint4*>(dst2)[c] = o;
    }
  }
}

// With every row (no list), a block's kLnWarps rows are consecutive tokens of
// one sample (seq is a multiple of 8): the block stages that sample's first
// five vectors (shift_a .. scale_m, 5D floats) in shared memory, loaded
// together with the rows.  A listed-row launch reads them from L2 per row.
__global__ void __launch_bounds__(kLnWarps * 32) adaln_rows_kernel(AdaLnArgs a) {
  extern __shared__ __align__(16) float s_mod[];  // [5, D] when staged
  pdl_entry();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int i = blockIdx.x * kLnWarps + warp;
  const int n = a.rows ? *a.n_rows : a.T;
  const bool staged = a.rows == nullptr;
  const int D = a.D, nvec = D / 8;
  int t = -1;
  if (i < n && i < a.T) {
    t = a.rows ? a.rows[i] : i;
    if (t < 0 || t >= a.T) {
      if (lane == 0) report_status(a.status, kStatusBadIndex, 7000000 + i);
      t = -1;
    }
  }
  const size_t off = static_cast<size_t>(t < 0 ? 0 : t) * D;
  uint4 v[kLnChunks], av[kLnChunks];
  const uint4* a4 =
      a.a ? reinterpret_cast<const uint4*>(static_cast<const __nv_bfloat16*>(a.a) + off) : nullptr;
  if (t >= 0 && (a.h_out || a4)) {
    // x and the cached attention row in flight together (and with the staging below).
    const uint4* x4 = reinterpret_cast<const uint4*>(static_cast<const __nv_bfloat16*>(a.x) + off);
#pragma unroll
    for (int q = 0; q < kLnChunks; ++q)
      if (lane + 32 * q < nvec) v[q] = x4[lane + 32 * q];
    if (a4) {
#pragma unroll
      for (int q = 0; q < kLnChunks; ++q)
        if (lane + 32 * q < nvec) av[q] = a4[lane + 32 * q];
    }
  }
  const int row0 = blockIdx.x * kLnWarps;
  if (staged) {
    if (row0 < a.T) {
      const float4* src = reinterpret_cast<const float4*>(a.mod + static_cast<size_t>(row0 / a.seq) * 6 * D);
      for (int j = threadIdx.x; j < 5 * D / 4; j += blockDim.x) reinterpret_cast<float4*>(s_mod)[j] = __ldg(src + j);
    }
    __syncthreads();
  }
  if (t < 0) return;
  // The sample's vectors: shared when the block staged this row's sample, else global.
  const float* md = staged && t / a.seq == row0 / a.seq ? s_mod : a.mod + static_cast<size_t>(t / a.seq) * 6 * D;
  __nv_bfloat16* u = static_cast<__nv_bfloat16*>(a.u) + off;
  float mean, rstd;
  if (a.h_out) {
    row_stats(v, nvec, lane, D, a.eps, mean, rstd);
    store_modulated(v, nvec, lane, mean, rstd, md, md + D, static_cast<__nv_bfloat16*>(a.h_out) + off, nullptr);
  }
  if (a4) {
    // u = bf16(x + gate_a a): one rounding of the fused product-sum.
#pragma unroll
    for (int q = 0; q < kLnChunks; ++q) {
      const int c = lane + 32 * q;
      if (c < nvec) {
        float xf[8], af[8], g[8];
        unpack_vec(v[q], xf, static_cast<__nv_bfloat16*>(nullptr));
        unpack_vec(av[q], af, static_cast<__nv_bfloat16*>(nullptr));
        load8(md + 2 * D + 8 * c, g);
#pragma unroll
        for (int j = 0; j < 8; ++j) xf[j] = fmaf(g[j], af[j], xf[j]);
        v[q] = pack8(xf);
        reinterpret_cast<uint4*>(u)[c] = v[q];
      }
    }
  } else if (a.m_out) {
#pragma unroll
    for (int q = 0; q < kLnChunks; ++q)
      if (lane + 32 * q < nvec) v[q] = reinterpret_cast<const uint4*>(u)[lane + 32 * q];
  }
  if (a.m_out) {
    row_stats(v, nvec, lane, D, a.eps, mean, rstd);
    store_modulated(v, nvec, lane, mean, rstd, md + 3 * D, md + 4 * D,
                    static_cast<__nv_bfloat16*>(a.m_out) + off,
                    a.m_copy ? static_cast<__nv_bfloat16*>(a.m_copy) + off : nullptr);
  }
}

constexpr int kDdpmThreads = 256;

template <bool BF>
__global__ void __launch_bounds__(kDdpmThreads) ddpm_kernel(DdpmArgs a) {
  pdl_entry();
  const long long nv = a.n / 8;
  for (long long c = static_cast<long long>(blockIdx.x) * kDdpmThreads + threadIdx.x; c < nv;
       c += static_cast<long long>(gridDim.x) * kDdpmThreads) {
    float x[8], e[8], z[8];
    load8f_rw(a.x_t + 8 * c, x);  // x_prev may alias x_t
    if constexpr (BF) {
      unpack_vec(__ldg(reinterpret_cast<const uint4*>(a.eps) + c), e, static_cast<__nv_bfloat16*>(nullptr));
    } else {
      load8f(static_cast<const float*>(a.eps) + 8 * c, e);
    }
    if (a.z) {
      load8f(a.z + 8 * c, z);
    } else {
#pragma unroll
      for (int j = 0; j < 8; ++j) z[j] = 0.f;
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) x[j] = fmaf(a.sigma, z[j], fmaf(-a.c1, e[j], x[j]) * a.inv_sqrt_alpha);
    float4* xp = reinterpret_cast<float4*>(a.x_prev + 8 * c);
    xp[0] = make_float4(x[0], x[1], x[2], x[3]);
    xp[1] = make_float4(x[4], x[5], x[6], x[7]);
    if (a.x_next) {
      if constexpr (BF) {
        reinterpret_cast<uint4*>(a.x_next)[c] = pack8(x);
      } else {
        float4* xn = reinterpret_cast<float4*>(a.x_next) + 2 * c;
        xn[0] = make_float4(x[0], x[1], x[2], x[3]);
        xn[1] = make_float4(x[4], x[5], x[6], x[7]);
      }
    }
  }
}

}  // namespace

size_t ada_mod_smem(int B, int D) { return static_cast<size_t>(B) * D * sizeof(float); }

cudaError_t launch_ada_mod(const AdaModArgs& a, int n_sms, cudaStream_t s) {
  const size_t smem = ada_mod_smem(a.B, a.D);
  if (smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(ada_mod_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
  }
  // Two blocks per SM (128 registers a thread), fewer when the staged
  // conditioning is large; the warps stride over groups of kModR rows.
  int per_sm = static_cast<int>((200 * 1024) / (smem + 1024));
  per_sm = per_sm < 1 ? 1 : (per_sm > 2 ? 2 : per_sm);
  const long long groups = static_cast<long long>(a.L) * 6 * a.D / kModR;
  long long grid = static_cast<long long>(n_sms) * per_sm;
  const long long need = (groups + kModWarps - 1) / kModWarps;
  if (grid > need) grid = need;
  return launch_pdl(ada_mod_kernel, dim3(static_cast<unsigned>(grid)), dim3(kModWarps * 32), smem, s, a);
}

cudaError_t launch_adaln_rows(const AdaLnArgs& a, cudaStream_t s) {
  if (a.T <= 0) return cudaSuccess;
  if (a.seq <= 0 || a.D % 64 || a.D > kAdaLnMaxD) return cudaErrorInvalidValue;
  const int grid = (a.T + kLnWarps - 1) / kLnWarps;
  const size_t smem = a.rows ? 0 : static_cast<size_t>(5) * a.D * sizeof(float);
  if (smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(adaln_rows_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
  }
  return launch_pdl(adaln_rows_kernel, dim3(grid), dim3(kLnWarps * 32), smem, s, a);
}

cudaError_t launch_ddpm(const DdpmArgs& a, cudaStream_t s) {
  if (a.n <= 0) return cudaSuccess;
  int dev = 0, n_sms = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&n_sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  // Grid-stride loop: eight 256-thread blocks per SM at most.
  long long blocks = (a.n / 8 + kDdpmThreads - 1) / kDdpmThreads;
  if (blocks > 8LL * n_sms) blocks = 8LL * n_sms;
  if (a.bf16) return launch_pdl(ddpm_kernel<true>, dim3(static_cast<unsigned>(blocks)), dim3(kDdpmThreads), 0, s, a);
  return launch_pdl(ddpm_kernel<false>, dim3(static_cast<unsigned>(blocks)), dim3(kDdpmThreads), 0, s, a);
}

}  // namespace moeca
