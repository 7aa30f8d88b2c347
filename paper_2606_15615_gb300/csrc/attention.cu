// Attention path of a DiT-MoE block (Sec. 4.1) for sm_103a, bf16 storage and
// fp32 arithmetic:
//   attn_residual_kernel  u = x + a^{t0}: the MoE input of every token on a
//                         cache step before its attention is (maybe) updated
//   attn_rows_kernel      ascending list of the tokens whose recompute set is
//                         non-empty (they recompute their attention output)
//   attn_core_kernel<DH>  multi-head self-attention of the listed query rows
//                         over all keys and values of their sample:
//                         o = softmax(q k^T / sqrt(dh)) v per head, one pass
//                         over the keys with a running maximum and sum
//                         (online softmax), bf16 tensor-core products
//                         (mma.sync m16n8k16) with fp32 accumulation.
// The query / key / value and output projections are tensor-core GEMMs
// (proj_tc.cu).
#include <cmath>

#include "common.cuh"
#include "kernels.h"

namespace moeca {

namespace {

constexpr int kQRows = 64;     // query rows per CTA, 16 per warp
constexpr int kKeys = 64;      // keys per block of the online softmax
constexpr int kCoreThreads = 128;

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, bool valid) {
  const int n = valid ? 16 : 0;  // 0: the 16 bytes are zero-filled, nothing is read
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(n) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}
// 2^x with the hardware approximation (ex2.approx; relative error about 2^-22).
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&h);
}

__global__ void __launch_bounds__(256) attn_residual_kernel(const uint4* x, const uint4* a, uint4* u, size_t nvec) {
  pdl_entry();
  for (size_t i = static_cast<size_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < nvec;
       i += static_cast<size_t>(gridDim.x) * blockDim.x) {
    float xv[8], av[8];
    unpack_vec(x[i], xv, static_cast<__nv_bfloat16*>(nullptr));
    unpack_vec(a[i], av, static_cast<__nv_bfloat16*>(nullptr));
#pragma unroll
    for (int j = 0; j < 8; ++j) xv[j] += av[j];
    uint4 r;
    __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&r);
#pragma unroll
    for (int j = 0; j < 4; ++j) h[j] = __floats2bfloat162_rn(xv[2 * j], xv[2 * j + 1]);
    u[i] = r;
  }
}

// One block of 1024 threads: thread j scans tokens [j per, (j + 1) per).
// Also writes where each sample's tokens start in the list (sample_lo[b] for
// sample b of S tokens, sample_lo[T / S] = the list's length).
__global__ void __launch_bounds__(1024) attn_rows_kernel(const uint8_t* any, int T, int S, int32_t* rows,
                                                         int* n_rows, int32_t* sample_lo, int32_t* inv) {
  pdl_entry();
  __shared__ int warp_tot[32];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int per = (T + 1023) / 1024;
  const int beg = min(tid * per, T), end = min(beg + per, T);
  int c = 0;
  for (int i = beg; i < end; ++i) c += any[i] != 0;
  int incl = c;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const int v = __shfl_up_sync(0xffffffffu, incl, d);
    if (lane >= d) incl += v;
  }
  if (lane == 31) warp_tot[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    int w = warp_tot[lane];
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
      const int v = __shfl_up_sync(0xffffffffu, w, d);
      if (lane >= d) w += v;
    }
    warp_tot[lane] = w;  // inclusive over warps
  }
  __syncthreads();
  int pos = incl - c + (warp ? warp_tot[warp - 1] : 0);
  for (int i = beg; i < end; ++i) {
    if (i % S == 0) sample_lo[i / S] = pos;
    if (any[i]) {
      inv[i] = pos;
      rows[pos++] = i;
    } else {
      inv[i] = -1;
    }
  }
  if (tid == 1023) {
    *n_rows = warp_tot[31];
    sample_lo[T / S] = warp_tot[31];
  }
}

// Key / value blocks in flight: a ring of NBUF blocks of 64 keys, NBUF - 1
// loading while one is used (a 256-key sample arrives in one round trip for
// heads up to 80 channels); two CTAs still fit on an SM.
template <int DH>
__host__ __device__ constexpr int core_nbuf() {
  return DH <= 80 ? 4 : (DH <= 96 ? 3 : 2);
}

// Shared memory of attn_core_kernel<DH>: Q [64][DK + 8], K [NBUF][64][DK + 8],
// V^T [NBUF][DH][64 + 8] (bf16; 16 bytes of padding per row keep ldmatrix
// free of bank conflicts).  DK = DH rounded up to 16 (the q k^T contraction).
constexpr int kLdVt = kKeys + 8;
template <int DH>
constexpr size_t core_smem() {
  constexpr int DK = (DH + 15) / 16 * 16;
  constexpr int NB = core_nbuf<DH>();
  return (static_cast<size_t>(kQRows) * (DK + 8) + NB * kKeys * (DK + 8) + NB * DH * kLdVt) * 2;
}

template <int DH>
__global__ void __launch_bounds__(kCoreThreads) attn_core_kernel(AttnArgs a, float scale_log2) {
  constexpr int DK = (DH + 15) / 16 * 16;
  constexpr int LDQ = DK + 8;
  constexpr int NT = DH / 8;   // 8-column tiles of the output
  constexpr int CH = DH / 8;   // 16-byte chunks of one head row
  constexpr int NB = core_nbuf<DH>();
  extern __shared__ __align__(16) uint8_t smem[];
  __nv_bfloat16* sQ = reinterpret_cast<__nv_bfloat16*>(smem);
  __nv_bfloat16* sK = sQ + kQRows * LDQ;
  __nv_bfloat16* sV = sK + NB * kKeys * LDQ;
  __shared__ int s_tok[kQRows];

  pdl_entry();
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int b = blockIdx.y, h = blockIdx.z;
  const int S = a.S, D = a.D, T = a.T;
  const int key0 = b * S;
  int lo = key0, hi = key0 + S;
  if (a.rows) {
    lo = a.sample_lo[b];
    hi = a.sample_lo[b + 1];
  }
  const int r0 = lo + blockIdx.x * kQRows;
  if (r0 >= hi) return;
  const int nq = min(kQRows, hi - r0);
  if (tid < kQRows) {
    int t = -1;
    if (tid < nq) {
      t = a.rows ? a.rows[r0 + tid] : r0 + tid;
      if (t < key0 || t >= key0 + S) {
        report_status(a.status, kStatusBadIndex, 7000000 + r0 + tid);
        t = -1;
      }
    }
    s_tok[tid] = t;
  }
  if (DK > DH) {
    // Columns DH..DK of the q and k rows take part in q k^T: keep them 0.
    for (int i = tid; i < kQRows + NB * kKeys; i += kCoreThreads) {
      __nv_bfloat16* row = i < kQRows ? sQ + i * LDQ : sK + (i - kQRows) * LDQ;
#pragma unroll
      for (int c = DH; c < DK; ++c) row[c] = __float2bfloat16_rn(0.f);
    }
  }
  __syncthreads();
  const __nv_bfloat16* qg = static_cast<const __nv_bfloat16*>(a.q);
  const __nv_bfloat16* kg = static_cast<const __nv_bfloat16*>(a.k);
  const __nv_bfloat16* vtg = static_cast<const __nv_bfloat16*>(a.vt);
  for (int i = tid; i < kQRows * CH; i += kCoreThreads) {
    const int r = i / CH, c = i % CH;
    const bool v = s_tok[r] >= 0;
    const __nv_bfloat16* src = qg + static_cast<size_t>(v ? r0 + r : 0) * D + h * DH + c * 8;
    cp_async16(smem_u32(sQ + r * LDQ + c * 8), src, v);
  }
  auto load_kv = [&](int kb, int buf) {
    for (int i = tid; i < kKeys * CH; i += kCoreThreads) {
      const int r = i / CH, c = i % CH;
      const int key = kb * kKeys + r;
      const bool v = key < S;
      const __nv_bfloat16* src = kg + static_cast<size_t>(key0 + (v ? key : 0)) * D + h * DH + c * 8;
      cp_async16(smem_u32(sK + (buf * kKeys + r) * LDQ + c * 8), src, v);
    }
    // v^T rows (channels) of this head, 8 keys per copy (S is a multiple of 8).
    for (int i = tid; i < DH * (kKeys / 8); i += kCoreThreads) {
      const int d = i / (kKeys / 8), c = i % (kKeys / 8);
      const int key = kb * kKeys + c * 8;
      const bool v = key < S;
      const __nv_bfloat16* src = vtg + static_cast<size_t>(h * DH + d) * T + key0 + (v ? key : 0);
      cp_async16(smem_u32(sV + (buf * DH + d) * kLdVt + c * 8), src, v);
    }
  };
  const int nkb = (S + kKeys - 1) / kKeys;
  // Groups: block 0 (with q), then one per block; empty groups keep the count.
#pragma unroll
  for (int j = 0; j < NB - 1; ++j) {
    if (j < nkb) load_kv(j, j);
    cp_async_commit();
  }

  const int g = lane >> 2, q4 = lane & 3;
  const int mat = lane >> 3, mr = lane & 7;
  float o[NT][4];
#pragma unroll
  for (int t = 0; t < NT; ++t) o[t][0] = o[t][1] = o[t][2] = o[t][3] = 0.f;
  float m_run[2] = {-INFINITY, -INFINITY}, l_run[2] = {0.f, 0.f};
  uint32_t qf[DK / 16][4];

  for (int kb = 0; kb < nkb; ++kb) {
    if (kb + NB - 1 < nkb) load_kv(kb + NB - 1, (kb + NB - 1) % NB);
    cp_async_commit();
    cp_async_wait<NB - 1>();  // block kb (and q) have landed
    __syncthreads();
    if (kb == 0) {
#pragma unroll
      for (int kc = 0; kc < DK / 16; ++kc)
        ldsm_x4(smem_u32(sQ + (warp * 16 + (mat & 1) * 8 + mr) * LDQ + kc * 16 + (mat >> 1) * 8), qf[kc][0],
                qf[kc][1], qf[kc][2], qf[kc][3]);
    }
    const __nv_bfloat16* kbuf = sK + (kb % NB) * kKeys * LDQ;
    const __nv_bfloat16* vbuf = sV + (kb % NB) * DH * kLdVt;
    // ---- scores of this warp's 16 rows against 64 keys
    float s[8][4];
#pragma unroll
    for (int t = 0; t < 8; ++t) s[t][0] = s[t][1] = s[t][2] = s[t][3] = 0.f;
#pragma unroll
    for (int np = 0; np < 4; ++np) {
#pragma unroll
      for (int kc = 0; kc < DK / 16; ++kc) {
        uint32_t b0, b1, b2, b3;
        ldsm_x4(smem_u32(kbuf + (np * 16 + (mat >> 1) * 8 + mr) * LDQ + kc * 16 + (mat & 1) * 8), b0, b1, b2, b3);
        mma_16816(s[2 * np], qf[kc][0], qf[kc][1], qf[kc][2], qf[kc][3], b0, b1);
        mma_16816(s[2 * np + 1], qf[kc][0], qf[kc][1], qf[kc][2], qf[kc][3], b2, b3);
      }
    }
    // ---- online softmax (base 2): scale, mask keys past the sample, rescale
    float mx[2] = {m_run[0], m_run[1]};
#pragma unroll
    for (int t = 0; t < 8; ++t) {
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int key = kb * kKeys + t * 8 + 2 * q4 + (j & 1);
        // One rounded product, used for the maximum and the exponent alike.
        const float v = key < S ? __fmul_rn(s[t][j], scale_log2) : -INFINITY;
        s[t][j] = v;
        mx[j >> 1] = fmaxf(mx[j >> 1], v);
      }
    }
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 1));
      mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 2));
    }
    float corr[2];
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      corr[r] = ex2(m_run[r] - mx[r]);  // 0 on the first block (m_run = -inf)
      m_run[r] = mx[r];
      l_run[r] *= corr[r];
    }
#pragma unroll
    for (int t = 0; t < NT; ++t) {
      o[t][0] *= corr[0]; o[t][1] *= corr[0];
      o[t][2] *= corr[1]; o[t][3] *= corr[1];
    }
#pragma unroll
    for (int t = 0; t < 8; ++t) {
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const float p = ex2(s[t][j] - mx[j >> 1]);
        s[t][j] = p;
        l_run[j >> 1] += p;
      }
    }
    // ---- o += p v: p (bf16) is the A operand straight from the score registers
#pragma unroll
    for (int kc = 0; kc < 4; ++kc) {
      const uint32_t a0 = pack_bf16(s[2 * kc][0], s[2 * kc][1]);
      const uint32_t a1 = pack_bf16(s[2 * kc][2], s[2 * kc][3]);
      const uint32_t a2 = pack_bf16(s[2 * kc + 1][0], s[2 * kc + 1][1]);
      const uint32_t a3 = pack_bf16(s[2 * kc + 1][2], s[2 * kc + 1][3]);
      // v^T rows are channels, keys contiguous: the B operand without transposing.
      const int kcol = kc * 16 + (mat & 1) * 8;
#pragma unroll
      for (int np = 0; np < NT / 2; ++np) {
        uint32_t b0, b1, b2, b3;
        ldsm_x4(smem_u32(vbuf + (np * 16 + (mat >> 1) * 8 + mr) * kLdVt + kcol), b0, b1, b2, b3);
        mma_16816(o[2 * np], a0, a1, a2, a3, b0, b1);
        mma_16816(o[2 * np + 1], a0, a1, a2, a3, b2, b3);
      }
      if (NT & 1) {
        uint32_t b0, b1;
        ldsm_x2(smem_u32(vbuf + ((NT - 1) * 8 + mr) * kLdVt + kcol), b0, b1);
        mma_16816(o[NT - 1], a0, a1, a2, a3, b0, b1);
      }
    }
    __syncthreads();
  }
  // ---- normalise and store rows r0 + (this warp's rows)
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    l_run[r] += __shfl_xor_sync(0xffffffffu, l_run[r], 1);
    l_run[r] += __shfl_xor_sync(0xffffffffu, l_run[r], 2);
  }
  __nv_bfloat16* out = static_cast<__nv_bfloat16*>(a.o);
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    const int row = warp * 16 + g + r * 8;
    if (row >= nq || s_tok[row] < 0) continue;
    const float inv = 1.f / l_run[r];
    uint32_t* dst = reinterpret_cast<uint32_t*>(out + static_cast<size_t>(r0 + row) * D + h * DH + 2 * q4);
#pragma unroll
    for (int t = 0; t < NT; ++t) dst[t * 4] = pack_bf16(o[t][2 * r] * inv, o[t][2 * r + 1] * inv);
  }
}

template <int DH>
cudaError_t run_core(const AttnArgs& a, cudaStream_t s) {
  const size_t smem = core_smem<DH>();
  cudaError_t e = cudaFuncSetAttribute(attn_core_kernel<DH>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  const float scale_log2 = 1.4426950408889634f / std::sqrt(static_cast<float>(DH));
  const dim3 grid((a.S + kQRows - 1) / kQRows, a.T / a.S, a.H);
  return launch_pdl(attn_core_kernel<DH>, grid, dim3(kCoreThreads), smem, s, a, scale_log2);
}

}  // namespace

bool attn_supported(int D, int H) {
  if (H < 1 || D % H || D % 64) return false;
  const int dh = D / H;
  return dh == 64 || dh == 72 || dh == 80 || dh == 96 || dh == 128;
}

cudaError_t launch_attn_core(const AttnArgs& a, cudaStream_t s) {
  if (!attn_supported(a.D, a.H) || a.S < 1 || a.S % 8 || a.T % a.S) return cudaErrorInvalidValue;
  switch (a.D / a.H) {
    case 64: return run_core<64>(a, s);
    case 72: return run_core<72>(a, s);
    case 80: return run_core<80>(a, s);
    case 96: return run_core<96>(a, s);
    default: return run_core<128>(a, s);
  }
}

cudaError_t launch_attn_residual(const void* x, const void* a, void* u, int T, int D, int* status, cudaStream_t s) {
  (void)status;
  const size_t nvec = static_cast<size_t>(T) * D / 8;
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  size_t want = (nvec + 255) / 256;
  const size_t cap = static_cast<size_t>(sms) * 8;
  const unsigned grid = static_cast<unsigned>(want < cap ? (want ? want : 1) : cap);
  return launch_pdl(attn_residual_kernel, dim3(grid), dim3(256), 0, s, static_cast<const uint4*>(x),
                    static_cast<const uint4*>(a), static_cast<uint4*>(u), nvec);
}

cudaError_t launch_attn_rows(const uint8_t* token_any, int T, int S, int32_t* rows, int* n_rows,
                             int32_t* sample_lo, int32_t* inv, cudaStream_t s) {
  return launch_pdl(attn_rows_kernel, dim3(1), dim3(1024), 0, s, token_any, T, S, rows, n_rows, sample_lo, inv);
}

}  // namespace moeca
