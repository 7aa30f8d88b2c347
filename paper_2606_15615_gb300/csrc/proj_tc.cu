// Tensor-core projection GEMM of the attention path (bf16 operands, fp32
// accumulation) for sm_103a.
//
//   C[m, n] = sum_k A[m, k] B[n, k] + bias[n]        0 <= m < M, 0 <= n < N
//
// with A [rows, K] row-major (the block input for the query / key / value
// projection, the attention rows for the output projection) and B [N, K] a
// weight matrix.  Two epilogues:
//   kProjStore     out[m, n] = bf16(C[m, n])
//   kProjQKV       N = 3D split into the attention's operand layouts: the q
//                  columns of token m go to row inv[m] of q_out (the token's
//                  place in the recomputing-token list; none if -1), the k
//                  columns to row m of k_out, and the v columns, transposed,
//                  to column m of vt_out [D, n_tok]
//   kProjResidual  row m belongs to token t = rows[m] (or m):
//                  a = bf16(C[m, :]), a_out[t, :] = a, u_out[t, :] = bf16(x[t, :] + a)
//                  (the attention output a_i and the MoE input u_i = x_i + a_i);
//                  u_i also goes to the token's FFN input rows when row_of is set
//   kProjResidualGated  as kProjResidual with u = bf16(x + g a), g the row's
//                  AdaLN gate (the sample's gate vector, Sec. 3); no FFN rows
// M is a host bound; when m_dev is set the launch reads the actual row count
// there (rows recomputed this step) and tiles past it return at once.
//
// One CTA per 128 x BN output tile, 6 warps:
//   warp 0    TMA producer: A 128 x 64 and B BN x 64 per stage, 128-byte
//             swizzle, into a ring of `nst` stages;
//   warp 1    allocates BN TMEM columns and issues tcgen05.mma (M = 128,
//             N = BN, K = 16) from one thread; tcgen05.commit frees a stage
//             and finally signals the finished accumulator;
//   warps 2-5 epilogue: warp w reads TMEM lanes 32 (w % 4) .. + 31 (its rows),
//             32 columns at a time, and adds the bias (staged in shared memory
//             while the MMAs run).  Store mode rounds to bf16 and writes
//             through a 2 KB shared-memory stage, so each store covers 64
//             contiguous bytes of 8 rows; residual mode loads the token's x
//             one chunk ahead and writes a and u, 64 bytes per lane.
// Every wait is bounded (about one second); a wait that runs out records the
// timeout status, raises a CTA abort flag, waits (bounded) for the copies and
// MMAs already issued, frees TMEM and returns.
#include <cuda.h>

#include <cstdio>
#include <type_traits>

#include "common.cuh"
#include "kernels.h"
#include "tc_common.cuh"

namespace moeca {

namespace {

constexpr int kPM = 128;
constexpr int kPThreads = 192;
constexpr int kPABytes = kPM * 64 * 2;  // 16 KB: A box of one stage
constexpr int kPEpiStage = 32 * 64;     // per epilogue warp: 32 rows x 32 bf16

struct ProjParams {
  int M, N, K;
  const int* m_dev;          // device row count (<= M), or null: M rows
  const float* bias;         // [N] or null
  int mode;                  // ProjMode
  __nv_bfloat16* out;        // kProjStore: [M, ldo]
  int ldo;
  const int32_t* rows;       // kProjResidual: token of row m, or null (m)
  int n_tok;                 // kProjResidual: tokens the x / a_out / u_out rows hold
  const __nv_bfloat16* x;    // kProjResidual: [n_tok, N]
  __nv_bfloat16* a_out;      // kProjResidual: [n_tok, N]
  __nv_bfloat16* u_out;      // kProjResidual: [n_tok, N]
  int nst;                   // ring stages
  unsigned long long* row_stat;
  const int32_t* row_of;     // kProjResidual: [n_tok, row_w] FFN rows of the token (-1: none), or null
  int row_w;
  __nv_bfloat16* xg;         // [rows, N] FFN input rows that also take u
  const int32_t* inv;        // kProjQKV: list place of token m (-1: none), or null (m)
  __nv_bfloat16* q_out;      // kProjQKV: [list rows, D]
  __nv_bfloat16* k_out;      // kProjQKV: [n_tok, D]
  __nv_bfloat16* vt_out;     // kProjQKV: [D, n_tok]
  const float* gate;         // kProjResidualGated: gate row of token t at gate + (t / seq) * gate_ld
  int gate_ld, seq;
  int* status;
};

constexpr int kMaxRowOf = kMaxTopK + 1;

// Store mode, one warp's 32 x 32 chunk: lane i holds row i's 32 values
// (bias added).  They are rounded to bf16 and staged, then written 16 bytes
// per lane with four lanes per row, so each store covers 64 contiguous bytes
// of 8 rows.  `dst` is this lane's row at the chunk's first column (null:
// not stored).
__device__ __forceinline__ void store_chunk_staged(uint8_t* stage, const float* v, __nv_bfloat16* dst, int lane) {
  uint32_t packed[16];
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    __nv_bfloat162 h2 = __floats2bfloat162_rn(v[2 * j], v[2 * j + 1]);
    packed[j] = *reinterpret_cast<uint32_t*>(&h2);
  }
#pragma unroll
  for (int j = 0; j < 4; ++j)
    *reinterpret_cast<uint4*>(stage + lane * 64 + ((j ^ ((lane >> 1) & 3)) << 4)) =
        make_uint4(packed[4 * j], packed[4 * j + 1], packed[4 * j + 2], packed[4 * j + 3]);
  __syncwarp();
  const unsigned long long d_mine = reinterpret_cast<unsigned long long>(dst);
#pragma unroll
  for (int it = 0; it < 4; ++it) {
    const int row = it * 8 + (lane >> 2), j = lane & 3;
    const uint4 val = *reinterpret_cast<const uint4*>(stage + row * 64 + ((j ^ ((row >> 1) & 3)) << 4));
    __nv_bfloat16* d = reinterpret_cast<__nv_bfloat16*>(__shfl_sync(0xffffffffu, d_mine, row));
    if (d) *reinterpret_cast<uint4*>(d + j * 8) = val;
  }
  __syncwarp();
}

// q/k/v mode, v columns: the warp's 32 x 32 chunk transposed through the
// stage, so each lane writes 16 bytes (8 consecutive tokens) of one v^T row.
// `vt` is v^T's row of the chunk's first column, `tok0` the warp's first
// token (a multiple of 32), `M` the token count (a multiple of 8).
__device__ __forceinline__ void store_chunk_transposed(uint8_t* stage, const float* v, __nv_bfloat16* vt, int tok0,
                                                       int M, size_t ld, int lane) {
  __nv_bfloat16* st = reinterpret_cast<__nv_bfloat16*>(stage);  // [32 columns][32 tokens]
#pragma unroll
  for (int j = 0; j < 32; ++j) st[j * 32 + lane] = __float2bfloat16_rn(v[j]);
  __syncwarp();
#pragma unroll
  for (int it = 0; it < 4; ++it) {
    const int j = it * 8 + (lane >> 2), seg = lane & 3;
    const int tok = tok0 + seg * 8;
    if (tok < M)
      *reinterpret_cast<uint4*>(vt + static_cast<size_t>(j) * ld + tok) =
          *reinterpret_cast<const uint4*>(st + j * 32 + seg * 8);
  }
  __syncwarp();
}

// Residual mode, one lane's row: a = bf16(v), u = bf16(x + a), each 64
// contiguous bytes (two full 32-byte sectors) written by the lane itself;
// u also goes to the token's FFN input rows (g_dst[q], or null).
__device__ __forceinline__ void store_residual(const float* v, const uint4* xv, __nv_bfloat16* a_dst,
                                               __nv_bfloat16* u_dst, __nv_bfloat16* const* g_dst, int n_g) {
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    uint4 av, uv;
    __nv_bfloat162* ah = reinterpret_cast<__nv_bfloat162*>(&av);
    __nv_bfloat162* uh = reinterpret_cast<__nv_bfloat162*>(&uv);
    const __nv_bfloat162* xh = reinterpret_cast<const __nv_bfloat162*>(&xv[j]);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      ah[q] = __floats2bfloat162_rn(v[8 * j + 2 * q], v[8 * j + 2 * q + 1]);
      const float2 af = __bfloat1622float2(ah[q]);
      const float2 xf = __bfloat1622float2(xh[q]);
      uh[q] = __floats2bfloat162_rn(xf.x + af.x, xf.y + af.y);
    }
    reinterpret_cast<uint4*>(a_dst)[j] = av;
    reinterpret_cast<uint4*>(u_dst)[j] = uv;
#pragma unroll
    for (int q = 0; q < kMaxRowOf; ++q)
      if (q < n_g && g_dst[q]) reinterpret_cast<uint4*>(g_dst[q])[j] = uv;
  }
}

// Gated residual (AdaLN block): a = bf16(v), u = bf16(x + g a), 32 columns.
__device__ __forceinline__ void store_residual_gated(const float* v, const uint4* xv, const float* g,
                                                     __nv_bfloat16* a_dst, __nv_bfloat16* u_dst) {
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const float4 g0 = __ldg(reinterpret_cast<const float4*>(g + 8 * j));
    const float4 g1 = __ldg(reinterpret_cast<const float4*>(g + 8 * j) + 1);
    const float gg[8] = {g0.x, g0.y, g0.z, g0.w, g1.x, g1.y, g1.z, g1.w};
    uint4 av, uv;
    __nv_bfloat162* ah = reinterpret_cast<__nv_bfloat162*>(&av);
    __nv_bfloat162* uh = reinterpret_cast<__nv_bfloat162*>(&uv);
    const __nv_bfloat162* xh = reinterpret_cast<const __nv_bfloat162*>(&xv[j]);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      ah[q] = __floats2bfloat162_rn(v[8 * j + 2 * q], v[8 * j + 2 * q + 1]);
      const float2 af = __bfloat1622float2(ah[q]);
      const float2 xf = __bfloat1622float2(xh[q]);
      uh[q] = __floats2bfloat162_rn(fmaf(gg[2 * q], af.x, xf.x), fmaf(gg[2 * q + 1], af.y, xf.y));
    }
    reinterpret_cast<uint4*>(a_dst)[j] = av;
    reinterpret_cast<uint4*>(u_dst)[j] = uv;
  }
}

__device__ __forceinline__ void load_x_chunk(const __nv_bfloat16* xr, uint4* xv) {
#pragma unroll
  for (int j = 0; j < 4; ++j) xv[j] = __ldg(reinterpret_cast<const uint4*>(xr) + j);
}

template <int BN, int MODE>
__global__ void __launch_bounds__(kPThreads, 1)
    proj_tc_kernel(const __grid_constant__ CUtensorMap amap, const __grid_constant__ CUtensorMap bmap,
                   const ProjParams p) {
  constexpr int kStage = kPABytes + BN * 128;
  constexpr bool kRes = MODE == kProjResidual || MODE == kProjResidualGated;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[8];
  __shared__ __align__(8) uint64_t empty_bar[8];
  __shared__ __align__(8) uint64_t acc_bar;
  __shared__ __align__(8) uint64_t drain_bar;
  __shared__ uint32_t tmem_sh;
  __shared__ volatile int abort_flag;
  __shared__ float s_bias[BN];

  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* epi = smem + p.nst * kStage;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n0 = blockIdx.x * BN, m0 = blockIdx.y * kPM;

  if (threadIdx.x == 0) {
    abort_flag = 0;
    for (int s = 0; s < p.nst; ++s) {
      mbar_init(smem_u32(&full_bar[s]), 1);
      mbar_init(smem_u32(&empty_bar[s]), 1);
    }
    mbar_init(smem_u32(&acc_bar), 1);
    mbar_init(smem_u32(&drain_bar), 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&amap)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&bmap)) : "memory");
  }
  pdl_entry();
  const int M = p.m_dev ? min(*reinterpret_cast<const volatile int*>(p.m_dev), p.M) : p.M;
  if (p.row_stat && blockIdx.x == 0 && blockIdx.y == 0 && threadIdx.x == 0)
    atomicAdd(p.row_stat, static_cast<unsigned long long>(M));
  if (m0 >= M) return;  // uniform over the CTA, before TMEM is taken
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&tmem_sh)),
                 "r"(BN < 32 ? 32 : BN)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    tc_fence_before();
  }
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_sh;
  const int KB = p.K / 64;
  const int nst = p.nst;
  int issued = 0;  // producer: stages issued

  if (warp == 0) {
    if (lane == 0) {
      for (int kb = 0; kb < KB; ++kb) {
        const int s = kb % nst;
        if (kb >= nst && !mbar_wait(smem_u32(&empty_bar[s]), ((kb / nst) & 1) ^ 1, &abort_flag)) {
          if (!abort_flag) report_status(p.status, kStatusWaitTimeout, 600);
          abort_flag = 1;
          break;
        }
        const uint32_t sa = smem_u32(smem + s * kStage);
        mbar_expect_tx(smem_u32(&full_bar[s]), kStage);
        tma_load_2d(sa, &amap, kb * 64, m0, smem_u32(&full_bar[s]));
        tma_load_2d(sa + kPABytes, &bmap, kb * 64, n0, smem_u32(&full_bar[s]));
        ++issued;
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = instr_desc(kPM, BN);
      bool ok = true;
      for (int kb = 0; kb < KB; ++kb) {
        const int s = kb % nst;
        if (!mbar_wait(smem_u32(&full_bar[s]), (kb / nst) & 1, &abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t sa = smem_u32(smem + s * kStage);
        const uint32_t sb = sa + kPABytes;
#pragma unroll
        for (int kk = 0; kk < 4; ++kk)
          mma_bf16(tmem, smem_desc(sa + kk * 32), smem_desc(sb + kk * 32), idesc, (kb | kk) != 0);
        mma_commit(smem_u32(&empty_bar[s]));
      }
      if (ok) {
        mma_commit(smem_u32(&acc_bar));
      } else {
        if (!abort_flag) report_status(p.status, kStatusWaitTimeout, 601);
        abort_flag = 1;
      }
      // Every MMA issued so far has completed once the drain barrier fires.
      mma_commit(smem_u32(&drain_bar));
      const unsigned long long t0 = globaltimer();
      while (!mbar_try(smem_u32(&drain_bar), 0) && globaltimer() - t0 < kTcWaitNs) {
      }
    }
  } else {
    const int quad = warp & 3;
    const int r = quad * 32 + lane;
    const int m = m0 + r;
    uint8_t* stage = epi + (warp - 2) * kPEpiStage;
    // While the MMAs run: the tile's bias into shared memory, this lane's
    // row pointers, and the residual rows' first chunk of x.
    for (int j = threadIdx.x - 64; j < BN; j += 128) s_bias[j] = p.bias ? __ldg(p.bias + n0 + j) : 0.f;
    __nv_bfloat16* dst = nullptr;
    const __nv_bfloat16* xr = nullptr;
    __nv_bfloat16* ur = nullptr;
    __nv_bfloat16* gr[kMaxRowOf];
#pragma unroll
    for (int q = 0; q < kMaxRowOf; ++q) gr[q] = nullptr;
    const int n_g = p.row_of ? p.row_w : 0;
    __nv_bfloat16* krow = nullptr;  // kProjQKV: this lane's k row (dst holds its q row)
    const float* grow = nullptr;    // kProjResidualGated: this lane's gate row
    if (m < M) {
      if constexpr (MODE == kProjStore) {
        dst = p.out + static_cast<size_t>(m) * p.ldo + n0;
      } else if constexpr (MODE == kProjQKV) {
        const int qi = p.inv ? p.inv[m] : m;
        const int Dm = p.N / 3;
        if (qi >= 0) dst = p.q_out + static_cast<size_t>(qi) * Dm;
        krow = p.k_out + static_cast<size_t>(m) * Dm;
      } else {
        const int t = p.rows ? p.rows[m] : m;
        if (t >= 0 && t < p.n_tok) {
          const size_t off = static_cast<size_t>(t) * p.N + n0;
          dst = p.a_out + off;
          xr = p.x + off;
          ur = p.u_out + off;
          if constexpr (MODE == kProjResidualGated) grow = p.gate + static_cast<size_t>(t / p.seq) * p.gate_ld + n0;
#pragma unroll
          for (int q = 0; q < kMaxRowOf; ++q) {
            if (q < n_g) {
              const int pos = p.row_of[static_cast<size_t>(t) * p.row_w + q];
              if (pos >= 0) gr[q] = p.xg + static_cast<size_t>(pos) * p.N + n0;
            }
          }
        } else {
          report_status(p.status, kStatusBadIndex, 6000000 + m);
        }
      }
    }
    uint4 xb[2][4];  // residual mode: x of chunks c and c + 1 in flight
    if constexpr (kRes) {
      if (xr) {
        load_x_chunk(xr, xb[0]);
        if (BN > 32) load_x_chunk(xr + 32, xb[1]);
      }
    }
    asm volatile("bar.sync 1, 128;" ::: "memory");  // the four epilogue warps: bias staged
    if (mbar_wait(smem_u32(&acc_bar), 0, &abort_flag)) {
      tc_fence_after();
      const uint32_t tbase = tmem + (static_cast<uint32_t>(quad * 32) << 16);
      if constexpr (kRes) {
#pragma unroll
        for (int c = 0; c < BN / 32; ++c) {
          uint4 xc[4];
#pragma unroll
          for (int j = 0; j < 4; ++j) xc[j] = xb[c & 1][j];
          if (xr && c + 2 < BN / 32) load_x_chunk(xr + (c + 2) * 32, xb[c & 1]);  // two chunks ahead
          uint32_t raw[32];
          tmem_ld32(tbase + c * 32, raw);
          float v[32];
#pragma unroll
          for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(raw[j]) + s_bias[c * 32 + j];
          if (dst) {
            if constexpr (MODE == kProjResidualGated) {
              store_residual_gated(v, xc, grow + c * 32, dst + c * 32, ur + c * 32);
            } else {
              __nv_bfloat16* gc[kMaxRowOf];
#pragma unroll
              for (int q = 0; q < kMaxRowOf; ++q) gc[q] = gr[q] ? gr[q] + c * 32 : nullptr;
              store_residual(v, xc, dst + c * 32, ur + c * 32, gc, n_g);
            }
          }
        }
      } else {
        // Store-type epilogues stay rolled: the chunk body is large and an
        // unrolled copy per chunk spills out of the instruction cache.
#pragma unroll 1
        for (int c = 0; c < BN / 32; ++c) {
          uint32_t raw[32];
          tmem_ld32(tbase + c * 32, raw);
          float v[32];
#pragma unroll
          for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(raw[j]) + s_bias[c * 32 + j];
          if constexpr (MODE == kProjStore) {
            store_chunk_staged(stage, v, dst ? dst + c * 32 : nullptr, lane);
          } else {
            // The chunk lies in one of q, k, v (D is a multiple of 64): warp-uniform.
            const int Dm = p.N / 3;
            const int col = n0 + c * 32;
            const int region = col / Dm, cc = col - region * Dm;
            if (region == 0) {
              store_chunk_staged(stage, v, dst ? dst + cc : nullptr, lane);
            } else if (region == 1) {
              store_chunk_staged(stage, v, krow ? krow + cc : nullptr, lane);
            } else {
              store_chunk_transposed(stage, v, p.vt_out + static_cast<size_t>(cc) * p.n_tok, m0 + quad * 32, M,
                                     static_cast<size_t>(p.n_tok), lane);
            }
          }
        }
      }
    } else if (lane == 0) {
      if (!abort_flag) report_status(p.status, kStatusWaitTimeout, 602);
      abort_flag = 1;
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0 && lane == 0 && abort_flag) {
    // Copies issued but never consumed still land in shared memory: wait for
    // the newest phase of every stage before the CTA exits.
    for (int s = 0; s < nst && s < issued; ++s) {
      const int last = issued - 1 - ((issued - 1 - s) % nst);  // newest k-block issued on stage s
      const unsigned long long t0 = globaltimer();
      while (!mbar_try(smem_u32(&full_bar[s]), (last / nst) & 1) && globaltimer() - t0 < kTcWaitNs) {
      }
    }
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(BN < 32 ? 32 : BN)
                 : "memory");
  }
}

template <int BN>
constexpr int stage_bytes() {
  return kPABytes + BN * 128;
}

}  // namespace

int proj_tile_n(int N, int want) {
  if (want) return (want == 64 || want == 128 || want == 256) && N % want == 0 ? want : 0;
  if (N % 256 == 0) return 256;
  if (N % 128 == 0) return 128;
  if (N % 64 == 0) return 64;
  return 0;
}

cudaError_t launch_proj_tc(const ProjArgs& a, cudaStream_t s) {
  const int BN = proj_tile_n(a.N, a.tile_n);
  if (BN == 0 || a.K % 64 || a.M <= 0) return cudaErrorInvalidValue;
  if (a.mode == kProjResidualGated && (!a.gate || a.seq <= 0 || a.row_of)) return cudaErrorInvalidValue;
  CUtensorMap amap, bmap;
  if (!encode_2d(&amap, a.A, static_cast<uint64_t>(a.a_rows), static_cast<uint64_t>(a.K), kPM) ||
      !encode_2d(&bmap, a.B, static_cast<uint64_t>(a.N), static_cast<uint64_t>(a.K), static_cast<uint32_t>(BN)))
    return cudaErrorInvalidValue;
  ProjParams p{};
  p.M = a.M; p.N = a.N; p.K = a.K; p.m_dev = a.m_dev; p.bias = a.bias; p.mode = a.mode;
  p.out = static_cast<__nv_bfloat16*>(a.out); p.ldo = a.ldo;
  p.rows = a.rows; p.n_tok = a.n_tok;
  p.x = static_cast<const __nv_bfloat16*>(a.x);
  p.a_out = static_cast<__nv_bfloat16*>(a.a_out);
  p.u_out = static_cast<__nv_bfloat16*>(a.u_out);
  p.row_stat = a.row_stat;
  p.row_of = a.row_of;
  p.row_w = a.row_w;
  p.xg = static_cast<__nv_bfloat16*>(a.xg);
  p.inv = a.inv;
  p.q_out = static_cast<__nv_bfloat16*>(a.q_out);
  p.k_out = static_cast<__nv_bfloat16*>(a.k_out);
  p.vt_out = static_cast<__nv_bfloat16*>(a.vt_out);
  p.gate = a.gate; p.gate_ld = a.gate_ld; p.seq = a.seq;
  p.status = a.status;
  const int kb = a.K / 64;
  const int stage = kPABytes + BN * 128;
  int nst = (200 * 1024) / stage;
  nst = nst > 8 ? 8 : nst;
  nst = nst > kb ? kb : nst;
  if (nst < 1) nst = 1;
  p.nst = nst;
  const size_t smem = static_cast<size_t>(nst) * stage + 4 * kPEpiStage + 1024;
  const dim3 grid(a.N / BN, (a.M + kPM - 1) / kPM);
  auto run = [&](auto kern) -> cudaError_t {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    return launch_pdl(kern, grid, dim3(kPThreads), smem, s, amap, bmap, p);
  };
  auto by_mode = [&](auto bn) -> cudaError_t {
    constexpr int kBN = decltype(bn)::value;
    switch (a.mode) {
      case kProjQKV: return run(proj_tc_kernel<kBN, kProjQKV>);
      case kProjResidual: return run(proj_tc_kernel<kBN, kProjResidual>);
      case kProjResidualGated: return run(proj_tc_kernel<kBN, kProjResidualGated>);
      default: return run(proj_tc_kernel<kBN, kProjStore>);
    }
  };
  switch (BN) {
    case 256: return by_mode(std::integral_constant<int, 256>{});
    case 128: return by_mode(std::integral_constant<int, 128>{});
    default: return by_mode(std::integral_constant<int, 64>{});
  }
}

}  // namespace moeca
