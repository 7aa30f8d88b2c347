// CUDA-core grouped expert FFN over the compacted recompute rows.
//
// Phase 1: hmid[r, :] = GELU(xg[r, :] W1_g^T)      (first half of Eq. 5's FFN)
// Phase 2: dst[list[r], :] = hmid[r, :] W2_g^T     (second half; rows land in
//          the branch cache slot token*k+slot, or the shared-expert row)
// Rows of group g are [offsets[g], offsets[g] + counts[g]).  The counts live
// on the device, so the grid covers the worst case and each block finds its
// (group, m-tile) from them; blocks past the last tile exit.  fp32 FFMA with
// fp32 accumulation: the fp32 debug-precision path, and a cross-check of the
// tensor-core kernel on bf16.
#include <type_traits>

#include "common.cuh"
#include "kernels.h"

namespace moeca {
namespace {

constexpr int BM = 64, BN = 64, BK = 16;

template <typename TI, int PHASE>
__global__ void __launch_bounds__(256) ffn_simt_kernel(FfnArgs a) {
  pdl_entry();
  const int N = PHASE == 1 ? a.F : a.D;
  const int K = PHASE == 1 ? a.D : a.F;
  int mt = blockIdx.y, g = -1, m0 = 0;
  for (int gg = 0; gg < a.G; ++gg) {
    const int tiles = (a.counts[gg] + BM - 1) / BM;
    if (mt < tiles) {
      g = gg;
      m0 = mt * BM;
      break;
    }
    mt -= tiles;
  }
  if (g < 0) return;
  const int rows = a.counts[g];
  const int row0 = a.offsets[g];
  const int n0 = blockIdx.x * BN;
  const TI* A = static_cast<const TI*>(PHASE == 1 ? a.xg : a.hmid);
  const TI* B;
  if (g < a.E) {
    B = static_cast<const TI*>(PHASE == 1 ? a.w1 : a.w2) + static_cast<size_t>(g) * a.F * a.D;
  } else {
    B = static_cast<const TI*>(PHASE == 1 ? a.ws1 : a.ws2);
  }
  __shared__ float As[BK][BM + 4];
  __shared__ float Bs[BK][BN + 4];
  const int t = threadIdx.x;
  const int ty = t / 16, tx = t % 16;
  const int lr = t / 4, lk = (t % 4) * 4;
  float acc[4][4];
#pragma unroll
  for (int r = 0; r < 4; ++r)
#pragma unroll
    for (int c = 0; c < 4; ++c) acc[r][c] = 0.f;
  for (int k0 = 0; k0 < K; k0 += BK) {
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int kk = k0 + lk + j;
      float av = 0.f, bv = 0.f;
      if (m0 + lr < rows && kk < K)
        av = Elem<TI>::to_f(A[static_cast<size_t>(row0 + m0 + lr) * K + kk]);
      if (n0 + lr < N && kk < K)
        bv = Elem<TI>::to_f(B[static_cast<size_t>(n0 + lr) * K + kk]);
      As[lk + j][lr] = av;
      Bs[lk + j][lr] = bv;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < BK; ++kk) {
      float av[4], bv[4];
#pragma unroll
      for (int r = 0; r < 4; ++r) av[r] = As[kk][ty * 4 + r];
#pragma unroll
      for (int c = 0; c < 4; ++c) bv[c] = Bs[kk][tx * 4 + c];
#pragma unroll
      for (int r = 0; r < 4; ++r)
#pragma unroll
        for (int c = 0; c < 4; ++c) acc[r][c] = fmaf(av[r], bv[c], acc[r][c]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int r = 0; r < 4; ++r) {
    const int m = m0 + ty * 4 + r;
    if (m >= rows) continue;
    const size_t row = static_cast<size_t>(row0 + m);
    if (PHASE == 1) {
      TI* H = static_cast<TI*>(a.hmid);
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const int n = n0 + tx * 4 + c;
        if (n < N) H[row * a.F + n] = Elem<TI>::from_f(gelu_f(acc[r][c], a.gelu_tanh));
      }
    } else {
      const int dr = a.list[row];
      const int lim = g < a.E ? a.T * a.k : a.T;
      if (dr < 0 || dr >= lim) {
        report_status(a.status, kStatusBadIndex, 2000000 + static_cast<int>(row));
        continue;
      }
      TI* dst = static_cast<TI*>(g < a.E ? a.cache_h : a.shared_h);
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const int n = n0 + tx * 4 + c;
        if (n < N) dst[static_cast<size_t>(dr) * a.D + n] = Elem<TI>::from_f(acc[r][c]);
      }
    }
  }
}

// fp32 form with the operand tiles brought into shared memory by cp.async,
// three stages in flight, so a block's K loop does not wait one memory
// round trip per tile.  Tiles keep K contiguous (rows padded to 36 floats);
// thread (ty, tx) owns outputs (ty + 16 r, tx + 16 c), so the 16-byte shared
// loads of a quarter warp fall in distinct banks.  Every output still sums
// its K terms in increasing order with one fmaf each, starting from zero, as
// the plain form does, so both give the same bits.
constexpr int PBN = 64, PBK = 32, PST = 4, PLD = PBK + 4;
template <int PBM>
constexpr size_t pipe_smem() { return static_cast<size_t>(PST) * (PBM + PBN) * PLD * sizeof(float); }

__device__ __forceinline__ void cp_async16_zf(uint32_t dst, const void* src, bool valid) {
  const int n = valid ? 16 : 0;  // 0: the 16 bytes are zero-filled
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(n) : "memory");
}

// PBM rows per tile (64 or 32), 4 PBM threads; thread (ty, tx) owns outputs
// (ty + PBM/4 r, tx + 16 c).
template <int PHASE, int PBM>
__global__ void __launch_bounds__(4 * PBM) ffn_simt_pipe_kernel(FfnArgs a) {
  constexpr int NT = 4 * PBM, RS = PBM / 4;
  pdl_entry();
  const int N = PHASE == 1 ? a.F : a.D;
  const int K = PHASE == 1 ? a.D : a.F;
  // The group sizes, loaded at once, then this block's (group, m-tile).
  __shared__ int cnt_sm[kMaxExperts + 1];
  for (int gg = threadIdx.x; gg < a.G; gg += NT) cnt_sm[gg] = a.counts[gg];
  __syncthreads();
  int mt = blockIdx.y, g = -1, m0 = 0;
  for (int gg = 0; gg < a.G; ++gg) {
    const int tiles = (cnt_sm[gg] + PBM - 1) / PBM;
    if (mt < tiles) {
      g = gg;
      m0 = mt * PBM;
      break;
    }
    mt -= tiles;
  }
  if (g < 0) return;
  const int rows = cnt_sm[g];
  const int row0 = a.offsets[g];
  const int n0 = blockIdx.x * PBN;
  const float* A = static_cast<const float*>(PHASE == 1 ? a.xg : a.hmid);
  const float* B;
  if (g < a.E) {
    B = static_cast<const float*>(PHASE == 1 ? a.w1 : a.w2) + static_cast<size_t>(g) * a.F * a.D;
  } else {
    B = static_cast<const float*>(PHASE == 1 ? a.ws1 : a.ws2);
  }
  extern __shared__ __align__(16) float sm_pipe[];
  float* As = sm_pipe;                    // [PST][PBM][PLD]
  float* Bs = sm_pipe + PST * PBM * PLD;  // [PST][PBN][PLD]
  const int t = threadIdx.x, ty = t >> 4, tx = t & 15;
  // K tiles of this block: all of them, or split z of blockIdx.z (second
  // GEMM with K splits: whole tiles per split, partials written to a.partial).
  const int KTA = (K + PBK - 1) / PBK, S = gridDim.z, z = blockIdx.z;
  const int kt0 = z * KTA / S, KT = (z + 1) * KTA / S;
  // Stage st <- K tile kt: rows x PBK / 4 chunks of 4 floats per operand (A:
  // PBM rows, B: 64); chunks past K or past the rows are zeros.
  constexpr int CPR = PBK / 4;
  auto load = [&](int kt, int st) {
    const int k0 = kt * PBK;
#pragma unroll
    for (int c = t; c < PBM * CPR; c += NT) {
      const int r = c / CPR, kc = (c % CPR) * 4;
      const bool va = k0 + kc < K && m0 + r < rows;
      cp_async16_zf(smem_u32(As + (st * PBM + r) * PLD + kc),
                    va ? A + static_cast<size_t>(row0 + m0 + r) * K + k0 + kc : A, va);
    }
#pragma unroll
    for (int c = t; c < PBN * CPR; c += NT) {
      const int r = c / CPR, kc = (c % CPR) * 4;
      const bool vb = k0 + kc < K && n0 + r < N;
      cp_async16_zf(smem_u32(Bs + (st * PBN + r) * PLD + kc),
                    vb ? B + static_cast<size_t>(n0 + r) * K + k0 + kc : B, vb);
    }
  };
  float acc[4][4];
#pragma unroll
  for (int r = 0; r < 4; ++r)
#pragma unroll
    for (int c = 0; c < 4; ++c) acc[r][c] = 0.f;
#pragma unroll
  for (int st = 0; st < PST - 1; ++st) {
    if (kt0 + st < KT) load(kt0 + st, st);
    asm volatile("cp.async.commit_group;" ::: "memory");
  }
  for (int kt = kt0; kt < KT; ++kt) {
    asm volatile("cp.async.wait_group %0;" ::"n"(PST - 2) : "memory");
    __syncthreads();  // tile kt is in; every thread is done with tile kt - 1
    const int st = (kt - kt0) % PST;
    const float* as = As + st * PBM * PLD;
    const float* bs = Bs + st * PBN * PLD;
#pragma unroll
    for (int kk = 0; kk < PBK; kk += 4) {
      float4 av[4], bv[4];
#pragma unroll
      for (int r = 0; r < 4; ++r) av[r] = *reinterpret_cast<const float4*>(as + (ty + RS * r) * PLD + kk);
#pragma unroll
      for (int c = 0; c < 4; ++c) bv[c] = *reinterpret_cast<const float4*>(bs + (tx + 16 * c) * PLD + kk);
#pragma unroll
      for (int r = 0; r < 4; ++r)
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          acc[r][c] = fmaf(av[r].x, bv[c].x, acc[r][c]);
          acc[r][c] = fmaf(av[r].y, bv[c].y, acc[r][c]);
          acc[r][c] = fmaf(av[r].z, bv[c].z, acc[r][c]);
          acc[r][c] = fmaf(av[r].w, bv[c].w, acc[r][c]);
        }
    }
    // Refill the stage tile kt - 1 used.
    const int nk = kt + PST - 1;
    if (nk < KT) load(nk, (nk - kt0) % PST);
    asm volatile("cp.async.commit_group;" ::: "memory");
  }
  asm volatile("cp.async.wait_group 0;" ::: "memory");
#pragma unroll
  for (int r = 0; r < 4; ++r) {
    const int m = m0 + ty + RS * r;
    if (m >= rows) continue;
    const size_t row = static_cast<size_t>(row0 + m);
    if (PHASE == 1) {
      float* H = static_cast<float*>(a.hmid);
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const int n = n0 + tx + 16 * c;
        if (n < N) H[row * a.F + n] = gelu_f(acc[r][c], a.gelu_tanh);
      }
    } else if (S > 1) {
      float* P = a.partial + (static_cast<size_t>(z) * a.max_rows + row) * a.D;
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const int n = n0 + tx + 16 * c;
        if (n < N) P[n] = acc[r][c];
      }
    } else {
      const int dr = a.list[row];
      const int lim = g < a.E ? a.T * a.k : a.T;
      if (dr < 0 || dr >= lim) {
        report_status(a.status, kStatusBadIndex, 2000000 + static_cast<int>(row));
        continue;
      }
      float* dst = static_cast<float*>(g < a.E ? a.cache_h : a.shared_h);
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const int n = n0 + tx + 16 * c;
        if (n < N) dst[static_cast<size_t>(dr) * a.D + n] = acc[r][c];
      }
    }
  }
}

// The second GEMM's K splits added in split order, one warp per listed row
// (rows of group g are [offsets[g], offsets[g + 1])), into the row's cache
// slot or shared-expert row.
__global__ void __launch_bounds__(256) ffn_split_sum_kernel(FfnArgs a) {
  pdl_entry();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = a.G, E = a.E, S = a.simt_split;
  __shared__ int off_sm[kMaxExperts + 2];  // group offsets, read once
  for (int g = threadIdx.x; g <= G; g += blockDim.x) off_sm[g] = a.offsets[g];
  __syncthreads();
  const int rows = off_sm[G];
  const int nv = a.D / 4;
  for (int r = blockIdx.x * 8 + warp; r < rows; r += gridDim.x * 8) {
    int lo = 0, hi = G - 1;  // group of row r: the last g with offsets[g] <= r
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (off_sm[mid] <= r) lo = mid;
      else hi = mid - 1;
    }
    const int dr = a.list[r];
    const int lim = lo < E ? a.T * a.k : a.T;
    if (dr < 0 || dr >= lim) {
      if (lane == 0) report_status(a.status, kStatusBadIndex, 2000000 + r);
      continue;
    }
    float4* dst = reinterpret_cast<float4*>(static_cast<float*>(lo < E ? a.cache_h : a.shared_h) +
                                            static_cast<size_t>(dr) * a.D);
    const float4* P = reinterpret_cast<const float4*>(a.partial + static_cast<size_t>(r) * a.D);
    const size_t stride = static_cast<size_t>(a.max_rows) * nv;  // float4s per split
    for (int c = lane; c < nv; c += 32) {
      float4 v = P[c];
      for (int q = 1; q < S; ++q) {
        const float4 w = P[q * stride + c];
        v.x += w.x;
        v.y += w.y;
        v.z += w.z;
        v.w += w.w;
      }
      dst[c] = v;
    }
  }
}

#ifndef PIPE_BM1
#define PIPE_BM1 64
#endif
#ifndef PIPE_BM2
#define PIPE_BM2 32
#endif

// Plain launches: the grid covers the worst case, and its blocks launched
// early under a programmatic dependency would sit resident beside the
// previous kernel's blocks and slow them (measured: 455 vs 209 us per step
// of the fp32 workload).
template <typename TI>
cudaError_t launch_t(const FfnArgs& a, int phase, cudaStream_t s) {
  const int N = phase == 1 ? a.F : a.D;
  auto al16 = [](const void* p) { return reinterpret_cast<uintptr_t>(p) % 16 == 0; };
  if (std::is_same_v<TI, float> && a.D % 4 == 0 && a.F % 4 == 0 && al16(a.xg) && al16(a.hmid) && al16(a.w1) &&
      al16(a.w2) && al16(a.ws1) && al16(a.ws2)) {
    // The pipelined form (16-byte row chunks: K a multiple of 4 floats, aligned operands).
    auto run = [&](auto kern, int bm, size_t smem, int splits) -> cudaError_t {
      const cudaError_t e = set_dyn_smem_on_device(reinterpret_cast<const void*>(kern), static_cast<int>(smem));
      if (e != cudaSuccess) return e;
      const dim3 grid((N + PBN - 1) / PBN, (a.max_rows + bm - 1) / bm + a.G, splits);
      kern<<<grid, 4 * bm, smem, s>>>(a);
      return cudaGetLastError();
    };
    if (phase == 1) return run(ffn_simt_pipe_kernel<1, PIPE_BM1>, PIPE_BM1, pipe_smem<PIPE_BM1>(), 1);
    // The second GEMM has few outputs and a long K: K splits give the SMs
    // more warps, and a second pass adds the splits in order.
    const int splits = a.partial && a.simt_split > 1 && a.D % 4 == 0 ? a.simt_split : 1;
    const cudaError_t e = run(ffn_simt_pipe_kernel<2, PIPE_BM2>, PIPE_BM2, pipe_smem<PIPE_BM2>(), splits);
    if (e != cudaSuccess || splits == 1) return e;
    ffn_split_sum_kernel<<<(a.max_rows + 7) / 8, 256, 0, s>>>(a);
    return cudaGetLastError();
  }
  const dim3 grid((N + BN - 1) / BN, (a.max_rows + BM - 1) / BM + a.G);
  if (phase == 1) ffn_simt_kernel<TI, 1><<<grid, 256, 0, s>>>(a);
  else ffn_simt_kernel<TI, 2><<<grid, 256, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_ffn_simt(const FfnArgs& a, bool bf16, int phase, cudaStream_t s) {
  return bf16 ? launch_t<__nv_bfloat16>(a, phase, s) : launch_t<float>(a, phase, s);
}

}  // namespace moeca
