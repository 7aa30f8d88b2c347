// Tensor-core attention core of the DiT-MoE block (Sec. 4.1) for sm_103a:
// for the listed query rows of one sample and one head,
//   o = softmax(q k^T / sqrt(dh)) v      over all keys of the sample,
// bf16 operands, fp32 scores and accumulation, one pass over the keys with a
// running maximum and sum (online softmax).
//
// One CTA per (128 query rows, sample, head), 10 warps (320 threads):
//   warp 0    TMA producers: lane 0 loads the q tile once, then per block of
//             128 keys the k block (K-major, 128-byte swizzle) into a ring of
//             two or three, freed as soon as q k^T has read it; lane 1 loads
//             the v^T block (channels x keys, K-major for p v) into a ring of
//             three, freed by p v;
//   warp 1    allocates 512 TMEM columns and issues tcgen05.mma from one
//             thread: S_j = q k_j^T into one of two S buffers (columns 0-127,
//             128-255), then O += P_{j-1} v_{j-1} (columns 256 ..), so the
//             scores of block j are computed while block j-1's softmax runs;
//   warps 2-9 softmax, two warps per TMEM lane quadrant (warp % 4), each
//             thread one query row and one half (64 keys) of each block; the
//             two halves of a row exchange their maxima through shared
//             memory and a bounded barrier.  Per thread:
//             reads S_j from TMEM (tcgen05.ld), keeps the row maximum m in
//             base 2, rescales the O row in TMEM only when m rises by more
//             than 2^8 (tcgen05.ld / st), writes P_j = 2^(s - m) in bf16 back
//             into S_j's own TMEM columns (two values per column), where p v
//             reads it as its A operand, and at the end writes o = O / l.
// The row sum l comes from the tensor core: each v^T tile carries one more
// channel row of ones (and 15 rows of zeros to keep N a multiple of 16), so
// O's column DKP accumulates sum_k P[k], from the same rounded P as O and
// rescaled with it.
// q k^T contracts over dh rounded up to 16 (heads of 72 channels: 80, the
// q tile's columns 72-79 zeroed in shared memory); p v produces dh rounded
// up to 16 columns, of which the first dh are stored.
// Every wait is bounded (about one second); a wait that runs out records the
// timeout status, raises the CTA's abort flag, drains what was issued, frees
// TMEM and returns.
#include <cuda.h>

#include <cmath>

#include "common.cuh"
#include "kernels.h"
#include "tc_common.cuh"

namespace moeca {

namespace {

constexpr int kTQ = 128;        // query rows per CTA (MMA M)
constexpr int kTK = 128;        // keys per block (N of q k^T, K of p v)
constexpr int kTThreads = 320;  // warps 0-1 copy and issue, warps 2-9 softmax
constexpr int kSoftThreads = 256;
constexpr int kSubBytes = 128 * 128;  // one 128-row x 64-column bf16 sub-block (16 KB)

template <int DH>
struct TcAttnShape {
  static constexpr int DKP = (DH + 15) / 16 * 16;   // q k^T contraction and p v width
  static constexpr int QSUB = (DKP + 63) / 64;      // 64-column sub-blocks of q and k rows
  static constexpr int KSTEPS = DKP / 16;           // MMAs of q k^T per block
  static constexpr int QBYTES = QSUB * kSubBytes;   // q tile
  static constexpr int KBYTES = QSUB * kSubBytes;   // k block: 128 keys
  static constexpr int NV = DKP + 16;               // p v width: the channels, then the ones row
  static constexpr int VSUB = NV * 128;             // v^T sub-block: NV rows x 64 keys
  static constexpr int VBYTES = 2 * VSUB;           // v^T block: 128 keys
  static constexpr int V_TX = 2 * DKP * 128;        // bytes TMA writes per v^T block
  // Separate rings: a k block is free once q k^T has used it, a v^T block
  // once p v has.  A strided v^T box takes about 2.7 us to land, so v^T runs
  // three blocks ahead; k three if that still fits, else two (a k block is
  // needed one softmax earlier but freed one p v earlier).
  static constexpr int NV_ST = 3;
  static constexpr int NK = QBYTES + 3 * KBYTES + NV_ST * VBYTES <= 212 * 1024 ? 3 : 2;
  static constexpr size_t SMEM = static_cast<size_t>(QBYTES) + NK * KBYTES + NV_ST * VBYTES + 1024;
};

__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t* v) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]),
        "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t* v) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
      "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16};"
      ::"r"(taddr), "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]),
        "r"(v[8]), "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15])
      : "memory");
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t* v) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
      "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, "
      "%17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};"
      ::"r"(taddr), "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]),
        "r"(v[8]), "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15]),
        "r"(v[16]), "r"(v[17]), "r"(v[18]), "r"(v[19]), "r"(v[20]), "r"(v[21]), "r"(v[22]), "r"(v[23]),
        "r"(v[24]), "r"(v[25]), "r"(v[26]), "r"(v[27]), "r"(v[28]), "r"(v[29]), "r"(v[30]), "r"(v[31])
      : "memory");
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

// D (TMEM) += A (TMEM, M rows on the lanes, K packed two bf16 per column) x B (shared memory).
__device__ __forceinline__ void mma_bf16_ta(uint32_t d_tmem, uint32_t a_tmem, uint64_t b, uint32_t idesc, uint32_t acc) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n}"
      ::"r"(d_tmem), "r"(a_tmem), "l"(b), "r"(idesc), "r"(acc)
      : "memory");
}

__device__ __forceinline__ float ex2f_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t pack2(float lo, float hi) {
  __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&h);
}

// Bounded wait on a barrier phase that no one may abort (draining).
__device__ __forceinline__ void drain_wait(uint32_t bar, uint32_t parity) {
  const unsigned long long t0 = globaltimer();
  while (!mbar_try(bar, parity) && globaltimer() - t0 < kTcWaitNs) {
  }
}

struct TcAttnParams {
  int T, D, S;
  const int32_t* rows;       // list of query tokens, or null (all tokens)
  const int32_t* sample_lo;  // with rows: sample b's rows are [sample_lo[b], sample_lo[b + 1])
  __nv_bfloat16* o;          // [rows, D]
  float scale_log2;          // log2(e) / sqrt(dh)
  int* status;
};


// All lanes of a warp take the same branch after a wait (tcgen05.ld / st
// are warp-collective): the warp proceeds only if every lane's wait ended.
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag) {
  return __all_sync(0xffffffffu, mbar_wait(bar, parity, abort_flag));
}

template <int DH>
__global__ void __launch_bounds__(kTThreads, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap qmap, const __grid_constant__ CUtensorMap kmap,
                   const __grid_constant__ CUtensorMap vmap, const TcAttnParams p) {
  using Sh = TcAttnShape<DH>;
  constexpr int NK = Sh::NK, NVS = Sh::NV_ST;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t q_full, q_ready, p_full, drain_bar;
  __shared__ __align__(8) uint64_t o_done[2];  // p v of block j completes a phase of o_done[j & 1]
  __shared__ __align__(8) uint64_t s_full[2], max_bar[2];
  __shared__ __align__(8) uint64_t k_full[NK], k_empty[NK], v_full[NVS], v_empty[NVS];
  __shared__ int s_issued[2];  // k and v^T blocks each producer lane issued (for the drain)
  __shared__ float s_max[2][2][kTQ];  // [block parity][key half][row]: partial row maxima
  __shared__ uint32_t tmem_sh;
  __shared__ volatile int abort_flag;

  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = smem;
  uint8_t* sK = smem + Sh::QBYTES;          // k ring: NK blocks of KBYTES
  uint8_t* sV = sK + NK * Sh::KBYTES;        // v^T ring: NVS blocks of VBYTES
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int b = blockIdx.y, h = blockIdx.z;
  const int S = p.S, key0 = b * S;

  if (threadIdx.x == 0) {
    abort_flag = 0;
    mbar_init(smem_u32(&q_full), 1);
    mbar_init(smem_u32(&q_ready), kSoftThreads);
    mbar_init(smem_u32(&p_full), kSoftThreads);
    mbar_init(smem_u32(&o_done[0]), 1);
    mbar_init(smem_u32(&o_done[1]), 1);
    mbar_init(smem_u32(&drain_bar), 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&s_full[i]), 1);
      mbar_init(smem_u32(&max_bar[i]), kSoftThreads);
    }
    for (int i = 0; i < NK; ++i) {
      mbar_init(smem_u32(&k_full[i]), 1);
      mbar_init(smem_u32(&k_empty[i]), 1);
    }
    for (int i = 0; i < NVS; ++i) {
      mbar_init(smem_u32(&v_full[i]), 1);
      mbar_init(smem_u32(&v_empty[i]), 1);
    }
    s_issued[0] = s_issued[1] = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&qmap)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&kmap)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&vmap)) : "memory");
  }
  pdl_entry();
  int lo = key0, hi = key0 + S;
  if (p.rows) {
    lo = p.sample_lo[b];
    hi = p.sample_lo[b + 1];
  }
  const int r0 = lo + blockIdx.x * kTQ;
  if (r0 >= hi) return;  // uniform over the CTA, before TMEM is taken
  const int nq = min(kTQ, hi - r0);
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&tmem_sh)),
                 "r"(512)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    tc_fence_before();
  }
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_sh;
  const int nkb = (S + kTK - 1) / kTK;
  if (warp == 0) {
    // Lane 0 fills the k ring (and loads q first), lane 1 the v^T ring; the
    // two lanes run independent loops.
    if (lane == 0) {
      mbar_expect_tx(smem_u32(&q_full), Sh::QBYTES);
      for (int sub = 0; sub < Sh::QSUB; ++sub)
        tma_load_2d(smem_u32(sQ + sub * kSubBytes), &qmap, h * DH + sub * 64, r0, smem_u32(&q_full));
      int n = 0;
      for (int j = 0; j < nkb; ++j) {
        const int s = j % NK;
        if (j >= NK && !mbar_wait(smem_u32(&k_empty[s]), ((j / NK) - 1) & 1, &abort_flag)) {
          if (!abort_flag) report_status(p.status, kStatusWaitTimeout, 700);
          abort_flag = 1;
          break;
        }
        const uint32_t bar = smem_u32(&k_full[s]);
        mbar_expect_tx(bar, Sh::KBYTES);
        for (int sub = 0; sub < Sh::QSUB; ++sub)
          tma_load_2d(smem_u32(sK + s * Sh::KBYTES + sub * kSubBytes), &kmap, h * DH + sub * 64, key0 + j * kTK, bar);
        ++n;
      }
      s_issued[0] = n;
    } else if (lane == 1) {
      int n = 0;
      for (int j = 0; j < nkb; ++j) {
        const int s = j % NVS;
        if (j >= NVS && !mbar_wait(smem_u32(&v_empty[s]), ((j / NVS) - 1) & 1, &abort_flag)) {
          if (!abort_flag) report_status(p.status, kStatusWaitTimeout, 703);
          abort_flag = 1;
          break;
        }
        const uint32_t bar = smem_u32(&v_full[s]);
        mbar_expect_tx(bar, Sh::V_TX);
        for (int sub = 0; sub < 2; ++sub)
          tma_load_2d(smem_u32(sV + s * Sh::VBYTES + sub * Sh::VSUB), &vmap, key0 + j * kTK + sub * 64, h * DH, bar);
        ++n;
      }
      s_issued[1] = n;
    }
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t id_s = instr_desc(kTQ, kTK), id_o = instr_desc(kTQ, Sh::NV);
      const uint32_t t_o = tmem + 256;
      bool ok = mbar_wait(smem_u32(&q_ready), 0, &abort_flag);
      // O += P_j v_j, then free block j's stage.
      auto pv = [&](int j) -> bool {
        if (!mbar_wait(smem_u32(&p_full), j & 1, &abort_flag) ||
            !mbar_wait(smem_u32(&v_full[j % NVS]), (j / NVS) & 1, &abort_flag))
          return false;
        tc_fence_after();
        // P_j sits in S_j's TMEM columns, two bf16 per column: 8 columns per 16 keys.
        const uint32_t pa = tmem + (j & 1) * kTK;
        const uint32_t vb = smem_u32(sV + (j % NVS) * Sh::VBYTES);
#pragma unroll
        for (int kk = 0; kk < kTK / 16; ++kk) {
          const int sub = kk >> 2, off = (kk & 3) * 32;
          mma_bf16_ta(t_o, pa + kk * 8, smem_desc(vb + sub * Sh::VSUB + off), id_o, (j > 0) || (kk > 0));
        }
        mma_commit(smem_u32(&o_done[j & 1]));
        mma_commit(smem_u32(&v_empty[j % NVS]));
        return true;
      };
      for (int j = 0; ok && j < nkb; ++j) {
        const int s = j % NK, bb = j & 1;
        // S_j overwrites S_{j-2} / P_{j-2}: p v of block j-2 was issued
        // before this, and MMAs of one thread run in issue order.
        if (!mbar_wait(smem_u32(&k_full[s]), (j / NK) & 1, &abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t qa = smem_u32(sQ), kb = smem_u32(sK + s * Sh::KBYTES);
#pragma unroll
        for (int kk = 0; kk < Sh::KSTEPS; ++kk) {
          const int sub = kk >> 2, off = (kk & 3) * 32;
          mma_bf16(tmem + bb * kTK, smem_desc(qa + sub * kSubBytes + off), smem_desc(kb + sub * kSubBytes + off),
                   id_s, kk > 0);
        }
        mma_commit(smem_u32(&s_full[bb]));
        mma_commit(smem_u32(&k_empty[s]));  // q k^T has read k block j
        if (j >= 1 && !pv(j - 1)) ok = false;
      }
      if (ok && !pv(nkb - 1)) ok = false;
      if (!ok) {
        if (!abort_flag) report_status(p.status, kStatusWaitTimeout, 701);
        abort_flag = 1;
      }
      // Every MMA issued so far has completed once the drain barrier fires.
      mma_commit(smem_u32(&drain_bar));
      drain_wait(smem_u32(&drain_bar), 0);
    }
  } else {
    // ---- softmax: one query row and one key half per thread
    const int quad = warp & 3;
    const int half = (warp - 2) >> 2;  // keys [half 64, half 64 + 64) of each block
    const int r = quad * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
    const uint32_t t_o = tmem + lane_off + 256;
    constexpr int NCH = Sh::NV / 16;      // O chunks of 16 columns (the row sum's included)
    constexpr int C0 = (NCH + 1) / 2;     // half 0 rescales / stores chunks [0, C0), half 1 the rest
    const int cb = half ? C0 : 0, ce = half ? NCH : C0;
    const float sc = p.scale_log2;
    // The ones row (channel DKP) and 15 zero rows after each v^T sub-block's
    // channels; TMA never writes them.  Rows DKP.. start an 8-row swizzle
    // group, and a row of equal chunks is the same under any chunk swizzle.
    for (int idx = threadIdx.x - 64; idx < NVS * 2 * 16 * 8; idx += kSoftThreads) {
      const int row = idx >> 3, ch = idx & 7;  // row over (stage, sub-block, 16 rows)
      const int sv = row >> 4, rr = row & 15;
      uint8_t* base = sV + (sv >> 1) * Sh::VBYTES + (sv & 1) * Sh::VSUB + (Sh::DKP + rr) * 128;
      const uint32_t one2 = 0x3F803F80u;       // two bf16 1.0
      *reinterpret_cast<uint4*>(base + ch * 16) =
          rr == 0 ? make_uint4(one2, one2, one2, one2) : make_uint4(0, 0, 0, 0);
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    bool ok = warp_wait(smem_u32(&q_full), 0, &abort_flag);
    if (ok && Sh::DKP > DH && half == 0) {
      // The q tile's columns DH .. DKP-1 hold the next head's values: zero
      // them so they add nothing to q k^T (k's columns there are finite).
#pragma unroll
      for (int cidx = DH / 8; cidx < Sh::DKP / 8; ++cidx) {
        const int sub = cidx >> 3, ch = cidx & 7;
        *reinterpret_cast<uint4*>(sQ + sub * kSubBytes + r * 128 + ((ch ^ (r & 7)) << 4)) = make_uint4(0, 0, 0, 0);
      }
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    mbar_arrive(smem_u32(&q_ready));
    float m = -INFINITY;  // this row's reference maximum (scaled, base 2)
    // Completions of each o_done barrier are observed in order.  At block j
    // the latest p v that can have completed is block j-1's, so neither
    // barrier is ever more than one completion past its next wait (no
    // parity aliasing).
    int obs[2] = {0, 1};  // next unobserved p v block of each parity
    auto wait_pv = [&](int i) -> bool {  // p v of block i complete
      if (i < 0) return true;
      const int b2 = i & 1;
      while (obs[b2] <= i) {
        if (!warp_wait(smem_u32(&o_done[b2]), (obs[b2] >> 1) & 1, &abort_flag)) return false;
        obs[b2] += 2;
      }
      tc_fence_after();
      return true;
    };
    for (int j = 0; ok && j < nkb; ++j) {
      const int bb = j & 1;
      if (!warp_wait(smem_u32(&s_full[bb]), (j >> 1) & 1, &abort_flag)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t t_s = tmem + lane_off + bb * kTK + half * 64;
      const int nvalid = S - j * kTK - half * 64;  // keys of this half inside the sample (may be <= 0)
      const bool full = nvalid >= 64;              // warp-uniform
      uint32_t sv[64];                             // this half's scores, kept for pass 2
      tmem_ld32(t_s, sv);
      tmem_ld32(t_s + 32, sv + 32);
      float mx = -INFINITY;
      if (full) {
#pragma unroll
        for (int q = 0; q < 64; ++q) mx = fmaxf(mx, __uint_as_float(sv[q]));
      } else {
#pragma unroll
        for (int q = 0; q < 64; ++q)
          if (q < nvalid) mx = fmaxf(mx, __uint_as_float(sv[q]));
      }
      // Exchange with the other half of the row; past this point both halves
      // have read S_j, so P_j may overwrite it.
      s_max[bb][half][r] = mx;
      tc_fence_before();
      mbar_arrive(smem_u32(&max_bar[bb]));
      if (!warp_wait(smem_u32(&max_bar[bb]), (j >> 1) & 1, &abort_flag)) {
        ok = false;
        break;
      }
      tc_fence_after();
      mx = fmaxf(mx, s_max[bb][half ^ 1][r]);
      // The maximum is taken on raw scores and scaled once: rounding is
      // monotonic, so fl(max s * sc) is the maximum of the fl(s * sc) that
      // pass 2 forms (no fused multiply-add).
      const float cand = fmaxf(m, __fmul_rn(mx, sc));
      // Lazy rescaling: the reference maximum moves (and O is rescaled) only
      // when some row of the warp rises by more than 2^8; otherwise P keeps
      // the old reference and stays below 2^8.  The rows of a warp are the
      // same in both halves, so both take the same decision.
      if (j == 0) {
        m = cand;
      } else if (__any_sync(0xffffffffu, cand > m + 8.f)) {
        if (!wait_pv(j - 2) || !wait_pv(j - 1)) {  // O is quiet: p v of every earlier block done
          ok = false;
          break;
        }
        const float alpha = ex2f_approx(m - cand);
        for (int c = cb; c < ce; ++c) {
          uint32_t v[16];
          tmem_ld16(t_o + c * 16, v);
#pragma unroll
          for (int q = 0; q < 16; ++q) v[q] = __float_as_uint(__uint_as_float(v[q]) * alpha);
          tmem_st16(t_o + c * 16, v);
        }
        m = cand;
      }
      // Keep the o_done observations in step: block j-2's p v finished long ago.
      if (!wait_pv(j - 2)) {
        ok = false;
        break;
      }
      // P_j = 2^(s sc - m) in bf16, packed two per column into S_j's own
      // columns: this half's 64 keys are columns [half 32, half 32 + 32).
      uint32_t pk[32];
#pragma unroll
      for (int q = 0; q < 32; ++q) {
        float p0 = ex2f_approx(__fmul_rn(__uint_as_float(sv[2 * q]), sc) - m);
        float p1 = ex2f_approx(__fmul_rn(__uint_as_float(sv[2 * q + 1]), sc) - m);
        if (!full) {
          p0 = 2 * q < nvalid ? p0 : 0.f;
          p1 = 2 * q + 1 < nvalid ? p1 : 0.f;
        }
        pk[q] = pack2(p0, p1);
      }
      tmem_st32(tmem + lane_off + bb * kTK + half * 32, pk);
      tc_fence_before();
      mbar_arrive(smem_u32(&p_full));
    }
    if (ok && (!wait_pv(nkb - 2) || !wait_pv(nkb - 1))) ok = false;
    if (ok) {
      uint32_t lv[16];
      tmem_ld16(t_o + Sh::DKP, lv);  // column DKP: the row sum l
      const float inv_l = 1.f / __uint_as_float(lv[0]);
      __nv_bfloat16* dst = p.o + static_cast<size_t>(r0 + r) * p.D + h * DH;
      for (int c = cb; c < ce; ++c) {
        if (c * 16 >= DH) break;        // warp-uniform: the row-sum chunk is not stored
        uint32_t v[16];
        tmem_ld16(t_o + c * 16, v);     // every lane: the load is warp-collective
        if (r < nq) {
#pragma unroll
          for (int hh = 0; hh < 2; ++hh) {
            const int col = c * 16 + hh * 8;
            if (col < DH) {
              uint4 w;
              w.x = pack2(__uint_as_float(v[hh * 8 + 0]) * inv_l, __uint_as_float(v[hh * 8 + 1]) * inv_l);
              w.y = pack2(__uint_as_float(v[hh * 8 + 2]) * inv_l, __uint_as_float(v[hh * 8 + 3]) * inv_l);
              w.z = pack2(__uint_as_float(v[hh * 8 + 4]) * inv_l, __uint_as_float(v[hh * 8 + 5]) * inv_l);
              w.w = pack2(__uint_as_float(v[hh * 8 + 6]) * inv_l, __uint_as_float(v[hh * 8 + 7]) * inv_l);
              *reinterpret_cast<uint4*>(dst + col) = w;
            }
          }
        }
      }
    } else if (lane == 0) {
      if (!abort_flag) report_status(p.status, kStatusWaitTimeout, 702);
      abort_flag = 1;
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0 && lane == 0 && abort_flag) {
    // Copies issued but never consumed still land in shared memory.
    drain_wait(smem_u32(&q_full), 0);
    const int nk_iss = s_issued[0], nv_iss = s_issued[1];
    for (int s = 0; s < NK && s < nk_iss; ++s) {
      const int last = nk_iss - 1 - ((nk_iss - 1 - s) % NK);  // newest block issued on stage s
      drain_wait(smem_u32(&k_full[s]), (last / NK) & 1);
    }
    for (int s = 0; s < NVS && s < nv_iss; ++s) {
      const int last = nv_iss - 1 - ((nv_iss - 1 - s) % NVS);
      drain_wait(smem_u32(&v_full[s]), (last / NVS) & 1);
    }
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(512) : "memory");
  }
}


template <int DH>
cudaError_t run_attn_tc(const AttnArgs& a, cudaStream_t s) {
  using Sh = TcAttnShape<DH>;
  CUtensorMap qm, km, vm;
  if (!encode_2d(&qm, a.q, static_cast<uint64_t>(a.T), static_cast<uint64_t>(a.D), kTQ) ||
      !encode_2d(&km, a.k, static_cast<uint64_t>(a.T), static_cast<uint64_t>(a.D), kTK) ||
      !encode_2d(&vm, a.vt, static_cast<uint64_t>(a.D), static_cast<uint64_t>(a.T), Sh::DKP))
    return cudaErrorInvalidValue;
  TcAttnParams p{};
  p.T = a.T; p.D = a.D; p.S = a.S; p.rows = a.rows; p.sample_lo = a.sample_lo;
  p.o = static_cast<__nv_bfloat16*>(a.o);
  p.scale_log2 = 1.4426950408889634f / std::sqrt(static_cast<float>(DH));
  p.status = a.status;
  cudaError_t e = cudaFuncSetAttribute(attn_tc_kernel<DH>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(Sh::SMEM));
  if (e != cudaSuccess) return e;
  const dim3 grid((a.S + kTQ - 1) / kTQ, a.T / a.S, a.H);
  return launch_pdl(attn_tc_kernel<DH>, grid, dim3(kTThreads), Sh::SMEM, s, qm, km, vm, p);
}

}  // namespace

cudaError_t launch_attn_tc(const AttnArgs& a, cudaStream_t s) {
  if (!attn_supported(a.D, a.H) || a.S < 1 || a.S % 8 || a.T % a.S) return cudaErrorInvalidValue;
  switch (a.D / a.H) {
    case 64: return run_attn_tc<64>(a, s);
    case 72: return run_attn_tc<72>(a, s);
    case 80: return run_attn_tc<80>(a, s);
    case 96: return run_attn_tc<96>(a, s);
    default: return run_attn_tc<128>(a, s);
  }
}

}  // namespace moeca
