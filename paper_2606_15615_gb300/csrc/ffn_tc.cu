// Tensor-core grouped expert FFN (bf16 operands, fp32 accumulation) for sm_103a.
//
// Computes the recompute branches of Eq. 5 / Eq. 6 over the compacted rows:
//   phase 1: hmid[r, :] = GELU(xg[r, :] W1_g^T)         N = F, K = D
//   phase 2: dst[list[r], :] = hmid[r, :] W2_g^T         N = D, K = F
// where rows r of expert group g are [offsets[g], offsets[g] + counts[g]) and
// dst is the branch cache (token*k + slot) or the shared-expert rows.
//
// Persistent kernel, one CTA per SM, 10 warps:
//   warp 0  TMA producer: 128 x 64 A tile and BN x 64 weight tile per stage,
//           128-byte swizzle, into a 192 KB shared-memory ring (4-8 stages);
//   warp 1  allocates 512 TMEM columns and issues tcgen05.mma (M = 128,
//           N = BN, K = 16) from one thread; tcgen05.commit frees each stage
//           and signals a finished accumulator;
//   warps 2-9  epilogue, two warps per TMEM lane quadrant (each takes half of
//           the columns): tcgen05.ld, GELU / bf16
//           rounding, row stores (phase 2 scatters through the row list).
// Two TMEM accumulators (2 x BN columns) let the epilogue of one tile overlap
// the MMAs of the next.  Tiles run group by group, n-tile major and m-tile
// minor, so CTAs working at the same time share weight tiles through L2.
// Group sizes stay on the device: every CTA derives the tile list from them.
//
// Every mbarrier wait is bounded (about one second of %globaltimer); a wait
// that runs out records MOECA's timeout status, raises a CTA-wide abort flag,
// drains the copies and MMAs this CTA issued, frees TMEM and returns.
#include <cuda.h>
#include <algorithm>
#include <cstdio>
#include <vector>

#include "common.cuh"
#include "kernels.h"
#include "tc_common.cuh"

namespace moeca {

namespace {

constexpr int kBM = 128;          // rows per tile (MMA M)
constexpr int kBK = 64;           // K per sub-block: 64 bf16 = one 128-byte swizzle row
constexpr int kMaxBN = 256;
constexpr int kMaxStages = 8;
constexpr int kRingBytes = 4 * (16384 + 256 * 128);  // 192 KB of stages, any tile width
constexpr int kThreads = 320;
constexpr int kEpiThreads = 256;  // warps 2-9
constexpr int kTmemCols = 512;
constexpr int kABytes = kBM * kBK * 2;        // 16 KB: one A sub-block
constexpr int kStageOut = 32 * 64;  // per epilogue warp: 32 rows x 32 bf16 columns
constexpr int kSmemBytes = kRingBytes + 8 * kStageOut + 1024;
constexpr int kMaxGroups = kMaxExperts + 1;
constexpr unsigned long long kWaitNs = 1000000000ull;
constexpr int kMaxSplit = 4;
constexpr int kPlanTab = 512;     // plan entries by m-tile count kept in shared memory
constexpr int kUQ = 4;            // unit queue from the producer to the MMA and epilogue roles

// Stage geometry of one phase at one candidate tile width, fixed per handle.
// A stage holds `sub` K sub-blocks of 64: sub x (A 128 x 64 | B BN x 64),
// A sub-blocks first.  Wider stages mean fewer ring round trips per byte.
struct TcShape {
  int BN;           // tile width (0 = candidate absent)
  int nt;           // N / BN
  int KB;           // stages along K: K / (64 sub)
  int sub;          // K sub-blocks per stage (1 or 2)
  int stage_bytes;  // sub x (16 KB + BN x 128)
  int nst;          // stages in the ring
  uint64_t nt_magic;  // floor(2^32 / nt) + 1: (n x magic) >> 32 is n / nt for n < 2^32 / nt
};

struct TcArgs {
  int G, E, k, T, gelu_tanh;
  int first, last;   // GEMM phases of this launch: 1..1, 2..2, or 1..2 (both, fused)
  int N[2];          // per phase: output width
  TcShape shp[2][3]; // per phase and candidate width
  const int* plan_tab;  // packed plans by m-tile count, [3][tab_n]: fused, phase 1 alone, phase 2 alone
  int tab_n;
  const int32_t* counts;
  const int32_t* offsets;
  const int32_t* list;
  void* hmid;      // phase 1 output [rows, F]
  void* cache_h;   // phase 2 routed destination [T*k, D]
  void* shared_h;  // phase 2 shared destination [T, D]
  float* partial;  // split-K partial tiles, [max_units][128][BN] fp32
  int* tile_sem;   // split-K arrival counters, [max_units], left at 0
  int* dep;        // fused launch: per (m-tile, phase-2 split) {phase-1 tiles stored, phase-2 units started}, left at 0
  int dep_pairs;   // capacity of dep (pairs); pair (mi, q) is at mi x 4 + q
  int* work;       // next unit ticket (units past each CTA's first go to whoever asks); the kernel
                   // after this one re-arms it to 0 (launch_ffn_tc's contract)
  int gather;      // phase 1: A rows gathered from the layer input by token (tile::gather4)
  int* status;
};

// Plan word: tile-width index of phase 1 (bits 0-3) and phase 2 (4-7), K splits (8-11).
__host__ __device__ constexpr int plan_word(int bi0, int bi1, int S) { return bi0 | (bi1 << 4) | (S << 8); }

// Weight and activation tensor maps of one phase: A (activation rows) and,
// for each candidate width, B (routed experts) and Bs (shared expert).
struct alignas(64) TcMaps {
  CUtensorMap a;
  CUtensorMap b[3];
  CUtensorMap bs[3];
};
struct TcMapPair {
  TcMaps p[2];
};

// Four rows (one 128-byte box column each) gathered by row index; the map's
// box is 64 x 1.  They land as 4 consecutive 128-byte rows at dst.
__device__ __forceinline__ void tma_gather4(uint32_t dst, const CUtensorMap* map, int col, int r0, int r1, int r2,
                                            int r3, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cta.global.tile::gather4.mbarrier::complete_tx::bytes "
      "[%0], [%1, {%2, %3, %4, %5, %6}], [%7];"
      ::"r"(dst), "l"(reinterpret_cast<uint64_t>(map)), "r"(col), "r"(r0), "r"(r1), "r"(r2), "r"(r3), "r"(bar)
      : "memory");
}

// Tanh-form GELU with the hardware tanh approximation (MUFU; relative error
// about 2^-11).  The result is rounded to bf16 (relative step 2^-8) right
// after, so the approximation stays below the output rounding.
__device__ __forceinline__ float gelu_tanh_hw(float z) {
  const float u = 0.7978845608028654f * fmaf(0.044715f * z, z * z, z);
  float t;
  asm("tanh.approx.f32 %0, %1;" : "=f"(t) : "f"(u));
  const float hz = 0.5f * z;
  return fmaf(hz, t, hz);
}

// One warp's 32 x 32 output chunk: lane i holds row i's 32 fp32 values.
// They go through GELU (phase 1) and bf16 rounding, then through a 2 KB
// shared-memory stage so that each global store writes 64 contiguous bytes
// of 8 rows (instead of 16 bytes of 32 rows).  `dst` is this lane's row at
// the chunk's first column, or null for a row that is not stored.  The stage
// is XOR-swizzled by row pairs so both of its accesses are conflict-free.
__device__ __forceinline__ void store_chunk(uint8_t* stage, __nv_bfloat16* dst, const uint32_t* v, bool gelu,
                                            int tanh_form, int lane) {
  uint32_t packed[16];
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    float x0 = __uint_as_float(v[2 * j]), x1 = __uint_as_float(v[2 * j + 1]);
    if (gelu) {
      x0 = tanh_form ? gelu_tanh_hw(x0) : gelu_f(x0, 0);
      x1 = tanh_form ? gelu_tanh_hw(x1) : gelu_f(x1, 0);
    }
    __nv_bfloat162 h2 = __floats2bfloat162_rn(x0, x1);
    packed[j] = *reinterpret_cast<uint32_t*>(&h2);
  }
#pragma unroll
  for (int j = 0; j < 4; ++j)
    *reinterpret_cast<uint4*>(stage + lane * 64 + ((j ^ ((lane >> 1) & 3)) << 4)) =
        make_uint4(packed[4 * j], packed[4 * j + 1], packed[4 * j + 2], packed[4 * j + 3]);
  __syncwarp();
  const unsigned long long mine = reinterpret_cast<unsigned long long>(dst);
#pragma unroll
  for (int it = 0; it < 4; ++it) {
    const int row = it * 8 + (lane >> 2), j = lane & 3;
    const uint4 val = *reinterpret_cast<const uint4*>(stage + row * 64 + ((j ^ ((row >> 1) & 3)) << 4));
    __nv_bfloat16* d = reinterpret_cast<__nv_bfloat16*>(__shfl_sync(0xffffffffu, mine, row));
    if (d) *reinterpret_cast<uint4*>(d + j * 8) = val;
  }
  __syncwarp();
}

// Shape of one phase for this launch, identical in every CTA.
struct PhaseShape {
  int BN, nt, KB, sub, stage_bytes, nst, S, units;
  uint64_t nt_magic;
};

__device__ __forceinline__ PhaseShape phase_shape(const TcArgs& a, int p, int bi, int S, int m_tiles) {
  const TcShape& t = a.shp[p][bi];
  PhaseShape r;
  r.BN = t.BN;
  r.nt = t.nt;
  r.KB = t.KB;
  r.sub = t.sub;
  r.stage_bytes = t.stage_bytes;
  r.nst = t.nst;
  r.S = S;
  r.units = m_tiles * t.nt * S;
  r.nt_magic = t.nt_magic;
  return r;
}

// One unit of work: phase p, tile (group g, m-tile m, n-tile n), K split sp.
// mi is the m-tile's index over all groups (the dependency slot).
struct Unit {
  int p, tile, sp, g, m, n, mi;
};

// Units of phase 0 come first, then those of phase 1.  Within a phase, tiles
// run m-tile major (groups in order) and n-tile minor: CTAs working at the
// same time share the A rows of an m-tile, and an expert's m-tiles, which
// read the same weight tiles, run close together.  Splits of a tile are a
// adjacent (consecutive CTAs), so the last of them to finish reduces soon.
__device__ __forceinline__ Unit decode_unit(int u, const PhaseShape& s0, const PhaseShape& s1, int U0,
                                            const int* mt_before, int G) {
  Unit r;
  r.p = u < U0 ? 0 : 1;
  const int v = u - (r.p ? U0 : 0);
  const int nt = r.p ? s1.nt : s0.nt;
  const int S = r.p ? s1.S : s0.S;
  if (S == 1) {
    r.tile = v;
    r.sp = 0;
  } else {
    r.tile = v / S;
    r.sp = v - r.tile * S;
  }
  r.mi = static_cast<int>((static_cast<uint64_t>(r.tile) * (r.p ? s1.nt_magic : s0.nt_magic)) >> 32);
  r.n = r.tile - r.mi * nt;
  // Last group whose first m-tile is at or before mi (empty groups precede
  // the non-empty group that shares their start).
  int lo = 0, hi = G - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (mt_before[mid] <= r.mi) lo = mid;
    else hi = mid - 1;
  }
  r.g = lo;
  r.m = r.mi - mt_before[lo];
  return r;
}

// First ring slot of the second phase of a fused launch: the one that starts
// at or after the end of the newest first-phase stage, so the first
// second-phase copies overwrite the oldest first-phase stages.
__device__ __forceinline__ int second_phase_first_slot(int issued0, const PhaseShape& s0, const PhaseShape& s1) {
  if (issued0 == 0) return 0;
  const int end = ((issued0 - 1) % s0.nst + 1) * s0.stage_bytes;
  return ((end + s1.stage_bytes - 1) / s1.stage_bytes) % s1.nst;
}

__device__ __forceinline__ int ld_acquire(const int* p) {
  int v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Bounded wait until *p >= target (another CTA's release).  False on timeout or abort.
__device__ __noinline__ bool wait_count(const int* p, int target, volatile int* abort_flag) {
  unsigned long long t0 = 0;
  for (uint32_t it = 1;; ++it) {
    if (ld_acquire(p) >= target) return true;
    if ((it & 15u) == 0) {
      if (*abort_flag) return false;
      const unsigned long long now = globaltimer();
      if (t0 == 0) t0 = now;
      else if (now - t0 > kWaitNs) return false;
    }
  }
}

__global__ void __launch_bounds__(kThreads, 1)
    ffn_tc_kernel(const __grid_constant__ TcMapPair maps, TcArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) uint64_t full_bar[2][kMaxStages];
  __shared__ __align__(8) uint64_t empty_bar[2][kMaxStages];
  __shared__ __align__(8) uint64_t tfull_bar[2];
  __shared__ __align__(8) uint64_t tempty_bar[2];
  __shared__ __align__(8) uint64_t drain_bar;
  __shared__ uint32_t tmem_base_sh;
  __shared__ int mt_before[kMaxGroups + 1];  // m-tiles ahead of each group; [G] = all
  __shared__ int cnt_sh[kMaxGroups];
  __shared__ int off_sh[kMaxGroups];
  __shared__ volatile int abort_flag;
  __shared__ int bi_sh[2], split_sh;
  __shared__ int plan_sh[kPlanTab];
  __shared__ int rows_sh[kBM];  // producer: token of each row of the current tile (gather)
  __shared__ volatile int ep_abort;
  __shared__ volatile int ep_last;
  __shared__ volatile int uq[kUQ];
  __shared__ __align__(8) uint64_t uq_full[kUQ];
  __shared__ __align__(8) uint64_t uq_empty[kUQ];

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = a.G;
  const int p_lo = a.first - 1, p_hi = a.last - 1;
  const bool fused = p_lo != p_hi;

  // Everything that does not read the previous kernel's output happens
  // before the programmatic-dependency wait: barriers, TMEM, map prefetch.
  if (threadIdx.x == 0) {
    abort_flag = 0;
    ep_abort = 0;
    for (int p = 0; p < 2; ++p) {
      for (int s = 0; s < kMaxStages; ++s) {
        mbar_init(smem_u32(&full_bar[p][s]), 1);
        mbar_init(smem_u32(&empty_bar[p][s]), 1);
      }
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(smem_u32(&tfull_bar[s]), 1);
      mbar_init(smem_u32(&tempty_bar[s]), kEpiThreads);
    }
    mbar_init(smem_u32(&drain_bar), 1);
    for (int q = 0; q < kUQ; ++q) {
      mbar_init(smem_u32(&uq_full[q]), 1);
      mbar_init(smem_u32(&uq_empty[q]), 2);  // the MMA thread and the epilogue leader
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;"
                 ::"r"(smem_u32(&tmem_base_sh)), "r"(kTmemCols) : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    tc_fence_before();
  }
  if (warp == 2 && lane < 14) {
    const TcMaps& m = maps.p[lane / 7];
    const int j = lane % 7;
    const CUtensorMap* t = j == 0 ? &m.a : (j < 4 ? &m.b[j - 1] : &m.bs[j - 4]);
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(t)) : "memory");
  }
  if (warp == 2) {
    // Bring the launch parameters into the constant cache while the previous
    // kernel finishes (the roles read them right after the wait).
    const TcShape& w = a.shp[lane / 3 & 1][lane % 3];
    asm volatile("" ::"r"(w.BN), "r"(w.nt), "r"(w.KB), "r"(w.sub), "r"(w.stage_bytes), "r"(w.nst), "l"(w.nt_magic));
    asm volatile("" ::"r"(a.N[lane & 1]), "l"(a.counts), "l"(a.list), "l"(a.hmid), "l"(a.dep), "l"(a.status),
                 "l"(a.cache_h), "r"(a.dep_pairs), "r"(a.gather), "l"(a.partial));
  }
  const int tab_n = min(a.tab_n, kPlanTab);
  if (warp == 0) {
    // This launch's plan table (it does not depend on the previous kernel).
    const int* tab = a.plan_tab + (fused ? 0 : a.first) * a.tab_n;
    for (int i = lane; i < tab_n; i += 32) plan_sh[i] = tab[i];
    __syncwarp();
  }
  pdl_entry();
  if (warp == 0) {
    // Group sizes, loaded by all lanes at once, and the m-tiles ahead of each group.
    int m_tiles = 0;
    for (int g0 = 0; g0 < G; g0 += 32) {
      const int g = g0 + lane;
      const int c = g < G ? a.counts[g] : 0;
      const int o = g < G ? a.offsets[g] : 0;
      const int mt = (c + kBM - 1) / kBM;
      int incl = mt;
#pragma unroll
      for (int d = 1; d < 32; d <<= 1) {
        const int v = __shfl_up_sync(0xffffffffu, incl, d);
        if (lane >= d) incl += v;
      }
      if (g < G) {
        cnt_sh[g] = c;
        off_sh[g] = o;
        mt_before[g] = m_tiles + incl - mt;
      }
      m_tiles += __shfl_sync(0xffffffffu, incl, 31);
    }
    if (lane == 0) {
      // Beyond the table, the largest tabulated count's widths, without splits.
      const int w = plan_sh[min(m_tiles, tab_n - 1)];
      mt_before[G] = m_tiles;
      bi_sh[0] = w & 15;
      bi_sh[1] = (w >> 4) & 15;
      split_sh = m_tiles >= tab_n ? 1 : (w >> 8) & 15;
      if (fused && m_tiles * kMaxSplit > a.dep_pairs) {
        report_status(a.status, kStatusBadIndex, 5000000 + m_tiles);
        abort_flag = 1;
      }
    }
  }
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base_sh;
  const int m_tiles = mt_before[G];
  // K splits apply to the launched phase alone, or to phase 2 of a fused launch.
  const PhaseShape s0 = phase_shape(a, 0, bi_sh[0], fused ? 1 : split_sh, m_tiles);
  const PhaseShape s1 = phase_shape(a, 1, bi_sh[1], split_sh, m_tiles);
  // Fused: phase-2 split q reads the hidden columns of phase-1 n-tiles
  // [q gq, (q + 1) gq); its dependency slot is (m-tile, q).
  const int gq = s0.nt / s1.S;
  const int U0 = p_lo == 0 ? s0.units : 0;
  const int total = abort_flag ? 0 : U0 + (p_hi == 1 ? s1.units : 0);

  if (warp == 0) {
    // ---------------- TMA producer (lane 0 issues; the warp fetches row indices) ----------------
    // Each phase has its own ring partition (slot size = its stage size) and
    // barriers; per-slot parity bits let the second phase start mid-ring.
    // A CTA's units run phase 0 first, so the state of the current phase
    // lives in (sl, par, used) and phase 0's is kept in (par0, used0).
    int cp = -1, sl = 0;
    uint32_t par = 0u, used = 0u;    // bit s: uses of slot s so far mod 2; slot s used at all
    uint32_t par0 = 0u, used0 = 0u;  // phase 0's, once phase 1 has begun
    int issued0 = 0;
    bool ok = true;
    // Units: blockIdx.x first, then tickets from the shared counter, in
    // increasing order (so phase 0 before phase 1 here too).  Each is passed
    // to the MMA and epilogue roles through the unit queue; -1 ends it.
    int qs = 0;
    uint32_t qpar = 0u;
    int u = static_cast<int>(blockIdx.x) < total ? static_cast<int>(blockIdx.x) : -1;
    for (;;) {
      if (lane == 0) {
        ok = mbar_wait(smem_u32(&uq_empty[qs]), qpar ^ 1u, &abort_flag);
        if (ok) {
          uq[qs] = u;
          mbar_arrive(smem_u32(&uq_full[qs]));
        }
      }
      if (++qs == kUQ) {
        qs = 0;
        qpar ^= 1u;
      }
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok || u < 0) break;
      const Unit t = decode_unit(u, s0, s1, U0, mt_before, G);
      const PhaseShape sh = t.p ? s1 : s0;
      if (t.p != cp) {
        if (cp == 0) {
          par0 = par;
          used0 = used;
          sl = second_phase_first_slot(issued0, s0, s1);
        } else {
          sl = 0;
        }
        par = 0u;
        used = 0u;
        cp = t.p;
      }
      const TcMaps& mp = maps.p[t.p];
      const int bsel = bi_sh[t.p];
      const CUtensorMap* tb = t.g < a.E ? &mp.b[bsel] : &mp.bs[bsel];
      const CUtensorMap* ta = &mp.a;
      const int brow = (t.g < a.E ? t.g * a.N[t.p] : 0) + t.n * sh.BN;
      const int arow = off_sh[t.g] + t.m * kBM;
      const int kb0 = sh.S == 1 ? 0 : t.sp * sh.KB / sh.S, kb1 = sh.S == 1 ? sh.KB : (t.sp + 1) * sh.KB / sh.S;
      const bool gather = a.gather && t.p == 0;
      if (gather) {
        // Token of each of the tile's 128 rows; rows past the group's end
        // repeat its first row (their results are never stored).
        const int valid = cnt_sh[t.g] - t.m * kBM;
#pragma unroll
        for (int j = 0; j < kBM / 32; ++j) {
          const int r = lane * (kBM / 32) + j;
          const int ent = a.list[arow + (r < valid ? r : 0)];
          int tok = t.g < a.E ? ent / a.k : ent;
          tok = tok < 0 ? 0 : (tok >= a.T ? a.T - 1 : tok);
          rows_sh[r] = tok;
        }
        __syncwarp();
      }
      if (lane == 0) {
        // Issue one stage: its weight half (B) and/or activation half (A).
        // A stage issued without A gets its A half later into the same slot
        // (the barrier already expects the whole stage).
        auto issue = [&](int kb, bool with_a, bool with_b, int slot) {
          uint8_t* sa = smem + slot * sh.stage_bytes;
          uint8_t* sb = sa + sh.sub * kABytes;
          const uint32_t fb = smem_u32(&full_bar[t.p][slot]);
          for (int j = 0; j < sh.sub; ++j) {
            const int x = (kb * sh.sub + j) * kBK;
            if (with_a) {
              if (gather) {
#pragma unroll 4
                for (int q = 0; q < kBM / 4; ++q)
                  tma_gather4(smem_u32(sa + j * kABytes + q * 512), ta, x, rows_sh[4 * q], rows_sh[4 * q + 1],
                              rows_sh[4 * q + 2], rows_sh[4 * q + 3], fb);
              } else {
                tma_load_2d(smem_u32(sa + j * kABytes), ta, x, arow, fb);
              }
            }
            if (with_b) tma_load_2d(smem_u32(sb + j * sh.BN * kBK * 2), tb, x, brow, fb);
          }
        };
        // Claim the next slot for a new stage: wait until it is free (and, on a
        // second-phase slot's first use, until the first-phase stages it
        // overlaps are consumed), arm its barrier for the whole stage.
        auto claim = [&]() -> bool {
          if (fused && t.p == 1 && !((used >> sl) & 1u)) {
            const int lo = sl * s1.stage_bytes / s0.stage_bytes;
            const int hi = min(((sl + 1) * s1.stage_bytes - 1) / s0.stage_bytes, s0.nst - 1);
            for (int q = lo; q <= hi; ++q)
              if (((used0 >> q) & 1u) &&
                  !mbar_wait(smem_u32(&empty_bar[0][q]), ((par0 >> q) & 1u) ^ 1u, &abort_flag))
                return false;
          }
          if (!mbar_wait(smem_u32(&empty_bar[t.p][sl]), ((par >> sl) & 1u) ^ 1u, &abort_flag)) return false;
          mbar_expect_tx(smem_u32(&full_bar[t.p][sl]), sh.stage_bytes);
          return true;
        };
        auto advance = [&]() {
          par ^= 1u << sl;
          used |= 1u << sl;
          if (t.p == 0) ++issued0;
          sl = sl + 1 == sh.nst ? 0 : sl + 1;
        };
        int pre = 0;
        if (fused && t.p == 1) {
          // The m-tile's hidden rows come from every phase-1 tile of it, stored
          // by other CTAs' epilogues with generic stores and read here by TMA.
          // While they are not all there, the weight halves of the first
          // stages (which do not depend on them) are already on their way.
          int* d = a.dep + 2 * (t.mi * kMaxSplit + t.sp);
          const int sl_pre = sl;
          if (ld_acquire(d) < gq) {
            const int P = min(sh.nst, kb1 - kb0);
            for (; pre < P && ok; ++pre) {
              ok = claim();
              if (ok) {
                issue(kb0 + pre, false, true, sl);
                advance();
              }
            }
          }
          if (ok && !wait_count(d, gq, &abort_flag)) ok = false;
          if (ok) {
            asm volatile("fence.proxy.async.global;" ::: "memory");
            // The last phase-2 unit to start on this m-tile re-arms its counters.
            if (atomicAdd(d + 1, 1) == s1.nt - 1) {
              d[0] = 0;
              d[1] = 0;
            }
            for (int j = 0; j < pre; ++j) {
              const int slot = (sl_pre + j) % sh.nst;
              issue(kb0 + j, true, false, slot);
            }
          }
        }
        for (int kb = kb0 + pre; kb < kb1 && ok; ++kb) {
          ok = claim();
          if (ok) {
            issue(kb, true, true, sl);
            advance();
          }
        }
      }
      ok = __shfl_sync(0xffffffffu, ok, 0);
      __syncwarp();
      if (!ok) break;
      int next = 0;
      if (lane == 0) next = static_cast<int>(gridDim.x) + atomicAdd(a.work, 1);
      next = __shfl_sync(0xffffffffu, next, 0);
      u = next < total ? next : -1;
    }
    if (!ok && lane == 0) {
      if (!abort_flag) report_status(a.status, kStatusWaitTimeout, 100 + a.first);
      abort_flag = 1;
      // Let the copies already issued land before the CTA can exit: wait for
      // the last use of every slot that was used.
      if (cp == 0) {
        par0 = par;
        used0 = used;
      }
      const uint32_t par1 = cp == 1 ? par : 0u, used1 = cp == 1 ? used : 0u;
      for (int p = 0; p < 2; ++p)
        for (int q = 0; q < kMaxStages; ++q)
          if ((((p ? used1 : used0)) >> q) & 1u) {
            const uint32_t ph = (((p ? par1 : par0) >> q) & 1u) ^ 1u;
            unsigned long long t0 = globaltimer();
            while (!mbar_try(smem_u32(&full_bar[p][q]), ph) && globaltimer() - t0 < kWaitNs) {
            }
          }
    }
  } else if (warp == 1 && lane == 0) {
    // ---------------- MMA issuer ----------------
    int cp = -1, sl = 0;
    uint32_t par = 0u;
    int consumed0 = 0;
    int acc = 0;
    uint32_t acc_phase = 0;
    bool ok = true;
    int qs = 0;
    uint32_t qpar = 0u;
    for (;;) {
      if (!mbar_wait(smem_u32(&uq_full[qs]), qpar, &abort_flag)) {
        ok = false;
        break;
      }
      const int u = uq[qs];
      mbar_arrive(smem_u32(&uq_empty[qs]));
      if (++qs == kUQ) {
        qs = 0;
        qpar ^= 1u;
      }
      if (u < 0) break;
      const Unit t = decode_unit(u, s0, s1, U0, mt_before, G);
      const PhaseShape sh = t.p ? s1 : s0;
      const int kb0 = sh.S == 1 ? 0 : t.sp * sh.KB / sh.S, kb1 = sh.S == 1 ? sh.KB : (t.sp + 1) * sh.KB / sh.S;
      const uint32_t idesc = instr_desc(kBM, sh.BN);
      if (t.p != cp) {
        sl = cp == 0 ? second_phase_first_slot(consumed0, s0, s1) : 0;
        par = 0u;
        cp = t.p;
      }
      if (!mbar_wait(smem_u32(&tempty_bar[acc]), acc_phase ^ 1u, &abort_flag)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t d_tmem = tmem + static_cast<uint32_t>(acc * kMaxBN);
      for (int kb = kb0; kb < kb1; ++kb) {
        if (!mbar_wait(smem_u32(&full_bar[t.p][sl]), (par >> sl) & 1u, &abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t sa = smem_u32(smem + sl * sh.stage_bytes);
        const uint32_t sb = sa + sh.sub * kABytes;
        for (int j = 0; j < sh.sub; ++j) {
#pragma unroll
          for (int kk = 0; kk < kBK / 16; ++kk) {
            mma_bf16(d_tmem, smem_desc(sa + j * kABytes + kk * 32), smem_desc(sb + j * sh.BN * kBK * 2 + kk * 32),
                     idesc, (kb != kb0) || j != 0 || kk != 0);
          }
        }
        mma_commit(smem_u32(&empty_bar[t.p][sl]));
        par ^= 1u << sl;
        if (t.p == 0) ++consumed0;
        sl = sl + 1 == sh.nst ? 0 : sl + 1;
      }
      if (!ok) break;
      mma_commit(smem_u32(&tfull_bar[acc]));
      if (++acc == 2) {
        acc = 0;
        acc_phase ^= 1u;
      }
    }
    if (!ok) {
      if (!abort_flag) report_status(a.status, kStatusWaitTimeout, 200 + a.first);
      abort_flag = 1;
    }
    // Every MMA this thread issued has completed once the drain barrier fires.
    mma_commit(smem_u32(&drain_bar));
    unsigned long long t0 = globaltimer();
    while (!mbar_try(smem_u32(&drain_bar), 0) && globaltimer() - t0 < kWaitNs) {
    }
  } else if (warp >= 2) {
    // ---------------- Epilogue ----------------
    // The 8 epilogue warps (256 threads) agree on every abort and every
    // split-K decision through named barrier 1, so none can wait alone.
    const int quad = warp & 3;         // TMEM lanes [32 quad, 32 quad + 32)
    const int half = (warp - 2) >> 2;  // which half of the tile's columns
    uint8_t* stage = smem + kRingBytes + (warp - 2) * kStageOut;  // this warp's store stage
    const int r = quad * 32 + lane;
    const bool leader = warp == 2 && lane == 0;
    int acc = 0;
    uint32_t acc_phase = 0;
    int qs = 0;
    uint32_t qpar = 0u;
    for (;;) {
      const bool gotq = __all_sync(0xffffffffu, mbar_wait(smem_u32(&uq_full[qs]), qpar, &abort_flag));
      const int u = uq[qs];
      if (!gotq && lane == 0) ep_abort = 1;
      asm volatile("bar.sync 1, 256;" ::: "memory");  // every epilogue thread has read the queue slot
      if (ep_abort) {
        if (leader && !abort_flag) report_status(a.status, kStatusWaitTimeout, 300 + a.first);
        abort_flag = 1;
        break;
      }
      if (leader) mbar_arrive(smem_u32(&uq_empty[qs]));
      if (++qs == kUQ) {
        qs = 0;
        qpar ^= 1u;
      }
      if (u < 0) break;
      const Unit t = decode_unit(u, s0, s1, U0, mt_before, G);
      const PhaseShape sh = t.p ? s1 : s0;
      const int BN = sh.BN, S = sh.S, N = a.N[t.p];
      const bool got = __all_sync(0xffffffffu, mbar_wait(smem_u32(&tfull_bar[acc]), acc_phase, &abort_flag));
      if (!got && lane == 0) ep_abort = 1;
      asm volatile("bar.sync 1, 256;" ::: "memory");
      if (ep_abort) {
        if (leader && !abort_flag) report_status(a.status, kStatusWaitTimeout, 300 + a.first);
        abort_flag = 1;
        break;
      }
      tc_fence_after();
      const int mrow = t.m * kBM + r;
      const bool live = mrow < cnt_sh[t.g];
      const size_t grow = static_cast<size_t>(off_sh[t.g]) + mrow;
      const int n0 = t.n * BN;
      __nv_bfloat16* dst = nullptr;
      if (live) {
        if (t.p == 0) {
          dst = static_cast<__nv_bfloat16*>(a.hmid) + grow * N + n0;
        } else {
          const int dr = a.list[grow];
          const int lim = t.g < a.E ? a.T * a.k : a.T;
          if (dr >= 0 && dr < lim) {
            dst = static_cast<__nv_bfloat16*>(t.g < a.E ? a.cache_h : a.shared_h) + static_cast<size_t>(dr) * N + n0;
          } else {
            report_status(a.status, kStatusBadIndex, 4000000 + static_cast<int>(grow));
          }
        }
      }
      const uint32_t tbase = tmem + (static_cast<uint32_t>(quad * 32) << 16) + static_cast<uint32_t>(acc * kMaxBN);
      const int nch = BN / 64;  // 32-column chunks per half
      const int c_lo = half * nch, c_hi = c_lo + nch;
      if (S == 1) {
        for (int c = c_lo; c < c_hi; ++c) {
          uint32_t v[32];
          tmem_ld32(tbase + c * 32, v);
          store_chunk(stage, dst ? dst + c * 32 : nullptr, v, t.p == 0, a.gelu_tanh, lane);
        }
        tc_fence_before();
        mbar_arrive(smem_u32(&tempty_bar[acc]));
        if (fused && t.p == 0) {
          // Publish this tile's hidden rows to the phase-2 units of its m-tile,
          // which read them through the async (TMA) proxy: every writer orders
          // its stores before later async-proxy accesses, the barrier collects
          // the writers, and one release add makes them visible with the count.
          asm volatile("fence.proxy.async.global;" ::: "memory");
          asm volatile("bar.sync 1, 256;" ::: "memory");
          if (leader)
            asm volatile("red.release.gpu.global.add.s32 [%0], 1;" ::"l"(a.dep + 2 * (t.mi * kMaxSplit + t.n / gq))
                         : "memory");
        }
      } else {
        // Split K: park this split's fp32 tile, free TMEM, then the last split
        // to arrive for the tile sums the splits in split order.  A parked
        // tile is laid out [32-column chunk][4-column group][row][4], so each
        // warp access covers 512 contiguous bytes.
        float4* mine = reinterpret_cast<float4*>(a.partial + (static_cast<size_t>(t.tile) * S + t.sp) * kBM * BN);
        for (int c = c_lo; c < c_hi; ++c) {
          uint32_t v[32];
          tmem_ld32(tbase + c * 32, v);
#pragma unroll
          for (int j = 0; j < 8; ++j)
            mine[(c * 8 + j) * kBM + r] = make_float4(__uint_as_float(v[4 * j]), __uint_as_float(v[4 * j + 1]),
                                                      __uint_as_float(v[4 * j + 2]), __uint_as_float(v[4 * j + 3]));
        }
        tc_fence_before();
        mbar_arrive(smem_u32(&tempty_bar[acc]));
        __threadfence();
        asm volatile("bar.sync 1, 256;" ::: "memory");
        if (leader) ep_last = atomicAdd(a.tile_sem + t.tile, 1) == S - 1;
        asm volatile("bar.sync 1, 256;" ::: "memory");
        if (ep_last) {
          __threadfence();
          const float4* base = reinterpret_cast<const float4*>(a.partial + static_cast<size_t>(t.tile) * S * kBM * BN);
          const size_t split_stride = static_cast<size_t>(kBM) * BN / 4;  // float4s per parked tile
          for (int c = c_lo; c < c_hi; ++c) {
            uint32_t v[32];
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              // All splits' 16 values in flight at once, then added in split order.
              float4 f[kMaxSplit][4];
#pragma unroll
              for (int q = 0; q < kMaxSplit; ++q) {
                if (q < S) {
#pragma unroll
                  for (int j = 0; j < 4; ++j) f[q][j] = __ldcg(base + q * split_stride + (c * 8 + h * 4 + j) * kBM + r);
                }
              }
#pragma unroll
              for (int j = 0; j < 4; ++j) {
                float4 acc4 = f[0][j];
#pragma unroll
                for (int q = 1; q < kMaxSplit; ++q) {
                  if (q < S) {
                    acc4.x += f[q][j].x;
                    acc4.y += f[q][j].y;
                    acc4.z += f[q][j].z;
                    acc4.w += f[q][j].w;
                  }
                }
                v[h * 16 + 4 * j] = __float_as_uint(acc4.x);
                v[h * 16 + 4 * j + 1] = __float_as_uint(acc4.y);
                v[h * 16 + 4 * j + 2] = __float_as_uint(acc4.z);
                v[h * 16 + 4 * j + 3] = __float_as_uint(acc4.w);
              }
            }
            store_chunk(stage, dst ? dst + c * 32 : nullptr, v, t.p == 0, a.gelu_tanh, lane);
          }
          if (leader) a.tile_sem[t.tile] = 0;
        }
      }
      if (++acc == 2) {
        acc = 0;
        acc_phase ^= 1u;
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
  }
}

}  // namespace

struct TcPlan {
  TcMaps p1, p2;         // phase 1 (N = F, K = D) and phase 2 (N = D, K = F)
  TcMaps p1g;            // phase 1 with A gathered from the layer input (box 64 x 1)
  const void* g_src = nullptr;  // layer input the gather map was encoded for
  int g_rows = 0;
  int bn1[3], bn2[3];
  TcShape shp[2][3];
  int* d_tab = nullptr;  // device plan table [3][tab_n]
  int tab_n = 0;
  int n_sms;
  int force_split;
};

size_t tc_split_units(int n_sms) { return static_cast<size_t>(4) * n_sms; }
size_t tc_partial_bytes(int n_sms) { return tc_split_units(n_sms) * kBM * kMaxBN * sizeof(float); }
// m-tiles a launch can have: every group's rows rounded up to 128.
static int max_mtiles_of(int max_rows, int G) { return (max_rows + kBM - 1) / kBM + G; }
size_t tc_dep_pairs(int max_rows, int G) { return static_cast<size_t>(max_mtiles_of(max_rows, G)) * kMaxSplit; }

namespace {

// Candidate widths for N: the widest of {256, 192} dividing N, then 128, 64.
void candidates(int n, int* bn) {
  bn[0] = n % 256 == 0 ? 256 : (n % 192 == 0 ? 192 : 0);
  bn[1] = n % 128 == 0 ? 128 : 0;
  bn[2] = n % 64 == 0 ? 64 : 0;
  if (!bn[0]) {  // keep slot 0 filled with the widest available width
    bn[0] = bn[1] ? bn[1] : bn[2];
    if (bn[0] == bn[1]) bn[1] = 0;
    else bn[2] = 0;
  }
}

// Stage geometry: two K sub-blocks per stage when the tile is at most 128
// wide (and K allows), so every stage moves 48-64 KB.
TcShape make_shape(int N, int K, int BN) {
  TcShape t{};
  if (!BN) return t;
  t.BN = BN;
  t.nt = N / BN;
  t.sub = (BN <= 128 && K % (2 * kBK) == 0) ? 2 : 1;
  t.KB = K / (kBK * t.sub);
  t.stage_bytes = t.sub * (kABytes + BN * kBK * 2);
  t.nst = std::min(kMaxStages, kRingBytes / t.stage_bytes);
  t.nt_magic = (1ull << 32) / static_cast<uint64_t>(t.nt) + 1;
  return t;
}

// Tile-width choice.  A unit moves (128 + BN) x K bf16 through its SM's
// ring, whose fill rate bounds it, and units run in waves of one per CTA:
// the width with the fewest waves x bytes per unit, the wider on a tie.
// Measured on the 12-layer D768 stack at ~60% reuse (16 m-tiles, one fused
// launch): phase-2 width 128 took 51 us, 64 took 59 us, and 256 (48 tiles)
// 56 us with two K splits; on the 28-layer D1152 stack (32 m-tiles) phase-2
// width 128 (288 tiles, 2 waves of 2.4 MB) beat 192 (192 tiles, 2 waves of
// 2.9 MB).  K splits are used only when forced: their parked partials and
// reductions cost 4-9 us of epilogue per unit.
int pick_width(const TcShape* shp, int mt, int grid, int force_bn) {
  int best = -1;
  double best_cost = 0.0;
  for (int i = 0; i < 3; ++i) {
    if (!shp[i].BN || (force_bn && shp[i].BN != force_bn)) continue;
    const long long units = static_cast<long long>(mt) * shp[i].nt;
    const long long waves = (units + grid - 1) / grid;
    const double K = static_cast<double>(shp[i].KB) * shp[i].sub * kBK;
    const double cost = static_cast<double>(waves) * (kBM + shp[i].BN) * K;
    if (best < 0 || cost < best_cost) {
      best = i;
      best_cost = cost;
    }
  }
  return best < 0 ? 0 : best;  // forced width absent: the widest
}

// Plan for `mt` m-tiles: fused (section 0) or one phase alone (section 1 + p).
// A fused launch splits phase 2 along K only when the split boundaries fall
// on phase-1 tile and stage boundaries.
int best_plan(const TcPlan* p, int section, int mt, int force_bn, int force_split) {
  const int grid = p->n_sms;
  const int max_units = static_cast<int>(tc_split_units(grid));
  if (section == 0) {
    const int i0 = pick_width(p->shp[0], mt, grid, force_bn), i1 = pick_width(p->shp[1], mt, grid, force_bn);
    const TcShape &a0 = p->shp[0][i0], &a1 = p->shp[1][i1];
    int S = force_split > 1 ? force_split : 1;
    if (S > 1 && (a0.nt % S || a1.KB % S || mt * a1.nt * S > max_units)) S = 1;
    return plan_word(i0, i1, S);
  }
  const int ph = section - 1;
  const int bi = pick_width(p->shp[ph], mt, grid, force_bn);
  const TcShape& t = p->shp[ph][bi];
  int S = force_split > 1 ? force_split : 1;
  if (S > 1 && (S > t.KB || mt * t.nt * S > max_units)) S = 1;
  return ph == 0 ? plan_word(bi, 0, S) : plan_word(0, bi, S);
}

bool encode_phase(TcMaps* m, const int* bn, const void* a_base, uint64_t rows, uint64_t K, const void* w,
                  uint64_t w_rows, const void* ws, uint64_t ws_rows) {
  if (!encode_2d(&m->a, a_base, rows, K, kBM)) return false;
  for (int i = 0; i < 3; ++i) {
    if (!bn[i]) {
      m->b[i] = m->b[0];
      m->bs[i] = m->bs[0];
      continue;
    }
    if (!encode_2d(&m->b[i], w, w_rows, K, bn[i])) return false;
    if (ws) {
      if (!encode_2d(&m->bs[i], ws, ws_rows, K, bn[i])) return false;
    } else {
      m->bs[i] = m->b[i];  // never read: there is no shared group
    }
  }
  return true;
}

}  // namespace

TcPlan* tc_plan_create(const FfnArgs& a, int n_sms, char* err, int errlen) {
  TcPlan* p = new TcPlan();
  p->n_sms = n_sms;
  p->force_split = a.split_k;
  candidates(a.F, p->bn1);
  candidates(a.D, p->bn2);
  const char* what = nullptr;
  if (!p->bn1[0] || !p->bn2[0] || a.D % kBK || a.F % kBK) what = "hidden and ffn must be multiples of 64";
  else if (!get_encoder()) what = "cuTensorMapEncodeTiled is unavailable";
  else if (!encode_phase(&p->p1, p->bn1, a.xg, a.max_rows, a.D, a.w1, static_cast<uint64_t>(a.E) * a.F, a.ws1, a.F) ||
           !encode_phase(&p->p2, p->bn2, a.hmid, a.max_rows, a.F, a.w2, static_cast<uint64_t>(a.E) * a.D, a.ws2, a.D))
    what = "tensor map encoding failed";
  if (!what) {
    for (int i = 0; i < 3; ++i) {
      p->shp[0][i] = make_shape(a.F, a.D, p->bn1[i]);
      p->shp[1][i] = make_shape(a.D, a.F, p->bn2[i]);
    }
    // One plan per possible m-tile count, for the fused launch and for each
    // phase alone.
    p->tab_n = std::min(max_mtiles_of(a.max_rows, a.G) + 1, kPlanTab);
    std::vector<int> tab(3 * static_cast<size_t>(p->tab_n));
    for (int sec = 0; sec < 3; ++sec)
      for (int mt = 0; mt < p->tab_n; ++mt)
        tab[sec * p->tab_n + mt] = best_plan(p, sec, mt, a.tile_n, a.split_k);
    if (cudaMalloc(&p->d_tab, tab.size() * sizeof(int)) != cudaSuccess ||
        cudaMemcpy(p->d_tab, tab.data(), tab.size() * sizeof(int), cudaMemcpyHostToDevice) != cudaSuccess) {
      cudaGetLastError();
      what = "cannot allocate the GEMM plan table";
    }
  }
  if (!what && cudaFuncSetAttribute(ffn_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes) !=
                   cudaSuccess) {
    cudaGetLastError();
    what = "cannot reserve shared memory for the tensor-core kernel";
  }
  if (what) {
    if (err && errlen > 0) snprintf(err, errlen, "%s", what);
    tc_plan_destroy(p);
    return nullptr;
  }
  return p;
}

void tc_plan_destroy(TcPlan* p) {
  if (!p) return;
  if (p->d_tab) cudaFree(p->d_tab);
  delete p;
}

cudaError_t launch_ffn_tc(TcPlan* p, const FfnArgs& a, int phase, cudaStream_t s) {
  TcArgs t{};
  t.G = a.G;
  t.E = a.E;
  t.k = a.k;
  t.T = a.T;
  t.gelu_tanh = a.gelu_tanh;
  // phase 0: both phases in one launch (two, without a dependency workspace).
  const bool fuse = phase == 0 && a.dep;
  if (phase == 0 && !fuse) {
    cudaError_t e = launch_ffn_tc(p, a, 1, s);
    return e != cudaSuccess ? e : launch_ffn_tc(p, a, 2, s);
  }
  t.first = fuse ? 1 : phase;
  t.last = fuse ? 2 : phase;
  t.N[0] = a.F;
  t.N[1] = a.D;
  for (int q = 0; q < 2; ++q)
    for (int i = 0; i < 3; ++i) t.shp[q][i] = p->shp[q][i];
  t.plan_tab = p->d_tab;
  t.tab_n = p->tab_n;
  t.counts = a.counts;
  t.offsets = a.offsets;
  t.list = a.list;
  t.hmid = a.hmid;
  t.cache_h = a.cache_h;
  t.shared_h = a.shared_h;
  t.partial = a.partial;
  t.tile_sem = a.tile_sem;
  t.dep = a.dep;
  t.dep_pairs = a.max_mtiles;
  t.work = a.work;
  t.status = a.status;
  TcMapPair maps;
  maps.p[0] = p->p1;
  maps.p[1] = p->p2;
  if (a.x && t.first == 1) {
    // Phase 1 reads its rows straight from the layer input; re-encode the
    // gather map when that buffer or its row count changes.
    if (a.x != p->g_src || a.T != p->g_rows) {
      p->p1g = p->p1;
      if (!encode_2d(&p->p1g.a, a.x, a.T, a.D, 1)) return cudaErrorInvalidValue;
      p->g_src = a.x;
      p->g_rows = a.T;
    }
    maps.p[0] = p->p1g;
    t.gather = 1;
  }
  return launch_pdl(ffn_tc_kernel, dim3(p->n_sms), dim3(kThreads), kSmemBytes, s, maps, t);
}

}  // namespace moeca
