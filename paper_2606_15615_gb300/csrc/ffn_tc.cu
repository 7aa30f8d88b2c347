// Tensor-core grouped expert FFN (bf16 operands, fp32 accumulation) for sm_103a.
//
// Computes the recompute branches of Eq. 5 / Eq. 6 over the compacted rows:
//   phase 1: hmid[r, :] = GELU(xg[r, :] W1_g^T)         N = F, K = D
//   phase 2: dst[list[r], :] = hmid[r, :] W2_g^T         N = D, K = F
// where rows r of expert group g are [offsets[g], offsets[g] + counts[g]) and
// dst is the branch cache (token*k + slot) or the shared-expert rows.
//
// Persistent kernel, one CTA per SM, 6 warps:
//   warp 0  TMA producer: 128 x 64 A tile and BN x 64 weight tile per stage,
//           128-byte swizzle, into a 192 KB shared-memory ring (4-8 stages);
//   warp 1  allocates 512 TMEM columns and issues tcgen05.mma (M = 128,
//           N = BN, K = 16) from one thread; tcgen05.commit frees each stage
//           and signals a finished accumulator;
//   warps 2-5  epilogue: tcgen05.ld of their TMEM lane quadrant, GELU / bf16
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
#include <cstdio>

#include "common.cuh"
#include "kernels.h"

namespace moeca {

namespace {

constexpr int kBM = 128;          // rows per tile (MMA M)
constexpr int kBK = 64;           // K per stage: 64 bf16 = one 128-byte swizzle row
constexpr int kMaxBN = 256;
constexpr int kMaxStages = 8;
constexpr int kRingBytes = 4 * (16384 + 256 * 128);  // 192 KB of stages, any tile width
constexpr int kThreads = 192;
constexpr int kTmemCols = 512;
constexpr int kABytes = kBM * kBK * 2;        // 16 KB
constexpr int kBBytesMax = kMaxBN * kBK * 2;  // 32 KB
constexpr int kSmemBytes = kRingBytes + 1024;
constexpr int kMaxGroups = kMaxExperts + 1;
constexpr unsigned long long kWaitNs = 1000000000ull;
constexpr int kMaxSplit = 4;

struct TcArgs {
  int G, E, N, K, BN, k, T, phase, gelu_tanh;
  const int32_t* counts;
  const int32_t* offsets;
  const int32_t* list;
  void* hmid;      // phase 1 output [rows, F]
  void* cache_h;   // phase 2 routed destination [T*k, D]
  void* shared_h;  // phase 2 shared destination [T, D]
  float* partial;  // split-K partial tiles, [max_units][128][BN] fp32
  int* tile_sem;   // split-K arrival counters, [max_units], left at 0
  int max_units;   // capacity of partial / tile_sem
  int gather;      // phase 1: A rows gathered from the layer input by token (tile::gather4)
  int bn[3];       // candidate tile widths (0 = none), matching the maps' B boxes
  int force_bn;    // 0: choose; else use this width
  int force_split; // 0: choose; else use this many K splits
  float split_cost;  // cost of one split unit's partial round trip, in BN-256 k-blocks
  int* status;
};

// Weight and activation tensor maps of one phase: A (activation rows) and,
// for each candidate width, B (routed experts) and Bs (shared expert).
struct alignas(64) TcMaps {
  CUtensorMap a;
  CUtensorMap b[3];
  CUtensorMap bs[3];
};

// Tile width and K split for this launch.  Every CTA evaluates the same cost
// model on the same device-resident counts.  A unit is one (tile, K range).
// Cost = waves of units over the grid x per-unit time, where per-unit time is
// k-blocks x stage time (a stage streams 128 + BN rows of 128 bytes; its MMAs
// take about 0.7 of a 256-wide stage's load time), plus one for pipeline fill
// and epilogue, plus, for split units, the fp32 partial round trip.
struct Plan {
  int bi, S;
};

__device__ Plan choose_plan(const TcArgs& a, int m_tiles, int KB, int grid) {
  Plan best{-1, 1};
  float best_cost = 3.0e38f;
  for (int bi = 0; bi < 3; ++bi) {
    const int BN = a.bn[bi];
    if (BN == 0 || (a.force_bn && BN != a.force_bn)) continue;
    const int tiles = m_tiles * (a.N / BN);
    const float stage = fmaxf((128.f + BN) / 384.f, 0.7f * BN / 256.f);
    for (int S = 1; S <= 4 && S <= KB; ++S) {
      if (a.force_split && S != a.force_split) continue;
      if (S > 1 && tiles * S > a.max_units) break;
      const int units = tiles * S;
      const int waves = (units + grid - 1) / grid;
      const float per = ((KB + S - 1) / S) * stage + 1.0f + (S > 1 ? a.split_cost * BN / 256.f : 0.f);
      const float cost = waves * per;
      if (cost < best_cost - 1e-3f) {
        best_cost = cost;
        best = Plan{bi, S};
      }
    }
  }
  if (best.bi < 0) best = Plan{0, 1};  // forced values matched nothing: widest tile, no split
  return best;
}

// Bounded wait for phase `parity` of a barrier.  False on timeout or abort.
__device__ __noinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag) {
  unsigned long long t0 = 0;
  for (uint32_t it = 1;; ++it) {
    if (mbar_try(bar, parity)) return true;
    if ((it & 255u) == 0) {
      if (*abort_flag) return false;
      const unsigned long long now = globaltimer();
      if (t0 == 0) t0 = now;
      else if (now - t0 > kWaitNs) return false;
    }
  }
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int x, int y, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];"
      ::"r"(dst), "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}

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

// Shared-memory matrix descriptor: K-major operand, 128-byte swizzle,
// 8-row groups 1024 bytes apart (stride byte offset), descriptor version 1.
__device__ __forceinline__ uint64_t smem_desc(uint32_t addr) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((addr & 0x3FFFFu) >> 4);          // start address
  d |= static_cast<uint64_t>(1) << 16;                          // leading byte offset (unused)
  d |= static_cast<uint64_t>(1024 >> 4) << 32;                  // stride byte offset
  d |= static_cast<uint64_t>(1) << 46;                          // version
  d |= static_cast<uint64_t>(2) << 61;                          // SWIZZLE_128B
  return d;
}

// Instruction descriptor of kind::f16: bf16 A and B, fp32 D, both K-major.
__host__ __device__ constexpr uint32_t instr_desc(int M, int N) {
  return (1u << 4)                                   // D format f32
         | (1u << 7)                                 // A format bf16
         | (1u << 10)                                // B format bf16
         | (static_cast<uint32_t>(N >> 3) << 17)     // N / 8
         | (static_cast<uint32_t>(M >> 4) << 24);    // M / 16
}

__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}"
      ::"r"(d_tmem), "l"(a), "l"(b), "r"(idesc), "r"(acc)
      : "memory");
}

__device__ __forceinline__ void mma_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t* v) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]),
        "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15]),
        "=r"(v[16]), "=r"(v[17]), "=r"(v[18]), "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]),
        "=r"(v[24]), "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// 32 fp32 values of one row -> (GELU) -> bf16 -> 64 contiguous bytes.
__device__ __forceinline__ void store_row32(__nv_bfloat16* dst, const uint32_t* v, bool gelu, int tanh_form) {
  uint32_t packed[16];
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    float x0 = __uint_as_float(v[2 * j]), x1 = __uint_as_float(v[2 * j + 1]);
    if (gelu) {
      x0 = gelu_f(x0, tanh_form);
      x1 = gelu_f(x1, tanh_form);
    }
    __nv_bfloat162 h2 = __floats2bfloat162_rn(x0, x1);
    packed[j] = *reinterpret_cast<uint32_t*>(&h2);
  }
  uint4* d4 = reinterpret_cast<uint4*>(dst);
#pragma unroll
  for (int j = 0; j < 4; ++j) d4[j] = make_uint4(packed[4 * j], packed[4 * j + 1], packed[4 * j + 2], packed[4 * j + 3]);
}

struct TileCoord {
  int g, m_tile, n_tile;
};

__device__ __forceinline__ TileCoord decode_tile(int tile, const int* tiles_before, const int* cnt, int G,
                                                 int n_tiles) {
  int g = 0;
  while (g + 1 < G && tile >= tiles_before[g + 1]) ++g;
  const int local = tile - tiles_before[g];
  const int mt = (cnt[g] + kBM - 1) / kBM;
  return TileCoord{g, local % mt, local / mt};
}

__global__ void __launch_bounds__(kThreads, 1)
    ffn_tc_kernel(const __grid_constant__ TcMaps maps, TcArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) uint64_t full_bar[kMaxStages];
  __shared__ __align__(8) uint64_t empty_bar[kMaxStages];
  __shared__ __align__(8) uint64_t tfull_bar[2];
  __shared__ __align__(8) uint64_t tempty_bar[2];
  __shared__ __align__(8) uint64_t drain_bar;
  __shared__ uint32_t tmem_base_sh;
  __shared__ int tiles_before[kMaxGroups + 1];
  __shared__ int cnt_sh[kMaxGroups];
  __shared__ int off_sh[kMaxGroups];
  __shared__ volatile int abort_flag;
  __shared__ int split_sh, bi_sh;
  __shared__ int rows_sh[kBM];  // producer: token of each row of the current tile (gather)
  __shared__ volatile int ep_abort;
  __shared__ volatile int ep_last;

  pdl_entry();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = a.G;
  const int KB = a.K / kBK;

  if (threadIdx.x == 0) {
    int m_tiles = 0;
    for (int g = 0; g < G; ++g) {
      const int c = a.counts[g];
      cnt_sh[g] = c;
      off_sh[g] = a.offsets[g];
      m_tiles += (c + kBM - 1) / kBM;
    }
    const Plan pl = choose_plan(a, m_tiles, KB, gridDim.x);
    bi_sh = pl.bi;
    split_sh = pl.S;
    const int nt = a.N / a.bn[pl.bi];
    int acc = 0;
    for (int g = 0; g < G; ++g) {
      tiles_before[g] = acc;
      acc += ((cnt_sh[g] + kBM - 1) / kBM) * nt;
    }
    tiles_before[G] = acc;
    abort_flag = 0;
    ep_abort = 0;
    for (int s = 0; s < kMaxStages; ++s) {
      mbar_init(smem_u32(&full_bar[s]), 1);
      mbar_init(smem_u32(&empty_bar[s]), 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(smem_u32(&tfull_bar[s]), 1);
      mbar_init(smem_u32(&tempty_bar[s]), 128);
    }
    mbar_init(smem_u32(&drain_bar), 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;"
                 ::"r"(smem_u32(&tmem_base_sh)), "r"(kTmemCols) : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    tc_fence_before();
  }
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base_sh;
  const int BN = a.bn[bi_sh];
  const int n_tiles = a.N / BN;
  // Ring depth for this width: as many stages as fit the 192 KB ring.
  const int stage_bytes = kABytes + BN * kBK * 2;
  const int nst = min(kMaxStages, kRingBytes / stage_bytes);
  const CUtensorMap* tmA = &maps.a;
  const CUtensorMap* tmB = &maps.b[bi_sh];
  const CUtensorMap* tmBs = &maps.bs[bi_sh];
  const int tiles = tiles_before[G];
  const int S = split_sh;
  const int total = tiles * S;  // units: unit u is tile u % tiles, K split u / tiles

  if (warp == 0) {
    // ---------------- TMA producer (lane 0 issues; the warp fetches row indices) ----------------
    int stage = 0;
    uint32_t phase = 0;
    int issued = 0;
    const uint32_t bbytes = static_cast<uint32_t>(BN) * kBK * 2;
    bool ok = true;
    for (int u = blockIdx.x; u < total; u += gridDim.x) {
      const int tile = u % tiles, sp = u / tiles;
      const TileCoord tc = decode_tile(tile, tiles_before, cnt_sh, G, n_tiles);
      const CUtensorMap* tb = tc.g < a.E ? tmB : tmBs;
      const int brow = (tc.g < a.E ? tc.g * a.N : 0) + tc.n_tile * BN;
      const int arow = off_sh[tc.g] + tc.m_tile * kBM;
      const int kb0 = sp * KB / S, kb1 = (sp + 1) * KB / S;
      if (a.gather) {
        // Token of each of the tile's 128 rows; rows past the group's end
        // repeat its first row (their results are never stored).
        const int valid = cnt_sh[tc.g] - tc.m_tile * kBM;
#pragma unroll
        for (int j = 0; j < kBM / 32; ++j) {
          const int r = lane * (kBM / 32) + j;
          const int ent = a.list[arow + (r < valid ? r : 0)];
          int tok = tc.g < a.E ? ent / a.k : ent;
          tok = tok < 0 ? 0 : (tok >= a.T ? a.T - 1 : tok);
          rows_sh[r] = tok;
        }
        __syncwarp();
      }
      if (lane == 0) {
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait(smem_u32(&empty_bar[stage]), phase ^ 1u, &abort_flag)) {
            ok = false;
            break;
          }
          const uint32_t fb = smem_u32(&full_bar[stage]);
          mbar_expect_tx(fb, kABytes + bbytes);
          uint8_t* sa = smem + stage * stage_bytes;
          if (a.gather) {
#pragma unroll 4
            for (int j = 0; j < kBM / 4; ++j)
              tma_gather4(smem_u32(sa + j * 512), tmA, kb * kBK, rows_sh[4 * j], rows_sh[4 * j + 1],
                          rows_sh[4 * j + 2], rows_sh[4 * j + 3], fb);
          } else {
            tma_load_2d(smem_u32(sa), tmA, kb * kBK, arow, fb);
          }
          tma_load_2d(smem_u32(sa + kABytes), tb, kb * kBK, brow, fb);
          ++issued;
          if (++stage == nst) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      ok = __shfl_sync(0xffffffffu, ok, 0);
      __syncwarp();
      if (!ok) break;
    }
    if (!ok && lane == 0) {
      if (!abort_flag) report_status(a.status, kStatusWaitTimeout, 100 + a.phase);
      abort_flag = 1;
      // Let the copies already issued land before the CTA can exit.
      const int pending = issued < nst ? issued : nst;
      int s = stage;
      uint32_t ph = phase;
      for (int j = 0; j < pending; ++j) {
        if (--s < 0) {
          s = nst - 1;
          ph ^= 1u;
        }
        unsigned long long t0 = globaltimer();
        while (!mbar_try(smem_u32(&full_bar[s]), ph) && globaltimer() - t0 < kWaitNs) {
        }
      }
    }
  } else if (warp == 1 && lane == 0) {
    // ---------------- MMA issuer ----------------
    int stage = 0;
    uint32_t phase = 0;
    int acc = 0;
    uint32_t acc_phase = 0;
    const uint32_t idesc = instr_desc(kBM, BN);
    bool ok = true;
    for (int u = blockIdx.x; u < total && ok; u += gridDim.x) {
      const int sp = u / tiles;
      const int kb0 = sp * KB / S, kb1 = (sp + 1) * KB / S;
      if (!mbar_wait(smem_u32(&tempty_bar[acc]), acc_phase ^ 1u, &abort_flag)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t d_tmem = tmem + static_cast<uint32_t>(acc * BN);
      for (int kb = kb0; kb < kb1; ++kb) {
        if (!mbar_wait(smem_u32(&full_bar[stage]), phase, &abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t sa = smem_u32(smem + stage * stage_bytes);
        const uint32_t sb = sa + kABytes;
#pragma unroll
        for (int kk = 0; kk < kBK / 16; ++kk) {
          mma_bf16(d_tmem, smem_desc(sa + kk * 32), smem_desc(sb + kk * 32), idesc, (kb != kb0) || kk != 0);
        }
        mma_commit(smem_u32(&empty_bar[stage]));
        if (++stage == nst) {
          stage = 0;
          phase ^= 1u;
        }
      }
      if (!ok) break;
      mma_commit(smem_u32(&tfull_bar[acc]));
      if (++acc == 2) {
        acc = 0;
        acc_phase ^= 1u;
      }
    }
    if (!ok) {
      if (!abort_flag) report_status(a.status, kStatusWaitTimeout, 200 + a.phase);
      abort_flag = 1;
    }
    // Every MMA this thread issued has completed once the drain barrier fires.
    mma_commit(smem_u32(&drain_bar));
    unsigned long long t0 = globaltimer();
    while (!mbar_try(smem_u32(&drain_bar), 0) && globaltimer() - t0 < kWaitNs) {
    }
  } else if (warp >= 2) {
    // ---------------- Epilogue ----------------
    // The 4 epilogue warps (128 threads) agree on every abort and every
    // split-K decision through named barrier 1, so none can wait alone.
    const int quad = warp & 3;  // TMEM lanes [32 quad, 32 quad + 32)
    const int r = quad * 32 + lane;
    const bool leader = warp == 2 && lane == 0;
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int u = blockIdx.x; u < total; u += gridDim.x) {
      const int tile = u % tiles, sp = u / tiles;
      const TileCoord tc = decode_tile(tile, tiles_before, cnt_sh, G, n_tiles);
      const bool got = __all_sync(0xffffffffu, mbar_wait(smem_u32(&tfull_bar[acc]), acc_phase, &abort_flag));
      if (!got && lane == 0) ep_abort = 1;
      asm volatile("bar.sync 1, 128;" ::: "memory");
      if (ep_abort) {
        if (leader && !abort_flag) report_status(a.status, kStatusWaitTimeout, 300 + a.phase);
        abort_flag = 1;
        break;
      }
      tc_fence_after();
      const int mrow = tc.m_tile * kBM + r;
      const bool live = mrow < cnt_sh[tc.g];
      const size_t grow = static_cast<size_t>(off_sh[tc.g]) + mrow;
      const int n0 = tc.n_tile * BN;
      __nv_bfloat16* dst = nullptr;
      if (live) {
        if (a.phase == 1) {
          dst = static_cast<__nv_bfloat16*>(a.hmid) + grow * a.N + n0;
        } else {
          const int dr = a.list[grow];
          const int lim = tc.g < a.E ? a.T * a.k : a.T;
          if (dr >= 0 && dr < lim) {
            dst = static_cast<__nv_bfloat16*>(tc.g < a.E ? a.cache_h : a.shared_h) + static_cast<size_t>(dr) * a.N + n0;
          } else {
            report_status(a.status, kStatusBadIndex, 4000000 + static_cast<int>(grow));
          }
        }
      }
      const uint32_t tbase = tmem + (static_cast<uint32_t>(quad * 32) << 16) + static_cast<uint32_t>(acc * BN);
      if (S == 1) {
        for (int c = 0; c < BN / 32; ++c) {
          uint32_t v[32];
          tmem_ld32(tbase + c * 32, v);
          if (dst) store_row32(dst + c * 32, v, a.phase == 1, a.gelu_tanh);
        }
        tc_fence_before();
        mbar_arrive(smem_u32(&tempty_bar[acc]));
      } else {
        // Split K: park this split's fp32 rows, free TMEM, then the last
        // split to arrive for the tile sums the splits in split order.
        float* mine = a.partial + (static_cast<size_t>(tile) * S + sp) * kBM * BN + static_cast<size_t>(r) * BN;
        for (int c = 0; c < BN / 32; ++c) {
          uint32_t v[32];
          tmem_ld32(tbase + c * 32, v);
          float4* d4 = reinterpret_cast<float4*>(mine + c * 32);
#pragma unroll
          for (int j = 0; j < 8; ++j)
            d4[j] = make_float4(__uint_as_float(v[4 * j]), __uint_as_float(v[4 * j + 1]),
                                __uint_as_float(v[4 * j + 2]), __uint_as_float(v[4 * j + 3]));
        }
        tc_fence_before();
        mbar_arrive(smem_u32(&tempty_bar[acc]));
        __threadfence();
        asm volatile("bar.sync 1, 128;" ::: "memory");
        if (leader) ep_last = atomicAdd(a.tile_sem + tile, 1) == S - 1;
        asm volatile("bar.sync 1, 128;" ::: "memory");
        if (ep_last) {
          __threadfence();
          const float* base = a.partial + static_cast<size_t>(tile) * S * kBM * BN + static_cast<size_t>(r) * BN;
          for (int c = 0; c < BN / 32; ++c) {
            uint32_t v[32];
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              // All splits' 16 values in flight at once, then added in split order.
              float4 f[kMaxSplit][4];
#pragma unroll
              for (int q = 0; q < kMaxSplit; ++q) {
                if (q < S) {
                  const float4* s4 = reinterpret_cast<const float4*>(
                      base + static_cast<size_t>(q) * kBM * BN + c * 32 + h * 16);
#pragma unroll
                  for (int j = 0; j < 4; ++j) f[q][j] = __ldcg(s4 + j);
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
            if (dst) store_row32(dst + c * 32, v, a.phase == 1, a.gelu_tanh);
          }
          if (leader) a.tile_sem[tile] = 0;
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

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn get_encoder() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

// 2-D bf16 map over [rows, cols] row-major, box {64, box_rows}, 128-byte swizzle.
bool encode_2d(CUtensorMap* m, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows) {
  EncodeTiledFn enc = get_encoder();
  if (!enc) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(kBK), box_rows};
  cuuint32_t estr[2] = {1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

struct TcPlan {
  TcMaps p1, p2;         // phase 1 (N = F, K = D) and phase 2 (N = D, K = F)
  TcMaps p1g;            // phase 1 with A gathered from the layer input (box 64 x 1)
  const void* g_src = nullptr;  // layer input the gather map was encoded for
  int g_rows = 0;
  int bn1[3], bn2[3];
  int n_sms;
  int force_bn, force_split;
  float split_cost;
};

size_t tc_split_units(int n_sms) { return static_cast<size_t>(4) * n_sms; }
size_t tc_partial_bytes(int n_sms) { return tc_split_units(n_sms) * kBM * kMaxBN * sizeof(float); }

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
  p->force_bn = a.tile_n;
  p->force_split = a.split_k;
  p->split_cost = 40.0f;  // measured: split units rarely pay for their partial round trip
  candidates(a.F, p->bn1);
  candidates(a.D, p->bn2);
  const char* what = nullptr;
  if (!p->bn1[0] || !p->bn2[0] || a.D % kBK || a.F % kBK) what = "hidden and ffn must be multiples of 64";
  else if (!get_encoder()) what = "cuTensorMapEncodeTiled is unavailable";
  else if (!encode_phase(&p->p1, p->bn1, a.xg, a.max_rows, a.D, a.w1, static_cast<uint64_t>(a.E) * a.F, a.ws1, a.F) ||
           !encode_phase(&p->p2, p->bn2, a.hmid, a.max_rows, a.F, a.w2, static_cast<uint64_t>(a.E) * a.D, a.ws2, a.D))
    what = "tensor map encoding failed";
  if (!what && cudaFuncSetAttribute(ffn_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes) !=
                   cudaSuccess) {
    cudaGetLastError();
    what = "cannot reserve shared memory for the tensor-core kernel";
  }
  if (what) {
    if (err && errlen > 0) snprintf(err, errlen, "%s", what);
    delete p;
    return nullptr;
  }
  return p;
}

void tc_plan_destroy(TcPlan* p) { delete p; }

cudaError_t launch_ffn_tc(TcPlan* p, const FfnArgs& a, int phase, cudaStream_t s) {
  TcArgs t{};
  t.G = a.G;
  t.E = a.E;
  t.N = phase == 1 ? a.F : a.D;
  t.K = phase == 1 ? a.D : a.F;
  t.k = a.k;
  t.T = a.T;
  t.phase = phase;
  t.gelu_tanh = a.gelu_tanh;
  t.counts = a.counts;
  t.offsets = a.offsets;
  t.list = a.list;
  t.hmid = a.hmid;
  t.cache_h = a.cache_h;
  t.shared_h = a.shared_h;
  t.partial = a.partial;
  t.tile_sem = a.tile_sem;
  t.max_units = a.partial ? static_cast<int>(tc_split_units(p->n_sms)) : 0;
  const int* bn = phase == 1 ? p->bn1 : p->bn2;
  for (int i = 0; i < 3; ++i) t.bn[i] = bn[i];
  t.force_bn = p->force_bn;
  t.force_split = p->force_split;
  t.split_cost = p->split_cost;
  t.status = a.status;
  const TcMaps* maps = phase == 1 ? &p->p1 : &p->p2;
  if (phase == 1 && a.x) {
    // Phase 1 reads its rows straight from the layer input; re-encode the
    // gather map when that buffer or its row count changes.
    if (a.x != p->g_src || a.T != p->g_rows) {
      p->p1g = p->p1;
      if (!encode_2d(&p->p1g.a, a.x, a.T, a.D, 1)) return cudaErrorInvalidValue;
      p->g_src = a.x;
      p->g_rows = a.T;
    }
    maps = &p->p1g;
    t.gather = 1;
  }
  return launch_pdl(ffn_tc_kernel, dim3(p->n_sms), dim3(kThreads), kSmemBytes, s, *maps, t);
}

}  // namespace moeca
