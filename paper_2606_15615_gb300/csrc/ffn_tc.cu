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
//           128-byte swizzle, into a kStages-deep shared-memory ring;
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
constexpr int kStages = 4;
constexpr int kThreads = 192;
constexpr int kTmemCols = 512;
constexpr int kABytes = kBM * kBK * 2;        // 16 KB
constexpr int kBBytesMax = kMaxBN * kBK * 2;  // 32 KB
constexpr int kStageBytes = kABytes + kBBytesMax;
constexpr int kSmemBytes = kStages * kStageBytes + 1024;
constexpr int kMaxGroups = kMaxExperts + 1;
constexpr unsigned long long kWaitNs = 1000000000ull;

struct TcArgs {
  int G, E, N, K, BN, k, T, phase, gelu_tanh;
  const int32_t* counts;
  const int32_t* offsets;
  const int32_t* list;
  void* hmid;      // phase 1 output [rows, F]
  void* cache_h;   // phase 2 routed destination [T*k, D]
  void* shared_h;  // phase 2 shared destination [T, D]
  int* status;
};

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ unsigned long long globaltimer() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ bool mbar_try(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
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
    ffn_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                  const __grid_constant__ CUtensorMap tmBs, TcArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) uint64_t full_bar[kStages];
  __shared__ __align__(8) uint64_t empty_bar[kStages];
  __shared__ __align__(8) uint64_t tfull_bar[2];
  __shared__ __align__(8) uint64_t tempty_bar[2];
  __shared__ __align__(8) uint64_t drain_bar;
  __shared__ uint32_t tmem_base_sh;
  __shared__ int tiles_before[kMaxGroups + 1];
  __shared__ int cnt_sh[kMaxGroups];
  __shared__ int off_sh[kMaxGroups];
  __shared__ volatile int abort_flag;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = a.G, BN = a.BN;
  const int n_tiles = a.N / BN;
  const int KB = a.K / kBK;

  if (threadIdx.x == 0) {
    int acc = 0;
    for (int g = 0; g < G; ++g) {
      const int c = a.counts[g];
      cnt_sh[g] = c;
      off_sh[g] = a.offsets[g];
      tiles_before[g] = acc;
      acc += ((c + kBM - 1) / kBM) * n_tiles;
    }
    tiles_before[G] = acc;
    abort_flag = 0;
    for (int s = 0; s < kStages; ++s) {
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
  const int total = tiles_before[G];

  if (warp == 0 && lane == 0) {
    // ---------------- TMA producer ----------------
    int stage = 0;
    uint32_t phase = 0;
    int issued = 0;
    const uint32_t bbytes = static_cast<uint32_t>(BN) * kBK * 2;
    bool ok = true;
    for (int tile = blockIdx.x; tile < total && ok; tile += gridDim.x) {
      const TileCoord tc = decode_tile(tile, tiles_before, cnt_sh, G, n_tiles);
      const CUtensorMap* tb = tc.g < a.E ? &tmB : &tmBs;
      const int brow = (tc.g < a.E ? tc.g * a.N : 0) + tc.n_tile * BN;
      const int arow = off_sh[tc.g] + tc.m_tile * kBM;
      for (int kb = 0; kb < KB; ++kb) {
        if (!mbar_wait(smem_u32(&empty_bar[stage]), phase ^ 1u, &abort_flag)) {
          ok = false;
          break;
        }
        const uint32_t fb = smem_u32(&full_bar[stage]);
        mbar_expect_tx(fb, kABytes + bbytes);
        uint8_t* sa = smem + stage * kStageBytes;
        tma_load_2d(smem_u32(sa), &tmA, kb * kBK, arow, fb);
        tma_load_2d(smem_u32(sa + kABytes), tb, kb * kBK, brow, fb);
        ++issued;
        if (++stage == kStages) {
          stage = 0;
          phase ^= 1u;
        }
      }
    }
    if (!ok) {
      if (!abort_flag) report_status(a.status, kStatusWaitTimeout, 100 + a.phase);
      abort_flag = 1;
      // Let the copies already issued land before the CTA can exit.
      const int pending = issued < kStages ? issued : kStages;
      int s = stage;
      uint32_t ph = phase;
      for (int j = 0; j < pending; ++j) {
        if (--s < 0) {
          s = kStages - 1;
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
    for (int tile = blockIdx.x; tile < total && ok; tile += gridDim.x) {
      if (!mbar_wait(smem_u32(&tempty_bar[acc]), acc_phase ^ 1u, &abort_flag)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t d_tmem = tmem + static_cast<uint32_t>(acc * BN);
      for (int kb = 0; kb < KB; ++kb) {
        if (!mbar_wait(smem_u32(&full_bar[stage]), phase, &abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t sa = smem_u32(smem + stage * kStageBytes);
        const uint32_t sb = sa + kABytes;
#pragma unroll
        for (int kk = 0; kk < kBK / 16; ++kk) {
          mma_bf16(d_tmem, smem_desc(sa + kk * 32), smem_desc(sb + kk * 32), idesc, (kb | kk) != 0);
        }
        mma_commit(smem_u32(&empty_bar[stage]));
        if (++stage == kStages) {
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
    const int quad = warp & 3;  // TMEM lanes [32 quad, 32 quad + 32)
    const int r = quad * 32 + lane;
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int tile = blockIdx.x; tile < total; tile += gridDim.x) {
      const TileCoord tc = decode_tile(tile, tiles_before, cnt_sh, G, n_tiles);
      // Warp-uniform outcome: tcgen05.ld below needs the whole warp converged.
      const bool got = __all_sync(0xffffffffu, mbar_wait(smem_u32(&tfull_bar[acc]), acc_phase, &abort_flag));
      if (!got) {
        if (lane == 0 && !abort_flag) report_status(a.status, kStatusWaitTimeout, 300 + a.phase);
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
      for (int c = 0; c < BN / 32; ++c) {
        uint32_t v[32];
        tmem_ld32(tbase + c * 32, v);
        if (dst) {
          uint32_t packed[16];
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            float x0 = __uint_as_float(v[2 * j]), x1 = __uint_as_float(v[2 * j + 1]);
            if (a.phase == 1) {
              x0 = gelu_f(x0, a.gelu_tanh);
              x1 = gelu_f(x1, a.gelu_tanh);
            }
            __nv_bfloat162 h2 = __floats2bfloat162_rn(x0, x1);
            packed[j] = *reinterpret_cast<uint32_t*>(&h2);
          }
          uint4* d4 = reinterpret_cast<uint4*>(dst + c * 32);
#pragma unroll
          for (int j = 0; j < 4; ++j)
            d4[j] = make_uint4(packed[4 * j], packed[4 * j + 1], packed[4 * j + 2], packed[4 * j + 3]);
        }
      }
      tc_fence_before();
      mbar_arrive(smem_u32(&tempty_bar[acc]));
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

int pick_bn(int n) {
  const int cands[] = {256, 192, 128, 64};
  for (int c : cands)
    if (n % c == 0) return c;
  return 0;
}

}  // namespace

struct TcPlan {
  CUtensorMap a1, b1, bs1, a2, b2, bs2;
  int bn1, bn2;
  int n_sms;
};

TcPlan* tc_plan_create(const FfnArgs& a, int n_sms, char* err, int errlen) {
  TcPlan* p = new TcPlan();
  p->n_sms = n_sms;
  p->bn1 = pick_bn(a.F);
  p->bn2 = pick_bn(a.D);
  const char* what = nullptr;
  if (!p->bn1 || !p->bn2 || a.D % kBK || a.F % kBK) what = "hidden and ffn must be multiples of 64";
  else if (!get_encoder()) what = "cuTensorMapEncodeTiled is unavailable";
  else if (!encode_2d(&p->a1, a.xg, a.max_rows, a.D, kBM) || !encode_2d(&p->a2, a.hmid, a.max_rows, a.F, kBM) ||
           !encode_2d(&p->b1, a.w1, static_cast<uint64_t>(a.E) * a.F, a.D, p->bn1) ||
           !encode_2d(&p->b2, a.w2, static_cast<uint64_t>(a.E) * a.D, a.F, p->bn2))
    what = "tensor map encoding failed";
  else if (a.ws1 && (!encode_2d(&p->bs1, a.ws1, a.F, a.D, p->bn1) || !encode_2d(&p->bs2, a.ws2, a.D, a.F, p->bn2)))
    what = "shared-expert tensor map encoding failed";
  if (!a.ws1) {
    p->bs1 = p->b1;  // never read: there is no shared group
    p->bs2 = p->b2;
  }
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
  t.BN = phase == 1 ? p->bn1 : p->bn2;
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
  t.status = a.status;
  const long long max_tiles =
      (static_cast<long long>(a.max_rows + kBM - 1) / kBM + a.G) * static_cast<long long>(t.N / t.BN);
  const int grid = static_cast<int>(max_tiles < p->n_sms ? max_tiles : p->n_sms);
  if (phase == 1) ffn_tc_kernel<<<grid, kThreads, kSmemBytes, s>>>(p->a1, p->b1, p->bs1, t);
  else ffn_tc_kernel<<<grid, kThreads, kSmemBytes, s>>>(p->a2, p->b2, p->bs2, t);
  return cudaGetLastError();
}

}  // namespace moeca
