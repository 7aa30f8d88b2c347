// Per-token branch decision of the branch-cached MoE layer (Sec. 4.2, Eq. 9),
// shared by select_kernel and the fused prep kernel.
//
//  * match each routed branch p against the token's cached branches by expert
//    id; an unmatched branch is always recomputed;
//  * score a matched branch  s = w_p + lambda1 |w_p - w_q^{t0}|
//    + lambda2 ||h_q|| / sum_j ||h_j||  and recompute iff s > tau_e;
//  * matched branches keep their slot q(p); unmatched ones take the slots whose
//    expert is no longer routed, ascending p -> ascending q; a full step
//    recomputes every branch with slot = p;
//  * write recompute / slot / matched, the new cache metadata and token_any.
#pragma once

#include "common.cuh"
#include "kernels.h"

namespace moeca {

template <int KMAX>
struct TokenDecisionT {
  int e[KMAX];
  int sl[KMAX];  // cache slot of each branch (valid tokens)
  bool rec[KMAX];
  bool any, bad, shared_row;
  int n_matched, n_rec, n_near;
};
using TokenDecision = TokenDecisionT<kMaxTopK>;

// The part of a token's decision that does not depend on the thresholds:
// routing, matching, slots and the scores of the matched branches.
template <int KMAX>
struct TokenPrepT {
  int e[KMAX];
  float w[KMAX];
  int sl[KMAX];
  bool mat[KMAX];
  float s[KMAX];  // score of a matched branch (Eq. 9)
  bool valid, bad;
  int n_matched;
};

// The token's inputs come through re/rw (routing, k entries) and ce/cw/cn
// (cached ids, weights, norms, k entries each), which may point to global or
// shared memory.  KMAX >= k bounds every loop at compile time.
template <int KMAX>
__device__ __forceinline__ void prepare_token(const SelectArgs& a, int i, bool valid, const int32_t* re,
                                              const float* rw, const int32_t* ce_in, const float* cw_in,
                                              const float* cn_in, TokenPrepT<KMAX>& t) {
  const int k = a.k, E = a.E;
  bool bad = false;
  int n_matched = 0;
#pragma unroll
  for (int p = 0; p < KMAX; ++p) {
    t.e[p] = -1;
    t.w[p] = 0.f;
    t.sl[p] = p;
    t.mat[p] = false;
    t.s[p] = 0.f;
  }
  if (valid) {
#pragma unroll
    for (int p = 0; p < KMAX; ++p) {
      if (p < k) {
        t.e[p] = re[p];
        t.w[p] = rw[p];
        if (t.e[p] < 0 || t.e[p] >= E) bad = true;
      }
    }
    if (bad) {
      report_status(a.status, kStatusBadIndex, 1000000 + i);
#pragma unroll
      for (int p = 0; p < KMAX; ++p) t.e[p] = -1;
    } else if (!a.refresh) {
      int ce[KMAX];
      float cw[KMAX], cn[KMAX];
      float nsum = 0.f;
      bool corrupt = false;
#pragma unroll
      for (int q = 0; q < KMAX; ++q) {
        ce[q] = -1;
        cw[q] = cn[q] = 0.f;
        if (q < k) {
          ce[q] = ce_in[q];
          cw[q] = cw_in[q];
          cn[q] = cn_in[q];
          nsum += cn[q];
          corrupt |= ce[q] < -1 || ce[q] >= E;  // -1: no cached branch
        }
      }
      // A cached expert id out of range (state written by the host) never
      // matches, so its branches are recomputed; the status word reports it.
      if (corrupt) report_status(a.status, kStatusBadIndex, 1100000 + i);
      unsigned used = 0u;
      int qof[KMAX];
#pragma unroll
      for (int p = 0; p < KMAX; ++p) {
        qof[p] = -1;
        if (p < k) {
#pragma unroll
          for (int q = KMAX - 1; q >= 0; --q)
            if (q < k && ce[q] == t.e[p]) qof[p] = q;  // lowest matching slot
          if (qof[p] >= 0) {
            const int q = qof[p];
            used |= 1u << q;
            t.mat[p] = true;
            ++n_matched;
            float cwq = 0.f, cnq = 0.f;
#pragma unroll
            for (int qq = 0; qq < KMAX; ++qq)
              if (qq == q) { cwq = cw[qq]; cnq = cn[qq]; }
            const float delta = fabsf(t.w[p] - cwq);
            const float o = nsum > 0.f ? cnq / nsum : 0.f;
            t.s[p] = ((a.score_terms & 1) ? t.w[p] : 0.f) + ((a.score_terms & 2) ? a.lambda1 * delta : 0.f) +
                     ((a.score_terms & 4) ? a.lambda2 * o : 0.f);
          }
        }
      }
      // Matched branches keep their slot; unmatched ones take the free slots
      // in ascending p -> ascending q order.
#pragma unroll
      for (int p = 0; p < KMAX; ++p) {
        if (p < k) {
          if (qof[p] >= 0) {
            t.sl[p] = qof[p];
          } else {
            int fq = 0;
            while ((used >> fq) & 1u) ++fq;
            used |= 1u << fq;
            t.sl[p] = fq;
          }
        }
      }
    }
  }
  t.valid = valid;
  t.bad = bad;
  t.n_matched = n_matched;
}

// The rest of the decision with the thresholds `tau` (global or shared
// memory): recompute iff unmatched or s > tau_e (every branch on a full
// step), token-level granularity, and the outputs: recompute / slot /
// matched, the new cache metadata and token_any at row i.
template <int KMAX>
__device__ __forceinline__ void finish_token(const SelectArgs& a, int i, const TokenPrepT<KMAX>& t,
                                             const float* tau, TokenDecisionT<KMAX>& d) {
  const int k = a.k;
  bool any = false;
  int n_rec = 0, n_near = 0;
#pragma unroll
  for (int p = 0; p < KMAX; ++p) {
    d.e[p] = t.e[p];
    d.sl[p] = t.sl[p];
    d.rec[p] = false;
  }
  if (t.valid && !t.bad) {
    const size_t base = static_cast<size_t>(i) * k;
    if (a.refresh) {
#pragma unroll
      for (int p = 0; p < KMAX; ++p) d.rec[p] = p < k;
    } else {
#pragma unroll
      for (int p = 0; p < KMAX; ++p) {
        if (p < k) {
          if (t.mat[p]) {
            const float tv = tau[t.e[p]];
            d.rec[p] = t.s[p] > tv;
            if (isfinite(tv) && fabsf(t.s[p] - tv) < 1e-5f * fabsf(tv)) ++n_near;
          } else {
            d.rec[p] = true;
          }
        }
      }
      if (a.token_level) {
        // Token-level granularity: one decision for all of the token's branches.
        bool anyr = false;
#pragma unroll
        for (int p = 0; p < KMAX; ++p) anyr |= (p < k) && d.rec[p];
#pragma unroll
        for (int p = 0; p < KMAX; ++p) d.rec[p] = (p < k) && anyr;
      }
    }
#pragma unroll
    for (int p = 0; p < KMAX; ++p) {
      if (p < k) {
        any |= d.rec[p];
        n_rec += d.rec[p];
        a.recompute[base + p] = d.rec[p];
        a.slot[base + p] = static_cast<int8_t>(t.sl[p]);
        a.matched[base + p] = t.mat[p];
        if (d.rec[p]) {
          a.cache_e[base + t.sl[p]] = t.e[p];
          a.cache_w[base + t.sl[p]] = t.w[p];
        } else if (a.reused_meta_policy) {
          a.cache_w[base + t.sl[p]] = t.w[p];
        }
      }
    }
    a.token_any[i] = any;
  }
  d.any = any;
  d.bad = t.bad;
  d.shared_row = t.valid && !t.bad && a.n_shared && (a.refresh || a.shared_policy || any);
  d.n_matched = t.n_matched;
  d.n_rec = n_rec;
  d.n_near = n_near;
}

template <int KMAX>
__device__ __forceinline__ void decide_token(const SelectArgs& a, int i, bool valid, const int32_t* re,
                                             const float* rw, const int32_t* ce_in, const float* cw_in,
                                             const float* cn_in, TokenDecisionT<KMAX>& d) {
  TokenPrepT<KMAX> t;
  prepare_token(a, i, valid, re, rw, ce_in, cw_in, cn_in, t);
  finish_token(a, i, t, a.tau, d);
}

}  // namespace moeca
