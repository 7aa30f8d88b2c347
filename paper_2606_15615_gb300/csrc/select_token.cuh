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

// The token's inputs come through re/rw (routing, k entries) and ce/cw/cn
// (cached ids, weights, norms, k entries each), which may point to global or
// shared memory; outputs go to a's global arrays at row i.
// KMAX >= k bounds every loop at compile time.
template <int KMAX>
__device__ __forceinline__ void decide_token(const SelectArgs& a, int i, bool valid, const int32_t* re,
                                             const float* rw, const int32_t* ce_in, const float* cw_in,
                                             const float* cn_in, TokenDecisionT<KMAX>& d) {
  const int k = a.k, E = a.E;
  int* e = d.e;
  bool* rec = d.rec;
  bool any = false;
  int n_matched = 0, n_rec = 0, n_near = 0;
  bool bad = false;
#pragma unroll
  for (int p = 0; p < KMAX; ++p) {
    e[p] = -1;
    rec[p] = false;
    d.sl[p] = p;
  }
  if (valid) {
    const size_t base = static_cast<size_t>(i) * k;
    float w[KMAX];
    int sl[KMAX];
    bool mat[KMAX];
#pragma unroll
    for (int p = 0; p < KMAX; ++p) {
      if (p < k) {
        e[p] = re[p];
        w[p] = rw[p];
        if (e[p] < 0 || e[p] >= E) bad = true;
      }
      mat[p] = false;
      sl[p] = p;
    }
    if (bad) {
      report_status(a.status, kStatusBadIndex, 1000000 + i);
#pragma unroll
      for (int p = 0; p < KMAX; ++p) e[p] = -1;
    } else if (a.refresh) {
#pragma unroll
      for (int p = 0; p < KMAX; ++p) rec[p] = p < k;
    } else {
      int ce[KMAX];
      float cw[KMAX], cn[KMAX];
      float nsum = 0.f;
#pragma unroll
      bool corrupt = false;
      for (int q = 0; q < KMAX; ++q) {
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
            if (q < k && ce[q] == e[p]) qof[p] = q;  // lowest matching slot
          if (qof[p] >= 0) {
            const int q = qof[p];
            used |= 1u << q;
            mat[p] = true;
            ++n_matched;
            float cwq = 0.f, cnq = 0.f;
#pragma unroll
            for (int qq = 0; qq < KMAX; ++qq)
              if (qq == q) { cwq = cw[qq]; cnq = cn[qq]; }
            const float delta = fabsf(w[p] - cwq);
            const float o = nsum > 0.f ? cnq / nsum : 0.f;
            const float s = ((a.score_terms & 1) ? w[p] : 0.f) + ((a.score_terms & 2) ? a.lambda1 * delta : 0.f) +
                            ((a.score_terms & 4) ? a.lambda2 * o : 0.f);
            const float tau = a.tau[e[p]];
            rec[p] = s > tau;
            if (isfinite(tau) && fabsf(s - tau) < 1e-5f * fabsf(tau)) ++n_near;
          } else {
            rec[p] = true;
          }
        }
      }
      if (a.token_level) {
        // Token-level granularity: one decision for all of the token's branches.
        bool anyr = false;
#pragma unroll
        for (int p = 0; p < KMAX; ++p) anyr |= (p < k) && rec[p];
#pragma unroll
        for (int p = 0; p < KMAX; ++p) rec[p] = (p < k) && anyr;
      }
#pragma unroll
      for (int p = 0; p < KMAX; ++p) {
        if (p < k) {
          if (qof[p] >= 0) {
            sl[p] = qof[p];
          } else {
            int fq = 0;
            while ((used >> fq) & 1u) ++fq;
            used |= 1u << fq;
            sl[p] = fq;
          }
        }
      }
    }
    if (!bad) {
#pragma unroll
      for (int p = 0; p < KMAX; ++p) {
        if (p < k) {
          any |= rec[p];
          n_rec += rec[p];
          a.recompute[base + p] = rec[p];
          a.slot[base + p] = static_cast<int8_t>(sl[p]);
          d.sl[p] = sl[p];
          a.matched[base + p] = mat[p];
          if (rec[p]) {
            a.cache_e[base + sl[p]] = e[p];
            a.cache_w[base + sl[p]] = w[p];
          } else if (a.reused_meta_policy) {
            a.cache_w[base + sl[p]] = w[p];
          }
        }
      }
      a.token_any[i] = any;
    }
  }
  d.any = any;
  d.bad = bad;
  d.shared_row = valid && !bad && a.n_shared && (a.refresh || a.shared_policy || any);
  d.n_matched = n_matched;
  d.n_rec = n_rec;
  d.n_near = n_near;
}

}  // namespace moeca
