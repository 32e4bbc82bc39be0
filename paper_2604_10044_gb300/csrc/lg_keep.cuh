// The retained set I_keep of one sequence (LoopGuard Sec. 5.3, Eq. 10, Eq. 11), shared by the
// kernels that form it: the loop-onset test (lg_detect_prune), the token-level monitor
// (lg_token_detect_prune) and the stand-alone retained-set kernel (lg_prune_compact).
#pragma once
#include <stdint.h>

#include "lg_common.cuh"
#include "lg_internal.h"

namespace lg {

// I_keep of one sequence in closed form (Sec. 5.3, Eq. 10, Eq. 11).  Its three pieces are
// disjoint ranges of slots taken in ascending order:
//   anchors   [0, cA), cA = min(N_anchor, n)
//   lattice   N_anchor + floor(j n_c / B_sparse), j < B_sparse, over the n_c rows between the
//             anchors and W^recent = [max(N_anchor, n - R), n); every such row if n_c <= B_sparse
//   recent    the last B_recent(level) rows of W^recent outside the span I_bad: the rows above
//             the span first, then, if they are fewer, the top rows below it
// so slot j of the kept list is a function of j alone and every thread writes its own slots.
struct KeepPlan {
  int count;              // rows kept
  int cA, cL;             // anchors, lattice rows
  int na, n_c, B_sp;      // lattice geometry
  int lo_start, lo_cnt;   // recent rows below the span
  int hi_start;           // recent rows above the span (up to n)
};

// false when the budget leaves no room for the pieces (B_sparse < 0)
__device__ __forceinline__ bool keep_plan(int n, int B, int flag, int span_lo, int span_hi,
                                          int level, const lg_guard_params &p, KeepPlan &k) {
  const int hd = min(p.headroom, B / 4);
  const int T = B - hd;
  const int R = B / 2;
  const int B_rec = (B / 4) >> (flag ? level : 0);  // a budget event prunes at level 0
  const int B_sp = T - p.n_anchor - B / 4;
  if (B_sp < 0) return false;
  const int na = p.n_anchor;
  const int rw_lo = min(max(na, n - R), n);
  k.na = na;
  k.B_sp = B_sp;
  k.cA = min(na, n);
  k.n_c = max(0, rw_lo - na);
  k.cL = min(k.n_c, B_sp);
  // the span clipped to W^recent; a budget event has none
  const int blo = flag ? max(span_lo, rw_lo) : 0;
  const int bhi = flag ? min(span_hi, n) : 0;
  int cR;
  if (blo < bhi) {
    const int above = n - bhi;
    if (above >= B_rec) {
      k.lo_start = blo;
      k.lo_cnt = 0;
      k.hi_start = n - B_rec;
      cR = B_rec;
    } else {
      const int below = min(B_rec - above, blo - rw_lo);
      k.lo_start = blo - below;
      k.lo_cnt = below;
      k.hi_start = bhi;
      cR = below + above;
    }
  } else {
    cR = min(B_rec, n - rw_lo);
    k.lo_start = n;
    k.lo_cnt = 0;
    k.hi_start = n - cR;
  }
  k.count = k.cA + k.cL + cR;
  return true;
}

__device__ __forceinline__ int keep_row(const KeepPlan &k, int j) {
  if (j < k.cA) return j;
  j -= k.cA;
  if (j < k.cL) return k.na + (k.n_c <= k.B_sp ? j : (int)(((int64_t)j * k.n_c) / k.B_sp));
  j -= k.cL;
  return j < k.lo_cnt ? k.lo_start + j : k.hi_start + (j - k.lo_cnt);
}

// One sequence's prune decision and kept list, written by the nthreads threads of a CTA:
// no prune (no trigger and n <= B) -> kept_count = -1; otherwise the kept list, its size,
// and len = that size.  Returns the status code to raise (0 = none).
__device__ __forceinline__ int write_keep(const lg_cache &c, int b, int n, int B, int flag,
                                          int span_lo, int span_hi, int level,
                                          const lg_guard_params &p, int32_t *kept_idx,
                                          int32_t *kept_count, int max_keep, int max_len,
                                          int tid, int nthreads) {
  if (!flag && n <= B) {
    if (tid == 0) kept_count[b] = -1;
    return 0;
  }
  if (n > max_len) return LG_ERR_CAPACITY;
  KeepPlan k;
  if (!keep_plan(n, B, flag, span_lo, span_hi, level, p, k) || B > max_keep) return LG_ERR_BUDGET;
  int32_t *out = kept_idx + (int64_t)b * max_keep;
  for (int j = tid; j < k.count; j += nthreads) out[j] = keep_row(k, j);
  if (tid == 0) {
    kept_count[b] = k.count;
    c.len[b] = k.count;
  }
  return 0;
}

}  // namespace lg
