// lg_votes.cuh -- how the loop-onset test takes its votes without dividing (Sec. 5.2, Eq. 8;
// App. B.2 for the stall test).  Host and device code: the detect kernel uses these functions,
// and a host test compiles the same source to check them against the fp64 quotients.
#pragma once

#include <math.h>
#include <stdint.h>

#include <vector_types.h>

#if defined(__CUDACC__)
#define LG_VOTE_FN __host__ __device__
#define LG_VOTE_INLINE __forceinline__
#define LG_VOTE_NOINLINE __noinline__
#else
#define LG_VOTE_FN
#define LG_VOTE_INLINE inline
#define LG_VOTE_NOINLINE __attribute__((noinline))
#endif

namespace lg {

constexpr double kFixUnit = 1.0 / 1099511627776.0;  // 2^-40: the statistics sums' unit

// The votes are the decisions of fp64 quotients against fp64 thresholds (vote 1: novel / w <
// theta_ttr; Stall: tail / stall_len < theta_nov; vote 2: sum H / (L H_q ln n) < theta_ent;
// vote 3: sum S n / (W_s L H_q) >= theta_lift).  Bounds formed beside the sums decide them
// without a division except next to the threshold, where the quotient itself is taken, so every
// vote is exactly the quotient's decision.
//
// Count votes, k / m < theta for 0 <= k <= m < 2^29: from t = RN(theta m), whose rounding error
// is below 2^-23 while |t| < 2^30, a = ceil(t - 2^-20) and z = floor(t + 2^-20) (count_bounds).
// A count k < a lies below theta m by more than 2^-20 - 2^-23, so k / m lies below theta by more
// than the quotient's rounding (2^-53 for k <= m); likewise k > z lies above.  Only a count
// within 2^-20 of theta m (an exact tie, in practice) divides.
LG_VOTE_FN LG_VOTE_INLINE int2 count_bounds(double t) {
  if (t != t) return int2{0, -1};  // NaN: every count is "above" (the vote fails)
  const double d = 0.00000095367431640625;  // 2^-20
  const double lo = fmin(fmax(t - d, -1.0), 1073741824.0);
  const double hi = fmin(fmax(t + d, -1.0), 1073741824.0);
  return int2{(int)ceil(lo), (int)floor(hi)};
}

// The quotients themselves, out of line: they run only next to a threshold, and a call keeps
// the compiler from evaluating their fp64 divisions on the common path.
static LG_VOTE_FN LG_VOTE_NOINLINE int count_quotient_below(int k, int m, double theta) {
  return (double)k / (double)m < theta;
}

// RN(RN(RN(x 2^-40) mul) / RN(den_a den_b)) against theta: below it, or at least it (at_least)
static LG_VOTE_FN LG_VOTE_NOINLINE int sum_quotient_vote(long long x, int mul, double den_a, double den_b,
                                              double theta, int at_least) {
  const double q = (double)x * kFixUnit * (double)mul / (den_a * den_b);
  return at_least ? q >= theta : q < theta;
}

LG_VOTE_FN LG_VOTE_INLINE bool count_vote(int k, int2 az, int m, double theta) {
  if (k < az.x) return true;
  if (k > az.y) return false;
  return count_quotient_below(k, m, theta);
}

// Sum votes on a fixed-point sum x (units of 2^-40) against t, the threshold times the quotient's
// divisor: b = ceil(RN(t) 2^40), and a margin within which the rounded quotient may land on
// either side of theta (each side carries a few fp64 roundings, relative 2^-50 at most; the
// margin is 2^-45 of b, plus 4).  x < b - margin is below, x > b + margin above; in between, and
// for a NaN or out-of-range t (margin < 0), the quotient decides.
struct FixBound {
  long long b, margin;
};

LG_VOTE_FN LG_VOTE_INLINE FixBound fix_bound(double t) {
  FixBound f;
  if (!(fabs(t) < 4194304.0)) {  // NaN, or |t| 2^40 >= 2^62
    f.b = 0;
    f.margin = -1;
    return f;
  }
  f.b = (long long)ceil(t * 1099511627776.0);  // the scaling by 2^40 is exact
  f.margin = ((f.b < 0 ? -f.b : f.b) >> 45) + 4;
  return f;
}

// -1: x 2^-40 is below t, +1: above, 0: too close to tell (take the quotient)
LG_VOTE_FN LG_VOTE_INLINE int fix_side(long long x, const FixBound &f) {
  if (f.margin < 0) return 0;
  if (x < f.b - f.margin) return -1;
  if (x > f.b + f.margin) return 1;
  return 0;
}

}  // namespace lg
