// Host check of paper_2604_10044_gb300/csrc/lg_votes.cuh, the functions the detect kernel uses
// to take its votes: compiled from the same source for the CPU and compared with the fp64
// quotient decisions they stand for (Sec. 5.2, Eq. 8), over every count of windows of up to
// 300 rows and over sums on both sides of each bound.  Exit status 0 when all agree.
#include <cmath>
#include <cstdio>
#include <random>
#include <vector>

#include "lg_votes.cuh"

using namespace lg;

static int fails = 0;

static void check(bool ok, const char *what, double a, double b, double c) {
  if (!ok && fails++ < 10) std::printf("mismatch %s %.17g %.17g %.17g\n", what, a, b, c);
}

int main() {
  std::vector<double> th = {0.2, 0.02, 0.7, 2.0, 0.5, 1.0, 0.0, 1e-9, 3e5, -0.1, NAN, INFINITY};
  for (int m0 : {3, 5, 7, 10, 64, 255, 256, 300})
    for (int j = 0; j <= m0; j += (m0 / 12 > 1 ? m0 / 12 : 1)) th.push_back((double)j / m0);
  std::mt19937_64 rng(3);
  std::uniform_real_distribution<double> u(0.0, 1.0);
  for (int i = 0; i < 20; ++i) th.push_back(u(rng));
  const size_t base = th.size();
  for (size_t i = 0; i < base; ++i) {
    th.push_back(std::nextafter(th[i], 2.0));
    th.push_back(std::nextafter(th[i], -1.0));
  }
  long counted = 0, divided = 0;
  for (double theta : th)
    for (int m = 1; m <= 300; ++m) {
      const int2 az = count_bounds(theta * (double)m);
      for (int k = 0; k <= m; ++k) {
        const bool want = (double)k / (double)m < theta;
        check(count_vote(k, az, m, theta) == want, "count", theta, m, k);
        ++counted;
        divided += k >= az.x && k <= az.y;
      }
    }
  // the entropy vote: sum H / (L H_q ln n) < theta_ent, the lift vote: sum S n / (W_s L H_q)
  // >= theta_lift, each on sums around its bound
  long sums = 0, decisive = 0;
  std::uniform_int_distribution<int> un(2, 140000), pick(0, 4);
  const int nhs[5] = {1, 16, 448, 1024, 2048};
  for (int it = 0; it < 4000; ++it) {
    const int nh = nhs[pick(rng)], n = un(rng);
    const double logn = std::log((double)n);
    const double te = it % 3 == 0 ? 0.7 : (it % 3 == 1 ? u(rng) : std::nextafter(0.7, 1.0));
    const FixBound fe = fix_bound(te * (double)nh * logn);
    const int ws = n < 64 ? n : 64;
    const double tl = it % 2 ? 2.0 : 1.0 + u(rng);
    const FixBound fl = fix_bound(tl * (double)ws * (double)nh / (double)n);
    for (long long dx : {-3LL, -1LL, 0LL, 1LL, 3LL}) {
      for (int which = 0; which < 2; ++which) {
        const FixBound &f = which ? fl : fe;
        const long long x = f.b + dx * (f.margin > 0 ? f.margin : 1) + (long long)(u(rng) * 7) - 3;
        const int side = fix_side(x, f);
        bool vote, want;
        if (!which) {
          want = (double)x * kFixUnit / ((double)nh * logn) < te;
          vote = side ? side < 0 : sum_quotient_vote(x, 1, (double)nh, logn, te, 0);
        } else {
          want = (double)x * kFixUnit * (double)n / ((double)ws * (double)nh) >= tl;
          vote = side ? side > 0 : sum_quotient_vote(x, n, (double)ws, (double)nh, tl, 1);
        }
        check(vote == want, which ? "lift" : "entropy", (double)x, (double)n, which ? tl : te);
        ++sums;
        decisive += side != 0;
      }
    }
  }
  std::printf("counts %ld (divided %ld), sums %ld (decided without dividing %ld), mismatches %d\n",
              counted, divided, sums, decisive, fails);
  return fails != 0 || decisive == 0;
}
