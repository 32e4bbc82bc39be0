"""The arithmetic behind the loop-onset test's votes on the GPU (Sec. 4.2's three signals and the
stall gate), checked on the host.  The detect kernel does not divide: it compares a count of
novel rows k with ceil(theta * m) (theta a float parameter, m the window or stall length) and a
fixed-point sum x (units of 2^-40) with ceil(t * 2^40).  These tests check that the count form
is the same decision as the fp64 quotient k / m < theta for every count and length the window
allows, thresholds on and next to the quotients included, and that the fixed-point form is the
exact comparison of the rational x 2^-40 with t."""
import math
from fractions import Fraction

import numpy as np


def count_bound(t):
    """the least integer c >= 0 with: k < t exactly when k < c, for every count k >= 0"""
    if not t > 0.0:
        return 0
    return 1 << 30 if t > 1073741824.0 else math.ceil(t)


def fix_bound(t):
    x = t * 1099511627776.0
    lim = 4611686018427387904.0
    if x >= lim:
        return 1 << 62
    if x <= -lim:
        return -(1 << 62)
    return math.ceil(x)


def _thresholds():
    th = {np.float32(v) for v in (0.2, 0.02, 0.7, 2.0, 0.5, 1.0, 0.0, 1e-9, 3e5)}
    for m0 in (3, 7, 10, 64, 255, 256):
        for j in range(0, m0 + 1, max(1, m0 // 16)):
            th.add(np.float32(j / m0))
    out = set()
    for v in th:
        out.update({v, np.nextafter(v, np.float32(2)), np.nextafter(v, np.float32(-1))})
    return sorted(float(v) for v in out)


def test_count_bound_is_the_quotient_decision():
    ms = np.arange(1, 301)
    k = np.arange(0, 301)
    K, M = np.meshgrid(k, ms, indexing="ij")
    ok = K <= M
    q = K.astype(np.float64) / M.astype(np.float64)  # correctly rounded, as the fp64 division
    for theta in _thresholds():
        bounds = np.array([count_bound(theta * float(m)) for m in ms])
        via_count = K < bounds[None, :]
        via_quot = q < theta
        assert np.array_equal(via_count[ok], via_quot[ok]), theta


def test_count_bound_edge_values():
    assert count_bound(float("nan")) == 0 and count_bound(-3.0) == 0 and count_bound(0.0) == 0
    assert count_bound(float("inf")) == 1 << 30
    assert count_bound(51.2) == 52 and count_bound(51.0) == 51  # k < 51 <=> k < 51


def test_fix_bound_is_the_exact_comparison():
    rng = np.random.default_rng(7)
    ts = [0.7 * 448 * math.log(3853), 2.0 * 64 * 448 / 3853, 0.2, 1e-12, 5e3, -1.5]
    ts += list(rng.uniform(0, 1e4, 50))
    for t in ts:
        b = fix_bound(t)
        exact = Fraction(t) * (1 << 40)
        for x in (b - 2, b - 1, b, b + 1, int(exact), int(exact) - 1):
            lhs = Fraction(x, 1 << 40) < Fraction(t)
            assert lhs == (x < b), (t, x)
            assert (Fraction(x, 1 << 40) >= Fraction(t)) == (x >= b), (t, x)
    assert fix_bound(1e30) == 1 << 62 and fix_bound(-1e30) == -(1 << 62)
