"""The arithmetic behind the loop-onset test's votes on the GPU (Sec. 5.2's votes and the stall
gate), checked on the host.  The detect kernel takes each vote as the decision of an fp64
quotient against an fp64 threshold, but divides only next to the threshold: a count k of novel
rows is compared with a = ceil(t - 2^-20) and z = floor(t + 2^-20), t = RN(theta m), and only
a <= k <= z (a count within 2^-20 of theta m) divides; a fixed-point sum x
(units of 2^-40) is compared with b = ceil(RN(t) 2^40) outside a margin of 2^-45 b + 4, and only
inside it divides.  These tests mirror that logic and check that it reproduces the quotient's
decision for every count the window allows and for sums on both sides of the threshold, with
thresholds on, next to and between the quotients."""
import math
import random

import numpy as np


def count_bounds(t):
    if t != t:
        return 0, -1
    d = 2.0 ** -20
    lo = min(max(t - d, -1.0), 1073741824.0)
    hi = min(max(t + d, -1.0), 1073741824.0)
    return math.ceil(lo), math.floor(hi)


def count_vote(k, az, m, theta):
    if k < az[0]:
        return True
    if k > az[1]:
        return False
    return k / m < theta


def fix_bound(t):
    if not abs(t) < 4194304.0:
        return 0, -1
    b = math.ceil(t * 1099511627776.0)
    return b, (abs(b) >> 45) + 4


def fix_side(x, bound):
    b, margin = bound
    if margin < 0:
        return 0
    if x < b - margin:
        return -1
    if x > b + margin:
        return 1
    return 0


UNIT = 1.0 / 1099511627776.0


def _thresholds():
    th = {0.2, 0.02, 0.7, 2.0, 0.5, 1.0, 0.0, 1e-9, 3e5, -0.1, float("nan"), float("inf")}
    for m0 in (3, 5, 7, 10, 64, 255, 256, 300):
        for j in range(0, m0 + 1, max(1, m0 // 12)):
            th.add(j / m0)
    rng = random.Random(3)
    th.update(rng.random() for _ in range(20))
    out = set()
    for v in th:
        out.update({v, float(np.nextafter(v, 2.0)), float(np.nextafter(v, -1.0))})
    return sorted(out, key=lambda v: (math.isnan(v), v))


def test_count_vote_is_the_quotient_decision():
    divided = 0
    for theta in _thresholds():
        for m in range(1, 301):
            az = count_bounds(theta * m)
            for k in range(0, m + 1):
                assert count_vote(k, az, m, theta) == (k / m < theta), (theta, m, k)
                divided += az[0] <= k <= az[1]
    # only exact ties divide: at most one count per (theta, m), and none for most
    assert divided <= len(_thresholds()) * 300


def test_count_bounds_of_the_default_gates():
    """theta_ttr = 0.2 over windows of 1..256 rows, theta_nov = 0.02 over the 4-row stall test:
    theta m is never within 2^-20 of an integer but at m = 5j, where 0.2 m rounds to j"""
    for m in range(1, 257):
        a, z = count_bounds(0.2 * m)
        assert (a > z) == (m % 5 != 0), m
    assert count_bounds(0.02 * 4) == (1, 0)


def test_count_bounds_edge_values():
    assert count_bounds(float("nan")) == (0, -1)
    assert count_bounds(-3.0) == (-1, -1) and count_bounds(0.0) == (0, 0)
    assert count_bounds(float("inf")) == (1 << 30, 1 << 30)
    assert count_bounds(51.2) == (52, 51) and count_bounds(51.0) == (51, 51)


def _sum_cases():
    """(x, quotient decision, bound) for the entropy vote: sum H / (L H_q ln n) < theta_ent"""
    rng = random.Random(11)
    for _ in range(400):
        nh = rng.choice([1, 16, 448, 1024, 2048])
        n = rng.randint(2, 140000)
        logn = math.log(n)
        theta = rng.choice([0.7, rng.random(), float(np.nextafter(0.7, 1.0))])
        bound = fix_bound(theta * nh * logn)
        b, margin = bound
        for dx in (-3 * margin, -margin - 1, -margin, -1, 0, 1, margin, margin + 1, 3 * margin,
                   rng.randint(-10 * margin, 10 * margin)):
            x = b + dx
            yield x, (x * UNIT) / (nh * logn) < theta, bound


def test_fix_side_agrees_with_the_quotient():
    decisive = 0
    for x, below, bound in _sum_cases():
        side = fix_side(x, bound)
        if side:
            decisive += 1
            assert (side < 0) == below, (x, bound)
    assert decisive > 1000


def test_fix_side_lift_vote():
    """vote 3: sum S n / (W_s L H_q) >= theta_lift against t = theta_lift W_s L H_q / n"""
    rng = random.Random(5)
    decisive = 0
    for _ in range(2000):
        nh, n = rng.choice([16, 448, 1024]), rng.randint(1, 140000)
        ws = min(64, n)
        theta = rng.choice([2.0, 1.0 + rng.random(), float(np.nextafter(2.0, 0.0))])
        bound = fix_bound(theta * ws * nh / n)
        b, margin = bound
        for x in (b - margin - 1, b + margin + 1, b + rng.randint(-5 * margin, 5 * margin)):
            side = fix_side(x, bound)
            if side:
                decisive += 1
                assert (side > 0) == ((x * UNIT) * n / (ws * nh) >= theta), (x, bound, n)
    assert decisive > 3000


def test_fix_bound_degenerate_thresholds_defer_to_the_quotient():
    assert fix_bound(float("nan"))[1] < 0 and fix_bound(1e30)[1] < 0
    assert fix_side(123, fix_bound(float("nan"))) == 0
