"""Pins of the oracle's loop-onset test (Sec. 5.2, Eq. 8, Eq. 9, App. B.2).

Sketch bits and row matching are checked on rows with known signs and known Hamming
distances; the windowed novelty rate, the stall gate, the suffix self-alignment period and
the bad span against brute force written here from the definitions on tiny inputs; the
vote, warmup, cooldown and level rules on scripted statistic sequences.
"""
import math

import numpy as np
import pytest

import oracle


def test_sketch_sign_bits_fp32_and_bf16():
    row = np.array([(-1.0) ** (j % 3 == 0) * (j + 1) for j in range(64)], dtype=np.float32)
    row[5] = -0.0     # raw sign bit: -0 counts as negative
    row[6] = 0.0
    words = oracle.sketch(row)
    expect = [0, 0]
    for j in range(64):
        if math.copysign(1.0, float(row[j])) < 0:
            expect[j // 32] |= 1 << (j % 32)
    assert words.tolist() == expect
    bits = row.view(np.uint32) >> 16
    assert oracle.sketch(bits.astype(np.uint16)).tolist() == expect


@pytest.mark.parametrize("dist,thr,ok", [(0, 0, True), (3, 3, True), (4, 3, False),
                                         (64, 64, True), (65, 64, False)])
def test_match_threshold_inclusive(dist, thr, ok):
    a = np.zeros(4, dtype=np.uint32)
    b = a.copy()
    for k in range(dist):
        b[k % 4] |= np.uint32(1 << (k // 4))
    assert oracle.match(a, b, thr) is ok


def _brute(sk, n, W, thr, stall_len, theta_nov, p_min, p_max, m_rep, l_min, R):
    """the definitions, written out directly on Python ints"""
    def match(i, j):
        return sum(bin(int(x) ^ int(y)).count("1") for x, y in zip(sk[i], sk[j])) <= thr
    w = min(W, n)
    lo = n - w
    novel = [all(not match(i, j) for j in range(lo, i)) for i in range(lo, n)]
    ttr = sum(novel) / w
    stall = w >= stall_len and sum(novel[-stall_len:]) / stall_len < theta_nov
    P = 0
    for p in range(p_min, p_max + 1):
        L = max(m_rep * p, l_min)
        if n < L + p:
            continue
        if all(match(i, i - p) for i in range(n - L, n)):
            P = p
            break
    span = (0, 0)
    if P:
        L = max(m_rep * P, l_min)
        lo_ext = max(P, n - R)
        s = n - L
        if s < lo_ext:
            s = lo_ext
        else:
            while s - 1 >= lo_ext and match(s - 1, s - 1 - P):
                s -= 1
        span = (max(s - P, n - R, 0), n)
    return ttr, stall, P, span


def _sketches(rng, n, nwords, period=None, start=None, flips=0):
    sk = rng.integers(0, 2 ** 32, size=(n, nwords), dtype=np.uint64).astype(np.uint32)
    if period:
        for i in range(start, n):
            sk[i] = sk[start - period + (i - start) % period]
            for _ in range(flips):
                w = rng.integers(nwords)
                sk[i, w] ^= np.uint32(1 << int(rng.integers(32)))
    return sk


def _stats_for(ebar, lbar, L, H, n, Ws):
    st = np.zeros((L, H, 4))
    st[..., 2] = ebar * math.log(n)
    st[..., 3] = lbar * Ws / n
    return st


@pytest.mark.parametrize("seed", range(12))
def test_novelty_tailrep_span_brute_force(seed):
    rng = np.random.default_rng(seed)
    nwords = 2
    n = int(rng.integers(20, 49))
    looping = seed % 3 != 0
    period = int(rng.integers(1, 7)) if looping else None
    start = int(rng.integers(period + 1, n - 2)) if looping else None
    sk = _sketches(rng, n, nwords, period, start, flips=int(rng.integers(0, 3)))
    prm = oracle.params(W=24, stall_len=4, p_min=1, p_max=12, m_rep=3, l_min=6,
                        tau_ham=0.06, t_min=0)
    thr = int(math.floor(prm.tau_ham * nwords * 32))
    budget = 40
    # force a trigger (strong signals) so the span is produced
    st = oracle.new_state(t_gen=10)
    stats = _stats_for(0.1, 9.0, 2, 3, n, min(prm.suffix_w, n))
    flag, span, diag = oracle.detect(stats, sk, budget, prm, st)
    ttr, stall, P, span_b = _brute(sk, n, prm.W, thr, prm.stall_len, prm.theta_nov, prm.p_min,
                                   prm.p_max, prm.m_rep, prm.l_min, budget // 2)
    assert diag["ttr"] == pytest.approx(ttr, abs=1e-15)
    assert bool(diag["stall"]) == stall
    assert int(diag["P"]) == P
    assert flag == int(stall or P > 0)
    if flag and P:
        assert span == span_b
    else:
        assert span == (0, 0)


def test_planted_period_found_and_span_covers_all_copies():
    rng = np.random.default_rng(7)
    n, P, start = 400, 24, 208
    sk = _sketches(rng, n, 16, P, start)
    prm = oracle.params()
    st = oracle.new_state()
    stats = _stats_for(0.4, 3.0, 1, 8, n, 64)
    budget = 1024          # R = 512 > n: the extension runs back to the loop's first copy
    flag, span, diag = oracle.detect(stats, sk, budget, prm, st)
    assert flag == 1 and int(diag["P"]) == P
    # rows from `start` match the row P earlier; the span includes the source block
    assert span == (start - P, n)
    budget = 256           # R = 128: I_bad is clipped to the recent window [n - R, n)
    st = oracle.new_state()
    flag, span, _ = oracle.detect(stats, sk, budget, prm, st)
    assert span == (n - 128, n)


def test_multiple_of_period_is_not_chosen():
    rng = np.random.default_rng(8)
    n, P, start = 300, 10, 100
    sk = _sketches(rng, n, 8, P, start)
    _, _, diag = oracle.detect(_stats_for(0.4, 3.0, 1, 2, n, 64), sk, 1024, oracle.params(),
                               oracle.new_state())
    assert int(diag["P"]) == P     # 20, 30, ... also align, the smallest period is reported


def test_vote_and_gates():
    """Warn = sum of 3 indicators >= K; Trigger needs warmup, cd = 0, Warn and a persistence
    gate.  Signals: diversity (novel fraction < 0.2), concentration (mean normalised entropy
    < theta_ent), locking (mean suffix lift >= theta_lift)."""
    rng = np.random.default_rng(9)
    n = 300
    looped = _sketches(rng, n, 8, 5, 40)        # TTR = 5/256 < 0.2, stall, period 5
    fresh = _sketches(rng, n, 8)                # every row novel, no period
    prm = oracle.params()
    cases = [  # (sketch, ebar, lbar, expect_warn, expect_trigger)
        (looped, 0.9, 1.0, False, False),       # diversity only: 1 vote
        (looped, 0.5, 1.0, True, True),         # diversity + concentration
        (looped, 0.9, 2.5, True, True),         # diversity + locking
        (fresh, 0.5, 2.5, True, False),         # 2 votes but no stall / tail repetition
        (fresh, 0.9, 2.5, False, False),
    ]
    for sk, e, lam, warn, trig in cases:
        st = oracle.new_state()
        flag, _, diag = oracle.detect(_stats_for(e, lam, 2, 4, n, 64), sk, 4096, prm, st)
        assert bool(diag["warn"]) == warn, (e, lam)
        assert flag == int(trig), (e, lam)
    # the lift vote is inclusive: S * n / W_s exactly 2.0 (n = 256, W_s = 64, S = 0.5) votes
    sk256 = _sketches(rng, 256, 8, 5, 40)
    st = oracle.new_state()
    stats = _stats_for(0.9, 2.0, 2, 4, 256, 64)
    assert np.all(stats[..., 3] == 0.5)
    flag, _, diag = oracle.detect(stats, sk256, 4096, prm, st)
    assert diag["lbar"] == 2.0 and diag["sig3"] == 1 and diag["sig2"] == 0 and flag == 1
    # NaN statistics switch their signal off
    st = oracle.new_state()
    stats = _stats_for(0.5, 2.5, 2, 4, n, 64)
    stats[0, 0, 2] = np.nan
    stats[1, 1, 3] = np.nan
    flag, _, diag = oracle.detect(stats, fresh, 4096, prm, st)
    assert diag["sig2"] == 0 and diag["sig3"] == 0 and flag == 0


def test_warmup_cooldown_and_levels():
    rng = np.random.default_rng(10)
    n = 300
    sk = _sketches(rng, n, 8, 5, 40)
    stats = _stats_for(0.5, 3.0, 1, 4, n, 64)
    prm = oracle.params()
    st = oracle.new_state(t_gen=0)
    fired = []
    for t in range(200):
        f, _, _ = oracle.detect(stats, sk, 4096, prm, st)
        fired.append((t, f, st.level))
    trig_steps = [t for t, f, _ in fired if f]
    # warmup: nothing before t_min = 64; then one trigger every cooldown + 1 = 33 steps
    assert trig_steps[0] == 64
    assert all(b - a == 33 for a, b in zip(trig_steps, trig_steps[1:]))
    # re-triggers within 64 steps raise the level by one, capped at 3
    levels = [lvl for t, f, lvl in fired if f]
    assert levels[:5] == [0, 1, 2, 3, 3]
    assert st.n_int == len(trig_steps)
    # a trigger long after the last one resets the level to 0
    st = oracle.new_state(t_gen=100)
    st.level, st.last_trig = 3, 0
    f, _, _ = oracle.detect(stats, sk, 4096, prm, st)
    assert f == 1 and st.level == 0 and st.cd == 32 and st.t_gen == 101


def test_short_sequences():
    prm = oracle.params()
    st = oracle.new_state()
    sk = np.zeros((1, 8), dtype=np.uint32)
    flag, span, diag = oracle.detect(_stats_for(1.0, 1.0, 1, 2, 2, 2)[:, :, :], sk, 256, prm, st)
    assert flag == 0 and span == (0, 0) and diag["ttr"] == 1.0


# --------------------------------------------------------------------------- threshold boundaries

def test_entropy_vote_normalises_by_ln_n():
    """stats with H = c ln n in every head give a mean normalised entropy of exactly c (up to
    rounding), for any n: the divisor is ln n (Sec. 5.2's concentration signal restated)"""
    rng = np.random.default_rng(12)
    for n in (2, 100, 4096):
        sk = _sketches(rng, n, 4)
        for c in (0.3, 0.9):
            _, _, diag = oracle.detect(_stats_for(c, 1.0, 2, 3, n, min(64, n)), sk, 8192,
                                       oracle.params(), oracle.new_state())
            assert diag["ebar"] == pytest.approx(c, rel=1e-12), (n, c)


def test_votes_are_strict_at_their_thresholds():
    """vote 1 fires for a novel fraction below theta_ttr, not at it; vote 2 for a mean
    normalised entropy below theta_ent, not at it (Eq. 8)"""
    rng = np.random.default_rng(13)
    base = _sketches(rng, 2, 4)
    sk = np.stack([base[i % 2] for i in range(10)])      # rows 0 and 1 novel, the rest repeats
    prm = oracle.params(W=10, stall_len=4)
    _, _, diag = oracle.detect(_stats_for(0.9, 1.0, 1, 2, 10, 10), sk, 4096, prm,
                               oracle.new_state())
    assert diag["ttr"] == 0.2 and diag["sig1"] == 0      # 2 / 10 == theta_ttr: no vote
    sk1 = np.stack([base[0]] * 10)
    _, _, diag = oracle.detect(_stats_for(0.9, 1.0, 1, 2, 10, 10), sk1, 4096, prm,
                               oracle.new_state())
    assert diag["ttr"] == 0.1 and diag["sig1"] == 1
    # the entropy vote at exactly theta_ent: take theta_ent from the oracle's own mean
    stats = _stats_for(0.6, 1.0, 2, 3, 300, 64)
    sk300 = _sketches(rng, 300, 4)
    _, _, d0 = oracle.detect(stats, sk300, 4096, oracle.params(), oracle.new_state())
    e = d0["ebar"]
    _, _, d1 = oracle.detect(stats, sk300, 4096, oracle.params(theta_ent=e), oracle.new_state())
    assert d1["sig2"] == 0
    _, _, d2 = oracle.detect(stats, sk300, 4096, oracle.params(theta_ent=float(np.nextafter(e, 2.0))),
                             oracle.new_state())
    assert d2["sig2"] == 1


def test_stall_counts_the_first_row_of_its_tail():
    """Stall looks at the last theta_stall = 4 rows: one novel row among them (the earliest,
    n - 4) gives a novel fraction of 1/4 >= theta_nov, so no stall; with it repeated too, stall"""
    rng = np.random.default_rng(14)
    sk = _sketches(rng, 20, 4)
    sk[17:20] = sk[0:3]                                  # rows 17..19 repeat earlier rows
    prm = oracle.params(W=20, stall_len=4)
    _, _, diag = oracle.detect(_stats_for(0.9, 1.0, 1, 2, 20, 20), sk, 4096, prm,
                               oracle.new_state())
    assert diag["stall"] == 0                            # row 16 is novel
    sk[16] = sk[5]
    _, _, diag = oracle.detect(_stats_for(0.9, 1.0, 1, 2, 20, 20), sk, 4096, prm,
                               oracle.new_state())
    assert diag["stall"] == 1


def test_tail_repetition_needs_l_min_rows():
    """TailRep checks the last max(m_rep P, l_min) rows (App. B.2 debounce): a period-4 repeat
    over the last 20 rows is not enough with l_min = 32 (m_rep P = 12), over the last 40 it is"""
    rng = np.random.default_rng(15)
    prm = oracle.params(m_rep=3, l_min=32, p_min=1, p_max=16)
    for tail, P in ((20, 0), (40, 4)):
        n = 100
        sk = _sketches(rng, n, 4, 4, n - tail)
        _, _, diag = oracle.detect(_stats_for(0.9, 1.0, 1, 2, n, 64), sk, 4096, prm,
                                   oracle.new_state())
        assert int(diag["P"]) == P, tail


def test_retrigger_exactly_at_the_window_escalates():
    """a trigger exactly retrig_window = 64 steps after the previous one counts as 'shortly
    after' (Sec. 5.3) and raises the level; one step later it resets the level"""
    rng = np.random.default_rng(16)
    n = 300
    sk = _sketches(rng, n, 8, 5, 40)
    stats = _stats_for(0.5, 3.0, 1, 4, n, 64)
    for gap, level in ((64, 2), (65, 0)):
        st = oracle.new_state(t_gen=200)
        st.level, st.last_trig = 1, 200 - gap
        f, _, _ = oracle.detect(stats, sk, 4096, oracle.params(), st)
        assert f == 1 and st.level == level, gap


def test_lift_of_a_cache_shorter_than_the_suffix():
    """W_s = min(64, n): with n = 40 rows the suffix is the whole cache, S = 1 and the lift is
    exactly 1 (uniform attention's value), not 40 / 64"""
    rng = np.random.default_rng(18)
    n = 40
    stats = np.zeros((1, 2, 4))
    stats[..., 2] = 0.5 * math.log(n)
    stats[..., 3] = 1.0
    _, _, diag = oracle.detect(stats, _sketches(rng, n, 4), 4096, oracle.params(),
                               oracle.new_state())
    assert diag["lbar"] == 1.0


def test_stall_with_a_window_of_exactly_theta_stall_rows():
    """the stall test runs once the window holds theta_stall rows (w >= theta_stall): four
    identical rows have one novel row, 1/4 < theta_nov = 0.5"""
    sk = np.zeros((4, 4), dtype=np.uint32)
    prm = oracle.params(W=4, stall_len=4, theta_nov=0.5)
    _, _, diag = oracle.detect(_stats_for(0.9, 1.0, 1, 2, 4, 4), sk, 4096, prm,
                               oracle.new_state())
    assert diag["stall"] == 1


def test_tail_repetition_at_the_shortest_cache_that_can_show_it():
    """a period P is testable once n >= max(m_rep P, l_min) + P: a cache of exactly 12 + 4 rows
    repeating with period 4 (m_rep 3, l_min 6) reports P = 4"""
    rng = np.random.default_rng(19)
    sk = _sketches(rng, 16, 4, 4, 4)
    prm = oracle.params(m_rep=3, l_min=6, p_min=4, p_max=8)
    _, _, diag = oracle.detect(_stats_for(0.9, 1.0, 1, 2, 16, 16), sk, 4096, prm,
                               oracle.new_state())
    assert int(diag["P"]) == 4


@pytest.mark.parametrize("theta_nov", [0.02, 0.1, 0.25, 0.2501, 0.3])
def test_stall_gate_takes_the_novel_fraction_of_the_last_rows(theta_nov):
    """Stall: the novel fraction of the last stall_len = 4 rows is below theta_nov.  The
    fraction takes only the values k/4, so every theta_nov in (0, 1/4] gives the same gate
    (none of the last 4 rows novel) and the paper's 0.02 acts as any of them; above 1/4 one
    novel row of four no longer blocks it"""
    rng = np.random.default_rng(17)
    n = 60
    prm = oracle.params(theta_nov=theta_nov, t_min=0)
    stats = _stats_for(0.4, 3.0, 1, 2, n, 64)
    for k_novel in (0, 1, 2):
        sk = _sketches(rng, n, 8)                  # random rows: every row novel
        for j, i in enumerate(range(n - 4, n)):
            if j >= k_novel:
                sk[i] = sk[10 + j]                 # a copy of an earlier window row
        _, _, diag = oracle.detect(stats, sk, 1024, prm, oracle.new_state())
        assert bool(diag["stall"]) == (k_novel / 4 < theta_nov), (k_novel, theta_nov)
