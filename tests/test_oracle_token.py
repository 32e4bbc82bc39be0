"""Pins of the oracle's token-level monitor (Sec. 4.3, Sec. 5.2, Eq. 8, Eq. 9, App. B.2) against
hand-worked parses, closed forms and invariants; nothing here re-types the oracle's loops.

Readings: comp() of the CR indicator is the greedy LZ77 parse over token ids (a phrase is the
longest earlier match of >= 2 tokens, overlap allowed, else one literal), CR = phrases / window,
evaluated every cr_every tokens; a token of the window is novel when no earlier token of the
window equals it (TTR = novel / window); Stall = novel fraction of the last theta_stall tokens
below theta_nov; the p_max streak counts steps with p_max strictly above theta_conf."""
import math

import numpy as np
import pytest

import oracle

# --------------------------------------------------------------------------- LZ77 phrases

@pytest.mark.parametrize("x,phrases", [
    ([5], 1),                          # one literal
    ([1, 2, 3, 4], 4),                 # four literals
    ([7, 7, 7, 7, 7, 7], 2),           # 7 | ref(dist 1, len 5, overlapping)
    ([1, 2, 1, 2, 1, 2, 1], 3),        # 1 | 2 | ref(dist 2, len 5)
    ([1, 2, 1, 3], 4),                 # "1 3" has no earlier match of 2 tokens: four literals
    ([1, 2, 3, 1, 2, 4, 1, 2, 3], 6),  # 1 | 2 | 3 | ref(1 2) | 4 | ref(1 2 3)
    # a b r a c a d a b r a: a | b | r | a | c | a | d | ref(a b r a)
    ([1, 2, 3, 1, 4, 1, 5, 1, 2, 3, 1], 8),
    # the longest earlier match wins, not the first: 1 | 2 | 9 | ref(1 2) | 3 | ref(1 2 3)
    ([1, 2, 9, 1, 2, 3, 1, 2, 3], 6),
])
def test_lz77_hand_worked(x, phrases):
    assert oracle.lz77_phrases(x) == phrases


@pytest.mark.parametrize("P,w", [(1, 5), (2, 9), (8, 256), (17, 200), (60, 121)])
def test_lz77_period_loop_closed_form(P, w):
    """a loop of P distinct tokens repeated to length w >= P + 2: P literals, then one
    overlapping reference to the end"""
    x = np.arange(w) % P + 100
    assert oracle.lz77_phrases(x) == P + 1


def test_lz77_bounds():
    """every first occurrence of a token starts a literal (a reference only copies earlier
    tokens), so distinct <= phrases <= length"""
    rng = np.random.default_rng(0)
    for k in range(200):
        w = int(rng.integers(1, 120))
        x = rng.integers(0, int(rng.integers(1, 12)), size=w)
        ph = oracle.lz77_phrases(x)
        assert len(set(x.tolist())) <= ph <= w
        assert oracle.lz77_phrases(np.arange(w)) == w


# --------------------------------------------------------------------------- the monitor

def _run(tokens, pmax, n0=4000, prm=None, tp=None, t_gen0=0, stop_at_trigger=True):
    """feed tokens one step at a time; the cache grows by one row per step from n0"""
    prm = prm or oracle.params()
    tp = tp or oracle.token_params()
    st, ts = oracle.new_state(t_gen0), oracle.new_token_state()
    events = []
    for t in range(len(tokens)):
        n = n0 + t + 1
        f, span, dg = oracle.token_detect(tokens[:t + 1], pmax[t], n, prm, tp, st, ts)
        if f:
            events.append((t, span, dg, n))
            if stop_at_trigger:
                break
    return events, st, ts


def _healthy_then_loop(H, P, L, base=10_000):
    healthy = np.arange(H, dtype=np.int32) + base           # H distinct tokens
    loop = (np.arange(L) % P + 1).astype(np.int32)          # P distinct tokens, repeated
    return np.concatenate([healthy, loop])


@pytest.mark.parametrize("P", [4, 8, 20])
def test_trigger_step_with_confidence_collapse(P):
    """W = 256, theta_ttr = 0.2: with the loop L tokens long the window holds 256 - L healthy
    distinct tokens and P loop tokens, so the diversity vote fires first at
    L* = floor(W + P - theta_ttr W) + 1; the p_max streak (0.95 > 0.9 for >= 6 steps) is the
    second vote, Stall and TailRep hold long before, and the CR vote has not fired yet."""
    H, W = 300, 256
    L_star = math.floor(W + P - 0.2 * W) + 1
    y = _healthy_then_loop(H, P, L_star + 40)
    pm = np.where(np.arange(len(y)) >= H, 0.95, 0.5)
    ev, st, _ = _run(y, pm)
    assert ev, "no trigger"
    t, span, dg, n = ev[0]
    assert t == H + L_star - 1, (t - H + 1, L_star)
    assert dg["sig1"] == 1 and dg["sig3"] == 1 and dg["sig2"] == 0 and dg["P"] == P
    # the span is the whole loop (the run extends back to its first period), in cache slots
    assert span == (n - L_star, n)
    assert st.n_int == 1 and st.cd == 32


def test_trigger_step_without_confidence():
    """p_max never above 0.9: Warn needs diversity and redundancy.  With the loop (P = 8) L
    tokens long the window parses into (256 - L) + P literals and one reference, so the CR vote
    holds from L > 256 + P + 1 - 0.12 W = 234.28; CR is evaluated when the token index is a
    multiple of 16: index 300 + L - 1, first at L = 245."""
    H, P = 300, 8
    y = _healthy_then_loop(H, P, 300)
    pm = np.full(len(y), 0.5)
    ev, _, _ = _run(y, pm)
    t, span, dg, n = ev[0]
    L = t - H + 1
    assert L == 245 and (H + L - 1) % 16 == 0
    assert dg["sig1"] == 1 and dg["sig2"] == 1 and dg["sig3"] == 0
    assert abs(dg["cr"] - (256 - L + P + 1) / 256) < 1e-12


def test_streak_is_strict_and_resets():
    """p_max = theta_conf exactly does not extend the streak; one low step resets it"""
    tp = oracle.token_params()
    prm = oracle.params()
    st, ts = oracle.new_state(0), oracle.new_token_state()
    seq = [0.95] * 5 + [0.9] + [0.91] * 7 + [0.2] + [0.99] * 3
    y = np.arange(len(seq), dtype=np.int32)
    streaks = []
    for t, p in enumerate(seq):
        _, _, dg = oracle.token_detect(y[:t + 1], p, 100 + t, prm, tp, st, ts)
        streaks.append(dg["streak"])
    assert streaks == [1, 2, 3, 4, 5, 0, 1, 2, 3, 4, 5, 6, 7, 0, 1, 2, 3]


def test_ttr_and_stall_definitions():
    """TTR over the last min(W, t) tokens; Stall from the last theta_stall tokens"""
    prm = oracle.params(W=8)
    tp = oracle.token_params()
    st, ts = oracle.new_state(0), oracle.new_token_state()
    y = np.array([1, 2, 3, 4, 5, 6, 7, 8, 1, 2, 3, 4, 9, 9, 9, 9, 9], dtype=np.int32)
    got = []
    for t in range(len(y)):
        _, _, dg = oracle.token_detect(y[:t + 1], 0.5, 50 + t, prm, tp, st, ts)
        got.append((dg["ttr"], dg["stall"]))
    # t = 7: window 1..8 all distinct; t = 11: window 5 6 7 8 1 2 3 4 all distinct (the
    # repeats are outside the window); t = 15: 1 2 3 4 9 9 9 9 -> 5 distinct
    assert got[7] == (1.0, 0) and got[11] == (1.0, 0)
    assert got[15][0] == 5 / 8 and got[15][1] == 0   # 9 (novel) 9 9 9 in the last four
    # t = 16: window 2 3 4 9 9 9 9 9 -> 4 distinct; the last four 9s all follow an earlier 9
    assert got[16][0] == 4 / 8 and got[16][1] == 1


def test_span_clipped_to_appended_rows():
    """after the cache changed otherwise than by one appended row, only the rows appended since
    then can be mapped to generated tokens"""
    H, P = 300, 8
    L_star = math.floor(256 + P - 51.2) + 1
    y = _healthy_then_loop(H, P, L_star)
    pm = np.where(np.arange(len(y)) >= H, 0.95, 0.5)
    prm, tp = oracle.params(), oracle.token_params()
    st, ts = oracle.new_state(0), oracle.new_token_state()
    n = 5000
    cut = len(y) - 50          # the cache is pruned (shrinks) before this token's step
    for t in range(len(y)):
        n = n + 1 if t != cut else 900
        f, span, dg = oracle.token_detect(y[:t + 1], pm[t], n, prm, tp, st, ts)
    assert f == 1 and span == (n - 50, n)


def test_cooldown_and_level():
    """a second trigger waits out the cooldown (32 steps); within retrig_window (64) of the
    first it raises the level"""
    H, P = 300, 8
    y = _healthy_then_loop(H, P, 400)
    pm = np.where(np.arange(len(y)) >= H, 0.95, 0.5)
    ev, st, _ = _run(y, pm, stop_at_trigger=False)
    assert len(ev) >= 2
    assert ev[1][0] - ev[0][0] == 33          # cd counts 32 steps down, the 33rd may fire
    assert st.level >= 1 and st.n_int == len(ev)


def test_no_trigger_on_healthy_stream():
    """a stream drawn from a large vocabulary never warns"""
    rng = np.random.default_rng(3)
    y = rng.integers(0, 50_000, size=700).astype(np.int32)
    pm = rng.uniform(0.1, 0.95, size=700)
    ev, _, _ = _run(y, pm, stop_at_trigger=False)
    assert ev == []


def test_span_follows_a_contiguous_kept_tail():
    """a prune that keeps the cache's last 400 rows in order (a budget cut keeps its recent rows
    so) leaves them consecutive generated tokens: given the kept list, the monitor keeps
    counting them, and the span later covers the whole loop (L* = 213 tokens) instead of the
    rows appended since the prune"""
    H, P = 300, 8
    L_star = math.floor(256 + P - 51.2) + 1
    y = _healthy_then_loop(H, P, L_star)
    pm = np.where(np.arange(len(y)) >= H, 0.95, 0.5)
    prm, tp = oracle.params(), oracle.token_params()
    st, ts = oracle.new_state(0), oracle.new_token_state()
    n = 5000
    cut = len(y) - 50
    for t in range(len(y)):
        kept = None
        if t == cut:
            kept = np.concatenate([np.arange(32), np.arange(n - 400, n)])
            n = len(kept)
        n += 1
        f, span, dg = oracle.token_detect(y[:t + 1], pm[t], n, prm, tp, st, ts, kept=kept)
    assert f == 1 and span == (n - L_star, n)
    assert ts.appended == 400 + 50


# --------------------------------------------------------------------------- threshold boundaries

def _last_diag(tokens, pmax, prm, tp):
    st, ts = oracle.new_state(0), oracle.new_token_state()
    dg = None
    for t in range(len(tokens)):
        _, _, dg = oracle.token_detect(tokens[:t + 1], pmax, 4000 + t + 1, prm, tp, st, ts)
    return dg


def test_token_votes_are_strict_at_their_thresholds():
    """W = 25, CR evaluated every token: the period-2 window 1 2 1 2 ... 1 of 25 tokens parses
    into 3 phrases, CR = 3/25 = theta_cr = 0.12, so the redundancy vote does not fire (strictly
    below); the window 1 2 3 4 5 1 1 ... 1 has 5 distinct of 25 tokens, TTR = 0.2 = theta_ttr,
    so the diversity vote does not fire either"""
    prm = oracle.params(W=25, t_min=10_000)
    tp = oracle.token_params(cr_every=1)
    dg = _last_diag((np.arange(25) % 2 + 1).astype(np.int32), 0.5, prm, tp)
    assert dg["cr"] == 3 / 25 and dg["sig2"] == 0
    assert dg["sig1"] == 1                                # TTR 2/25 < 0.2
    dg = _last_diag(np.array([1, 2, 3, 4, 5] + [1] * 20, dtype=np.int32), 0.5, prm, tp)
    assert dg["ttr"] == 5 / 25 and dg["sig1"] == 0


def test_streak_vote_fires_at_theta_streak():
    """the confidence vote fires once the streak reaches theta_streak = 6 steps (Eq. 8: >=)"""
    prm = oracle.params(t_min=10_000)
    tp = oracle.token_params()
    toks = (np.arange(200) + 7).astype(np.int32)
    pm = np.full(200, 0.95)
    st, ts = oracle.new_state(0), oracle.new_token_state()
    seen = []
    for t in range(8):
        _, _, dg = oracle.token_detect(toks[:t + 1], pm[t], 4000 + t + 1, prm, tp, st, ts)
        seen.append((int(dg["streak"]), int(dg["sig3"])))
    assert seen[4] == (5, 0) and seen[5] == (6, 1) and seen[6] == (7, 1)


def test_span_reaches_back_no_further_than_the_kept_history():
    """the span extends back over tokens the monitor still holds (the last hist tokens): with
    hist = 64 the loop's span is exactly those 64 tokens, with the default 512 it is the whole
    loop (its L* tokens, first period included)"""
    H, P = 300, 8
    L_star = math.floor(256 + P - 51.2) + 1
    y = _healthy_then_loop(H, P, L_star)
    pm = np.where(np.arange(len(y)) >= H, 0.95, 0.5)
    for hist, length in ((64, 64), (512, L_star)):
        ev, _, _ = _run(y, pm, prm=oracle.params(), tp=oracle.token_params(hist=hist))
        t, span, dg, n = ev[0]
        assert span[1] - span[0] == length, (hist, span)
