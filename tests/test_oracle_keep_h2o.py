"""Pins of the oracle's retained set I_keep (Sec. 5.3, Eq. 10, Eq. 11), its index-gather, and
the H2O comparator (Sec. 2.2, Sec. 6.1).

I_keep is a union of a prefix, an integer lattice and a contiguous range with a hole, so its
size and members have closed forms; the invariants (|I_keep| <= B, anchors kept, I_bad
dropped, ascending) are checked on every case.  H2O selection and the single eviction are
checked against brute force on tiny inputs.
"""
import numpy as np
import pytest

import oracle


def _sizes(B, level, headroom=64, n_anchor=32):
    hd = min(headroom, B // 4)
    T = B - hd
    return T, B // 2, (B // 4) >> level, T - n_anchor - B // 4


@pytest.mark.parametrize("n,B,flag,span,level", [
    (8193, 4096, 0, (0, 0), 0),       # first step of the 8192-row workload: budget event
    (8193, 4096, 1, (7000, 8193), 0),
    (4097, 4096, 0, (0, 0), 0),       # one row over budget: every history row fits the lattice
    (3000, 4096, 1, (2500, 3000), 2),
    (513, 256, 1, (385, 513), 0),
    (513, 256, 1, (450, 500), 1),
    (40, 256, 1, (10, 40), 0),
    (300, 256, 1, (0, 0), 3),         # trigger without a detected tail
])
def test_keep_set_closed_form(n, B, flag, span, level):
    prm = oracle.params()
    kept = oracle.keep_set(n, B, flag, span, level, prm)
    T, R, B_rec, B_sp = _sizes(B, level if flag else 0)
    lo_bad, hi_bad = span if flag else (0, 0)
    A = min(32, n)
    rw_lo = min(max(32, n - R), n)
    n_c = max(0, rw_lo - 32)
    n_recent_cand = (n - rw_lo) - max(0, min(hi_bad, n) - max(lo_bad, rw_lo))
    expect_size = A + min(n_c, B_sp) + min(B_rec, n_recent_cand)
    assert len(kept) == expect_size
    assert len(kept) <= T <= B
    assert np.all(np.diff(kept) > 0)
    assert set(range(A)) <= set(kept.tolist())
    # I_bad is a subset of W^recent (Sec. 5.3); anchors stay even if a span reaches them
    assert not (set(kept.tolist()) & set(range(max(lo_bad, rw_lo), hi_bad)))
    # sparse part: a uniform lattice over [32, rw_lo) starting at 32, gaps differ by <= 1
    sparse = kept[(kept >= 32) & (kept < rw_lo)]
    if n_c:
        assert sparse[0] == 32
        if n_c > B_sp:
            gaps = np.diff(sparse)
            assert gaps.max() - gaps.min() <= 1
            assert np.array_equal(sparse, 32 + (np.arange(B_sp, dtype=np.int64) * n_c) // B_sp)
        else:
            assert np.array_equal(sparse, np.arange(32, rw_lo))
    # recent part: the last B_recent rows of W^recent outside I_bad
    recent = kept[kept >= rw_lo]
    cand = [i for i in range(rw_lo, n) if not lo_bad <= i < hi_bad]
    assert recent.tolist() == cand[len(cand) - min(B_rec, len(cand)):]


def test_keep_set_numbers_of_the_8192_row_workload():
    prm = oracle.params()
    # n = 8193 > B = 4096: 32 anchors + 2976 lattice rows + the last 1024 rows = 4032 = B - 64
    assert len(oracle.keep_set(8193, 4096, 0, (0, 0), 0, prm)) == 4032
    # n = 4097: history [32, 2049) fits the lattice budget: 32 + 2017 + 1024 = 3073
    assert len(oracle.keep_set(4097, 4096, 0, (0, 0), 0, prm)) == 3073
    # not over budget and not flagged: untouched
    assert np.array_equal(oracle.keep_set(4000, 4096, 0, (0, 0), 0, prm), np.arange(4000))
    with pytest.raises(ValueError):
        oracle.keep_set(300, 60, 1, (0, 0), 0, prm)     # budget too small for the anchors


def test_compact_rows_is_an_ordered_gather():
    rng = np.random.default_rng(0)
    rows = rng.integers(0, 2 ** 16, size=(500, 64), dtype=np.uint16)
    before = rows.copy()
    kept = np.sort(rng.choice(500, size=137, replace=False)).astype(np.int32)
    oracle.compact_rows(rows, kept)
    assert np.array_equal(rows[:137], before[kept])
    assert np.array_equal(rows[137:], before[137:])


def _h2o_brute(score, pos, B, pos_now):
    n = len(score)
    R = B // 2
    recent = [i for i in range(n) if pos[i] > pos_now - R]
    rest = [i for i in range(n) if pos[i] <= pos_now - R]
    rest.sort(key=lambda i: (-score[i], -pos[i]))       # heaviest first, newer first on ties
    keep = set(recent) | set(rest[:max(0, B - len(recent))])
    return sorted(keep)


@pytest.mark.parametrize("seed", range(10))
def test_h2o_select_brute_force(seed):
    rng = np.random.default_rng(seed)
    n = int(rng.integers(10, 60))
    B = int(rng.integers(4, n))
    pos = rng.permutation(n).astype(np.int32) + 5
    pos_now = int(pos.max())
    score = rng.integers(0, 6, size=n).astype(np.float64) / 4   # many exact ties
    kept = oracle.h2o_select(score, pos, B, pos_now)
    assert kept.tolist() == _h2o_brute(score, pos, B, pos_now)
    assert len(kept) == B
    # argmin: the first row the brute-force order would drop
    x = oracle.h2o_argmin(score, pos, n - 1, pos_now)
    R = (n - 1) // 2
    cand = [i for i in range(n) if pos[i] <= pos_now - R]
    assert x == min(cand, key=lambda i: (score[i], pos[i]))
    assert sorted(set(range(n)) - {x}) == oracle.h2o_select(score, pos, n - 1, pos_now).tolist()


def test_h2o_path_keeps_budget_and_mass():
    """whole-step H2O comparator on a tiny workload: length <= B after every step, distinct
    positions in every (layer, kv-head) stream, the B/2 most recent positions all present (the
    scores' bookkeeping: tests/test_oracle_guard_steps.py)"""
    import synth
    w = synth.make_workload(2, L=2, batch=3, n=200, budget=128, steps=6, H_q=4, H_kv=2,
                            tail=(60, 80), periods=(5, 9))
    K, V = synth.host_cache(w)
    g = oracle.OracleGuard(w, K, V, policy="h2o")
    seqs = w.seqs.copy()
    pos = w.n0.astype(np.int64)
    for step in range(w.steps):
        q, kn, vn = synth.host_step(w, pos, seqs)
        before = g.len.copy()
        r = g.step(q, kn, vn, pos)
        assert np.all(r["len"] <= w.budget)
        assert np.all(r["len"] == np.minimum(before + 1, w.budget))
        for b in range(w.batch):
            o, n = w.seq_off[b], r["len"][b]
            # recent window fully present
            for layer in range(w.L):
                for kvh in range(w.H_kv):
                    ps = g.pos[layer, kvh, o:o + n]
                    assert len(set(ps.tolist())) == n
                    assert set(range(int(pos[b]) - w.budget[b] // 2 + 1, int(pos[b]) + 1)) <= \
                        set(ps.tolist())
        pos = pos + 1


@pytest.mark.parametrize("seed", range(6))
def test_streaming_select_brute_force(seed):
    """StreamingLLM: the first n_sink positions and the budget - n_sink newest stay"""
    rng = np.random.default_rng(seed)
    n = int(rng.integers(12, 60))
    B = int(rng.integers(6, n))
    pos = rng.permutation(n).astype(np.int32)
    pos_now = int(pos.max())
    kept = oracle.streaming_select(pos, B, 4, pos_now)
    order = sorted(range(n), key=lambda i: -pos[i])
    expect = sorted({i for i in range(n) if pos[i] < 4} | set(
        [i for i in order if pos[i] >= 4][:B - 4]))
    assert kept.tolist() == expect and len(kept) == B
    x = oracle.streaming_oldest(pos, 4)
    assert pos[x] == 4                       # positions 0..n-1 are all present


def test_budget_event_prunes_at_level_zero():
    """a budget event (no trigger) keeps B/4 recent rows whatever level the guard is at; only a
    trigger prunes at the progressive level (Sec. 5.3)"""
    prm = oracle.params()
    base = oracle.keep_set(8193, 4096, 0, (0, 0), 0, prm)
    for level in (1, 2, 3):
        assert np.array_equal(oracle.keep_set(8193, 4096, 0, (0, 0), level, prm), base)
    assert len(oracle.keep_set(8193, 4096, 1, (0, 0), 2, prm)) < len(base)


def test_h2o_scores_add_every_head_of_the_group():
    """four query heads of one kv-head, each attending almost only to its own key row: the
    accumulated score of each of those rows is about 1, every other row about 0 (the score sums
    the attention the row receives from every head of its group)"""
    import synth
    w = synth.make_workload(2, L=1, batch=1, n=64, budget=64, steps=1, H_q=4, H_kv=1,
                            tail=(20, 24), periods=(8, 8))
    n = int(w.n0[0])
    rng = np.random.default_rng(17)
    Kf = (rng.standard_normal((w.L, w.H_kv, w.S_total, w.d)) * 0.01).astype(np.float32)
    qf = np.zeros((w.L, w.batch, w.H_q, w.d), dtype=np.float32)
    rows = [3, 13, 23, 33]
    for h, r in enumerate(rows):
        Kf[0, 0, r, 32 * h:32 * (h + 1)] = 1.0
        qf[0, 0, h, 32 * h:32 * (h + 1)] = 4.0
    Vf = rng.standard_normal((w.L, w.H_kv, w.S_total, w.d)).astype(np.float32)
    from test_oracle_attention import bf16_bits
    g = oracle.OracleGuard(w, bf16_bits(Kf), bf16_bits(Vf), policy="h2o")
    g.attend(bf16_bits(qf))
    sc = g.h2o[0, 0, :n]
    for r in rows:
        assert 0.99 < sc[r] < 1.0, r
    others = np.delete(sc, rows)
    assert others.max() < 0.01
    assert sc.sum() == pytest.approx(w.g, rel=1e-12)


def test_a_cache_exactly_at_its_budget_is_not_pruned():
    """Sec. 5.3 prunes on a trigger or when the cache outgrows B: n == B keeps every row"""
    prm = oracle.params()
    assert np.array_equal(oracle.keep_set(4096, 4096, 0, (0, 0), 0, prm), np.arange(4096))
    assert len(oracle.keep_set(4097, 4096, 0, (0, 0), 0, prm)) < 4096
