"""Pins of the oracle's step bookkeeping (OracleGuard): what each decode step carries along with
the cache rows.  Sketches follow their rows through appends and prunes (Sec. 5.3's index-gather
moves every per-row quantity); a trigger prunes at the guard's current level; on the H2O and
StreamingLLM paths every row keeps its own position and accumulated score through swap-removes
and cuts; a new row starts with no score; the attention scale is 1/sqrt(d) (Eq. 1); each
sequence's test uses its own budget.  Each check follows from the definitions, not from a
previous run."""
import math

import numpy as np

import oracle
import synth


def _small(policy_steps=8, budget=128):
    return synth.make_workload(2, L=2, batch=3, n=200, budget=budget, steps=policy_steps, H_q=4,
                               H_kv=2, tail=(60, 80), periods=(5, 9))


def _check_sketches(g, w):
    gl = g.prm.guard_layer
    for b in range(w.batch):
        o = int(w.seq_off[b])
        for j in range(int(g.len[b])):
            want = oracle.sketch(np.ascontiguousarray(g.V[gl, :, o + j, :]))
            assert np.array_equal(g.sk[o + j], want), (b, j)


def test_sketches_follow_their_rows_through_appends_and_prunes():
    w = _small()
    K, V = synth.host_cache(w)
    g = oracle.OracleGuard(w, K, V)
    _check_sketches(g, w)
    seqs, pos = w.seqs.copy(), w.n0.astype(np.int64)
    pruned = 0
    for _ in range(w.steps):
        q, kn, vn = synth.host_step(w, pos, seqs)
        before = g.len.copy()
        r = g.step(q, kn, vn, pos)
        pruned += int((r["len"] < before + 1).sum())
        _check_sketches(g, w)
        synth.note_interventions(seqs, pos, r["flags"])
        pos = pos + 1
    assert pruned > 0          # the first step cuts every sequence to its budget


def test_prune_reads_the_guards_level():
    """n = 600, B = 512, a trigger with span [550, 600): W^recent = [344, 600), the lattice
    keeps 288 of the 312 rows between the anchors and W^recent, and level 2 keeps
    (512 / 4) >> 2 = 32 recent rows outside the span: 32 + 288 + 32 = 352 rows"""
    w = synth.make_workload(2, L=1, batch=1, n=600, budget=512, steps=1, H_q=2, H_kv=1,
                            tail=(100, 100), periods=(8, 8))
    K, V = synth.host_cache(w)
    g = oracle.OracleGuard(w, K, V)
    g.state[0].level = 2
    kept = g.prune(np.array([1]), np.array([[550, 600]]), np.array([512]))
    assert len(kept[0]) == 352 and g.len[0] == 352
    assert np.array_equal(kept[0][-32:], np.arange(518, 550))


def _pairs(g, w, b, layer, kvh, n):
    o = int(w.seq_off[b])
    return sorted(zip(g.pos[layer, kvh, o:o + n].tolist(), g.h2o[layer, kvh, o:o + n].tolist()))


def test_h2o_rows_keep_their_position_and_score():
    """after each eviction the (position, score) pairs of a stream are the pairs it had before,
    less the evicted ones, and every K row is the row that carried that position"""
    w = _small()
    K, V = synth.host_cache(w)
    g = oracle.OracleGuard(w, K, V, policy="h2o")
    seqs, pos = w.seqs.copy(), w.n0.astype(np.int64)
    for _ in range(4):
        q, kn, vn = synth.host_step(w, pos, seqs)
        g.append(kn, vn, pos)
        g.attend(q)
        snap = {}
        rows = {}
        for b in range(w.batch):
            o, n = int(w.seq_off[b]), int(g.len[b])
            for layer in range(w.L):
                for kvh in range(w.H_kv):
                    snap[(b, layer, kvh)] = _pairs(g, w, b, layer, kvh, n)
                    rows[(b, layer, kvh)] = {int(p): g.K[layer, kvh, o + i].copy()
                                             for i, p in enumerate(g.pos[layer, kvh, o:o + n])}
        g.h2o_evict(pos)
        for (b, layer, kvh), before in snap.items():
            o, n = int(w.seq_off[b]), int(g.len[b])
            after = _pairs(g, w, b, layer, kvh, n)
            left = list(before)
            for pr in after:
                assert pr in left, (b, layer, kvh, pr)
                left.remove(pr)
            assert len(left) == len(before) - n
            for i in range(n):
                p = int(g.pos[layer, kvh, o + i])
                assert np.array_equal(g.K[layer, kvh, o + i], rows[(b, layer, kvh)][p])
        pos = pos + 1


def test_new_rows_start_without_score():
    """from fresh scores, one step adds exactly g per (layer, kv-head, sequence): the g heads'
    attention over the appended cache, the new row included, each summing to 1"""
    w = _small(budget=1000)
    K, V = synth.host_cache(w)
    g = oracle.OracleGuard(w, K, V, policy="h2o")
    pos = w.n0.astype(np.int64)
    q, kn, vn = synth.host_step(w, pos, w.seqs.copy())
    g.step(q, kn, vn, pos)
    for b in range(w.batch):
        o, n = int(w.seq_off[b]), int(g.len[b])
        for layer in range(w.L):
            for kvh in range(w.H_kv):
                assert abs(g.h2o[layer, kvh, o:o + n].sum() - w.g) < 1e-12


def test_streaming_rows_keep_their_position():
    w = _small()
    K, V = synth.host_cache(w)
    g = oracle.OracleGuard(w, K, V, policy="streaming")
    seqs, pos = w.seqs.copy(), w.n0.astype(np.int64)
    for _ in range(4):
        q, kn, vn = synth.host_step(w, pos, seqs)
        g.append(kn, vn, pos)
        rows = {}
        for b in range(w.batch):
            o, n = int(w.seq_off[b]), int(g.len[b])
            for layer in range(w.L):
                for kvh in range(w.H_kv):
                    rows[(b, layer, kvh)] = {int(p): g.K[layer, kvh, o + i].copy()
                                             for i, p in enumerate(g.pos[layer, kvh, o:o + n])}
        g.streaming_evict(pos)
        for (b, layer, kvh), by_pos in rows.items():
            o, n = int(w.seq_off[b]), int(g.len[b])
            ps = g.pos[layer, kvh, o:o + n].tolist()
            assert len(set(ps)) == n
            for i, p in enumerate(ps):
                assert np.array_equal(g.K[layer, kvh, o + i], by_pos[p])
        pos = pos + 1


def test_attention_scale_is_one_over_sqrt_d():
    w = _small(budget=1000)
    K, V = synth.host_cache(w)
    g = oracle.OracleGuard(w, K, V)
    q, _, _ = synth.host_step(w, w.n0.astype(np.int64), w.seqs.copy())
    out, stats = g.attend(q)
    b, layer, kvh = 1, 1, 1
    o, n = int(w.seq_off[b]), int(g.len[b])
    heads = slice(kvh * w.g, (kvh + 1) * w.g)
    out1, st1, _ = oracle.attend_group(np.ascontiguousarray(q[layer, b, heads]),
                                       np.ascontiguousarray(K[layer, kvh, o:o + n]),
                                       np.ascontiguousarray(V[layer, kvh, o:o + n]),
                                       scale=1.0 / math.sqrt(w.d))
    assert np.array_equal(out[layer, b, heads], out1)
    assert np.array_equal(stats[layer, b, heads], st1)


def test_each_sequence_is_tested_against_its_own_budget():
    """two sequences with the same looping sketches: the span of the one with B = 256 is
    clipped to its recent window [n - 128, n); the one with B = 1024 reaches further back"""
    w = synth.make_workload(2, L=1, batch=2, n=300, budget=256, steps=1, H_q=2, H_kv=1,
                            tail=(200, 200), periods=(8, 8))
    K, V = synth.host_cache(w)
    g = oracle.OracleGuard(w, K, V, t_gen0=100)
    loop_b = int(np.argmax(w.seqs["looping"]))
    other = 1 - loop_b
    n = int(g.len[loop_b])
    g.sk[w.seq_off[other]:w.seq_off[other] + n] = g.sk[w.seq_off[loop_b]:w.seq_off[loop_b] + n]
    g.len[other] = n
    stats = np.zeros((1, 2, 2, 4))
    stats[..., 2] = 0.3 * math.log(n)          # concentration vote
    stats[..., 3] = 3.0 * 64 / n               # locking vote
    budgets = np.zeros(2, dtype=np.int64)
    budgets[loop_b], budgets[other] = 1024, 256
    flags, spans, _ = g.detect_all(stats, budgets)
    assert flags.tolist() == [1, 1]
    assert spans[other].tolist() == [n - 128, n]
    assert spans[loop_b][0] < n - 128
