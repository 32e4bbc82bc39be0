"""Shared helpers of the GPU parity tests: run the oracle and the CUDA path side by side on the
same seeded inputs, step by step, and compare every output.

Tolerances (written here once, used by every parity test):
  attention output, bf16 cache: |gpu - ref| <= 1e-3 + 2e-2 |ref|   (bf16 output rounding)
  attention output, fp32 cache: |gpu - ref| <= 1e-5 + 1e-4 |ref|
  statistics m, l, H, S (fp32): |gpu - ref| <= 1e-6 + 1e-4 |ref|
  flags, spans, lengths, kept-index lists, compacted K/V/sketch bytes: bit-exact
"""
import numpy as np
import torch

import oracle
import synth
from paper_2604_10044_gb300 import lg

OUT_TOL = {"bf16": (2e-2, 1e-3), "f32": (1e-4, 1e-5)}
STAT_TOL = (1e-4, 1e-6)


def assert_close(got, ref, rtol, atol, what):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    bad = ~(np.abs(got - ref) <= atol + rtol * np.abs(ref))   # NaN on either side is bad
    if bad.any():
        i = np.argwhere(bad)[0]
        raise AssertionError("%s: %d/%d outside tolerance, first at %s: gpu %r ref %r" % (
            what, int(bad.sum()), bad.size, tuple(i), got[tuple(i)], ref[tuple(i)]))


def compare_cache(w, ref, cache, lens, what):
    """rows [0, len[b]) of every (layer, kv-head) and the sketches, byte for byte"""
    K, V = cache.to_host()
    sk = cache.sketch.cpu().numpy().view(np.uint32) if cache.sketch is not None else None
    for b in range(w.batch):
        o, n = int(w.seq_off[b]), int(lens[b])
        assert np.array_equal(K[:, :, o:o + n], ref.K[:, :, o:o + n]), "%s K seq %d" % (what, b)
        assert np.array_equal(V[:, :, o:o + n], ref.V[:, :, o:o + n]), "%s V seq %d" % (what, b)
        if sk is not None and ref.policy == "loopguard":
            assert np.array_equal(sk[o:o + n], ref.sk[o:o + n]), "%s sketch seq %d" % (what, b)


def run_loopguard(w, device, steps=None, n_layers_per_call=None, params=None, check_cache=True,
                  fused_prune=True):
    """The guarded decode path of workload w on the GPU and in the oracle, compared each step
    (fused_prune: lg_detect_prune, else lg_detect + lg_prune_compact).
    Returns counters of what the run exercised."""
    steps = w.steps if steps is None else steps
    K, V = synth.host_cache(w)
    prm_o = oracle.params(**(params or {}))
    prm_g = lg.lg_default_params(**(params or {}))
    ref = oracle.OracleGuard(w, K.copy(), V.copy(), prm_o)
    cache = lg.Cache.from_host(w, K, V, device, params=prm_g)
    guard = lg.Guard(cache, w.H_q, prm_g, n_layers_per_call=n_layers_per_call,
                     fused_prune=fused_prune)
    seqs = w.seqs.copy()
    pos = w.n0.astype(np.int64)
    rt, ra = OUT_TOL[w.dtype]
    counts = dict(triggers=0, prunes=0, steps=0)
    for t in range(steps):
        q, kn, vn = synth.host_step(w, pos, seqs)
        r_ref = ref.step(q, kn, vn, pos)
        r = guard.step_host(q, kn, vn, w.budget)
        tag = "step %d" % t
        assert_close(r["out"], r_ref["out"], rt, ra, tag + " out")
        assert_close(r["stats"], r_ref["stats"], *STAT_TOL, what=tag + " stats")
        for b in range(w.batch):
            dg, dr = r["diag"][b], r_ref["diags"][b]
            ctx = (tag, b, dg.tolist(), dr)
            assert np.isfinite(dg[:2]).all(), ctx
            assert abs(dg[0] - dr["ebar"]) <= 1e-4 * abs(dr["ebar"]) + 1e-6, ctx
            assert abs(dg[1] - dr["lbar"]) <= 1e-4 * abs(dr["lbar"]) + 1e-6, ctx
            assert dg[2] == dr["ttr"] and dg[6] == dr["stall"] and dg[7] == dr["P"], ctx
        assert np.array_equal(r["flags"], r_ref["flags"]), (tag, r["flags"], r_ref["flags"],
                                                           [d and (d["ebar"], d["lbar"])
                                                            for d in r_ref["diags"]])
        assert np.array_equal(r["spans"], r_ref["spans"]), (tag, r["spans"], r_ref["spans"])
        assert np.array_equal(r["len"], r_ref["len"]), (tag, r["len"], r_ref["len"])
        for b in range(w.batch):
            kept = r_ref["kept"][b]
            n_before = int(r_ref["len"][b]) if r["kept_count"][b] < 0 else None
            if r["kept_count"][b] < 0:
                assert np.array_equal(kept, np.arange(len(kept))), (tag, b)
                assert n_before == len(kept)
            else:
                assert r["kept_count"][b] == len(kept), (tag, b)
                assert np.array_equal(r["kept_idx"][b, :len(kept)], kept), (tag, b)
                counts["prunes"] += 1
        st = r["state"].reshape(w.batch, 8)
        for b in range(w.batch):
            s = ref.state[b]
            assert tuple(st[b, :5]) == (s.t_gen, s.cd, s.level, s.last_trig, s.n_int), (tag, b)
        if check_cache:
            compare_cache(w, ref, cache, r["len"], tag)
        counts["triggers"] += int(r["flags"].sum())
        counts["steps"] += 1
        synth.note_interventions(seqs, pos, r_ref["flags"])
        pos = pos + 1
    return counts


def run_h2o(w, device, steps=None, n_layers_per_call=None):
    """The H2O comparator path of workload w on the GPU and in the oracle, compared each step:
    outputs and statistics within tolerance, accumulated scores within 1e-4 relative, the
    selector of the oracle applied to the GPU's fp32 scores reproducing the GPU's choice
    exactly, and cache rows / positions bit-exact."""
    steps = w.steps if steps is None else steps
    K, V = synth.host_cache(w)
    ref = oracle.OracleGuard(w, K.copy(), V.copy(), policy="h2o")
    cache = lg.Cache.from_host(w, K, V, device, policy="h2o")
    guard = lg.Guard(cache, w.H_q, policy="h2o", n_layers_per_call=n_layers_per_call)
    pos = w.n0.astype(np.int64)
    rt, ra = OUT_TOL[w.dtype]
    dev = cache.device
    budget_d = torch.as_tensor(w.budget.astype(np.int32), device=dev)
    events = 0
    for t in range(steps):
        q, kn, vn = synth.host_step(w, pos)
        pos_d = torch.as_tensor(pos.astype(np.int32), device=dev)
        # GPU: begin, append, attend with accumulation; stop before the eviction
        c, p = cache, guard.p
        lg.lg_begin_step(c)
        lg.lg_append(c, 0, w.L, lg.host_to_device(kn, dev, w.dtype),
                     lg.host_to_device(vn, dev, w.dtype), pos_d, p)
        lg.lg_decode_attend(c, 0, w.L, lg.host_to_device(q, dev, w.dtype), w.H_q, guard.scale,
                            guard.out, guard.stats, p.suffix_w, 1, guard.max_len, guard.ws)
        torch.cuda.synchronize()
        scores_gpu = cache.h2o.cpu().numpy().copy()
        pos_gpu = cache.pos.cpu().numpy().copy()
        lens_gpu = cache.lengths().copy()
        # oracle: the same step
        ref.append(kn, vn, pos)
        out_ref, stats_ref = ref.attend(q)
        r = guard.results()
        tag = "h2o step %d" % t
        assert_close(r["out"], out_ref, rt, ra, tag + " out")
        assert_close(r["stats"], stats_ref, *STAT_TOL, what=tag + " stats")
        for b in range(w.batch):
            o, n = int(w.seq_off[b]), int(lens_gpu[b])
            assert_close(scores_gpu[:, :, o:o + n], ref.h2o[:, :, o:o + n], 1e-4, 1e-6,
                         tag + " scores seq %d" % b)
        # the GPU's eviction, and the oracle's selector on the GPU's own scores
        lg.lg_h2o_evict(c, budget_d, pos_d, guard.max_len)
        torch.cuda.synchronize()
        assert lg.lg_read_device_status(c) == 0
        Kg, Vg = cache.to_host()
        sc_after = cache.h2o.cpu().numpy()
        ps_after = cache.pos.cpu().numpy()
        for b in range(w.batch):
            o, n, B = int(w.seq_off[b]), int(lens_gpu[b]), int(w.budget[b])
            if n <= B:
                continue
            events += 1
            for layer in range(w.L):
                for kvh in range(w.H_kv):
                    sc = scores_gpu[layer, kvh, o:o + n].astype(np.float64)
                    ps = pos_gpu[layer, kvh, o:o + n]
                    if n == B + 1:
                        x = oracle.h2o_argmin(sc, ps, B, int(pos[b]))
                        slots = list(range(n))
                        slots[x] = n - 1
                        expect = np.array(slots[:B])
                    else:
                        expect = oracle.h2o_select(sc, ps, B, int(pos[b]))
                    assert np.array_equal(ps_after[layer, kvh, o:o + B], ps[expect]), \
                        (tag, b, layer, kvh)
        # oracle eviction on its own scores; rows and positions must agree bit for bit
        ref.h2o_evict(pos)
        for b in range(w.batch):
            o, n = int(w.seq_off[b]), int(ref.len[b])
            assert np.array_equal(ps_after[:, :, o:o + n], ref.pos[:, :, o:o + n]), (tag, b)
            assert np.array_equal(Kg[:, :, o:o + n], ref.K[:, :, o:o + n]), (tag, b)
            assert np.array_equal(Vg[:, :, o:o + n], ref.V[:, :, o:o + n]), (tag, b)
        assert np.array_equal(cache.lengths(), ref.len)
        pos = pos + 1
    return events


def run_streaming(w, device, steps=None):
    """The StreamingLLM comparator (sinks + sliding window) on the GPU and in the oracle:
    outputs and statistics within tolerance, rows and positions bit-exact every step."""
    steps = w.steps if steps is None else steps
    K, V = synth.host_cache(w)
    ref = oracle.OracleGuard(w, K.copy(), V.copy(), policy="streaming")
    cache = lg.Cache.from_host(w, K, V, device, policy="streaming")
    guard = lg.Guard(cache, w.H_q, policy="streaming")
    pos = w.n0.astype(np.int64)
    rt, ra = OUT_TOL[w.dtype]
    for t in range(steps):
        q, kn, vn = synth.host_step(w, pos)
        r_ref = ref.step(q, kn, vn, pos)
        r = guard.step_host(q, kn, vn, w.budget, pos.astype(np.int32))
        tag = "streaming step %d" % t
        assert_close(r["out"], r_ref["out"], rt, ra, tag + " out")
        assert_close(r["stats"], r_ref["stats"], *STAT_TOL, what=tag + " stats")
        assert np.array_equal(r["len"], r_ref["len"]), tag
        Kg, Vg = cache.to_host()
        ps = cache.pos.cpu().numpy()
        for b in range(w.batch):
            o, n = int(w.seq_off[b]), int(r_ref["len"][b])
            assert np.array_equal(ps[:, :, o:o + n], ref.pos[:, :, o:o + n]), (tag, b)
            assert np.array_equal(Kg[:, :, o:o + n], ref.K[:, :, o:o + n]), (tag, b)
            assert np.array_equal(Vg[:, :, o:o + n], ref.V[:, :, o:o + n]), (tag, b)
        pos = pos + 1
