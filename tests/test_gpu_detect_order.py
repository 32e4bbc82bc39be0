"""The loop-onset test (Sec. 5.2, Eq. 8, Eq. 9) called in orders where the kernel before it
writes what its early phase reads.

detect_kernel compares the new row with the window before its dependency wait, then reads the
length, the synced length and the new row again and recomputes the window when any of them
changed.  In the usual step the kernel before it is the attention pass, which writes none of
them; these tests put other kernels there:
  - lg_detect_prune straight after lg_append (the statistics supplied by the caller before the
    step, so that no attention pass runs in between): the early phase races the append of the
    very row it compares;
  - lg_detect twice on the same step: the second call's early phase races the first call's
    update of the synced length and the monitor state.
Every decision, span, kept list, guard state and compacted byte must equal the oracle's.
"""
import numpy as np
import pytest
import torch

import oracle
import synth
from paper_2604_10044_gb300 import lg
from parity_util import compare_cache

pytestmark = pytest.mark.gpu


def _workload():
    return synth.make_workload(2, L=2, batch=4, n=1200, budget=768, steps=40, tail=(300, 500),
                               periods=(8, 40))


def _check_detect(r_gpu, flags_o, spans_o, diags_o, state_o, tag):
    assert np.array_equal(r_gpu["flags"], flags_o), (tag, r_gpu["flags"], flags_o)
    assert np.array_equal(r_gpu["spans"], spans_o), (tag, r_gpu["spans"], spans_o)
    st = r_gpu["state"].reshape(-1, 8)
    for b, s in enumerate(state_o):
        assert tuple(st[b, :5]) == (s.t_gen, s.cd, s.level, s.last_trig, s.n_int), (tag, b)
    for b, d in enumerate(diags_o):
        dg = r_gpu["diag"][b]
        assert dg[2] == d["ttr"] and dg[6] == d["stall"] and dg[7] == d["P"], (tag, b)


def test_detect_prune_straight_after_append(cuda):
    """caller-supplied statistics (the oracle's attention, rounded to fp32 for both sides), then
    begin, append and lg_detect_prune with no attention pass between append and detect"""
    w = _workload()
    K, V = synth.host_cache(w)
    prm_o, prm_g = oracle.params(), lg.lg_default_params()
    ref = oracle.OracleGuard(w, K.copy(), V.copy(), prm_o)
    cache = lg.Cache.from_host(w, K, V, cuda, params=prm_g)
    guard = lg.Guard(cache, w.H_q, prm_g)
    budget = torch.as_tensor(w.budget.astype(np.int32), device=cuda)
    seqs, pos = w.seqs.copy(), w.n0.astype(np.int64)
    triggers = prunes = 0
    for t in range(w.steps):
        q, kn, vn = synth.host_step(w, pos, seqs)
        ref.append(kn, vn, pos)
        _, stats = ref.attend(q)
        stats32 = stats.astype(np.float32)
        guard.stats.copy_(torch.from_numpy(stats32))
        kd, vd = (lg.host_to_device(x, cuda, w.dtype) for x in (kn, vn))
        lg.lg_begin_step(cache)
        lg.lg_append(cache, 0, w.L, kd, vd, None, prm_g)
        lg.lg_detect_prune(cache, guard.stats, w.H_q, guard.state, budget, prm_g, guard.flags,
                           guard.spans, guard.diag, guard.dstate, guard.kept_idx,
                           guard.kept_count, guard.max_keep, guard.max_len)
        torch.cuda.synchronize()
        assert lg.lg_read_device_status(cache) == 0
        flags, spans, diags = ref.detect_all(stats32.astype(np.float64))
        kept = ref.prune(flags, spans)
        r = dict(flags=guard.flags.cpu().numpy(), spans=guard.spans.cpu().numpy(),
                 state=guard.state.cpu().numpy(), diag=guard.diag.cpu().numpy())
        tag = "step %d" % t
        _check_detect(r, flags, spans, diags, ref.state, tag)
        kc = guard.kept_count.cpu().numpy()
        ki = guard.kept_idx.cpu().numpy()
        for b in range(w.batch):
            if kc[b] >= 0:
                prunes += 1
                assert np.array_equal(ki[b, :kc[b]], kept[b]), (tag, b)
        assert np.array_equal(cache.lengths(), ref.len), tag
        compare_cache(w, ref, cache, ref.len, tag)
        triggers += int(flags.sum())
        synth.note_interventions(seqs, pos, flags)
        pos = pos + 1
    assert triggers >= 1 and prunes >= w.batch, (triggers, prunes)


def test_detect_twice_on_one_step(cuda):
    """a step whose lg_detect is called twice on the same statistics: the second call's early
    phase reads the synced length and the monitor state the first call is writing; both calls
    must match the oracle's detect called twice"""
    w = _workload()
    K, V = synth.host_cache(w)
    prm_o, prm_g = oracle.params(), lg.lg_default_params()
    ref = oracle.OracleGuard(w, K.copy(), V.copy(), prm_o)
    cache = lg.Cache.from_host(w, K, V, cuda, params=prm_g)
    guard = lg.Guard(cache, w.H_q, prm_g, fused_prune=False)
    budget = torch.as_tensor(w.budget.astype(np.int32), device=cuda)
    seqs, pos = w.seqs.copy(), w.n0.astype(np.int64)
    for t in range(12):
        q, kn, vn = synth.host_step(w, pos, seqs)
        qd, kd, vd = (lg.host_to_device(x, cuda, w.dtype) for x in (q, kn, vn))
        lg.lg_begin_step(cache)
        lg.lg_append(cache, 0, w.L, kd, vd, None, prm_g)
        lg.lg_decode_attend(cache, 0, w.L, qd, w.H_q, guard.scale, guard.out, guard.stats,
                            prm_g.suffix_w, 0, guard.max_len, guard.ws)
        ref.append(kn, vn, pos)
        _, _ = ref.attend(q)
        stats_g = None
        for k in range(2):
            lg.lg_detect(cache, guard.stats, w.H_q, guard.state, budget, prm_g, guard.flags,
                         guard.spans, guard.diag, guard.dstate)
            torch.cuda.synchronize()
            assert lg.lg_read_device_status(cache) == 0
            if stats_g is None:
                stats_g = guard.stats.cpu().numpy().astype(np.float64)
            flags, spans, diags = ref.detect_all(stats_g)
            r = dict(flags=guard.flags.cpu().numpy(), spans=guard.spans.cpu().numpy(),
                     state=guard.state.cpu().numpy(), diag=guard.diag.cpu().numpy())
            _check_detect(r, flags, spans, diags, ref.state, "step %d call %d" % (t, k))
        # the prune of the second call's decision on both sides, then the next step
        lg.lg_prune_compact(cache, guard.flags, guard.spans, guard.state, budget, prm_g,
                            guard.kept_idx, guard.kept_count, guard.max_keep, guard.max_len)
        kept = ref.prune(flags, spans)
        torch.cuda.synchronize()
        assert np.array_equal(cache.lengths(), ref.len), t
        compare_cache(w, ref, cache, ref.len, "step %d" % t)
        synth.note_interventions(seqs, pos, flags)
        pos = pos + 1
