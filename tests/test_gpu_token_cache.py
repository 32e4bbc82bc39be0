"""The token-level path on a real cache: lg_token_detect_prune (the token-level monitor, Sec. 5.2,
Eq. 8, Eq. 9, App. B.2, with the retained set of Sec. 5.3, Eq. 10, Eq. 11 formed in its kernel)
after append and the attention pass, on a bf16 cache of the paper's shape (2 of its 28 layers,
16/8 heads, d = 128, the 3853-row prompt, B = 1024), step by step against the oracle: the first
budget cut, the periodic ones, and a trigger on the planted loop's generated tokens, after which
the sequence's tokens and rows turn loop-free.  Flags, spans, guard state, kept lists and
lengths are compared exactly every step, attention outputs and statistics within the parity
tolerances, and every compacted K/V row and sketch byte after each prune."""
import numpy as np
import pytest
import torch

import oracle
import synth
from paper_2604_10044_gb300 import lg
from parity_util import OUT_TOL, STAT_TOL, assert_close, compare_cache

pytestmark = pytest.mark.gpu

STEPS = 300


def test_token_path_on_the_paper_shaped_cache(cuda):
    w = synth.make_workload(6, L=2, onset=(30, 40), steps=STEPS)
    K, V = synth.host_cache(w)
    tl, tf, pl, pf = synth.token_streams(w, STEPS)
    prm_o, prm_g = oracle.params(), lg.lg_default_params()
    tp_o, tp_g = oracle.token_params(), lg.lg_default_token_params()
    # the token monitor counts generated tokens from 0
    ref = oracle.OracleGuard(w, K.copy(), V.copy(), prm_o, t_gen0=0)
    ts_o = [oracle.new_token_state() for _ in range(w.batch)]
    cache = lg.Cache.from_host(w, K, V, cuda, params=prm_g)
    g = lg.Guard(cache, w.H_q, prm_g)
    lg.lg_state_init(cache, g.state, 0)
    tstate = torch.zeros(lg.lg_token_state_size(cache, prm_g, tp_g) // 4, dtype=torch.int32,
                         device=cuda)
    budget = torch.as_tensor(w.budget.astype(np.int32), device=cuda)
    g.kept_count.fill_(-1)
    seqs, pos = w.seqs.copy(), w.n0.astype(np.int64)
    hist = np.zeros((STEPS, w.batch), dtype=np.int32)
    prev_kept = [None] * w.batch
    rt, ra = OUT_TOL[w.dtype]
    triggers = prunes = 0
    for t in range(STEPS):
        tag = "step %d" % t
        # each sequence's generated token: loop-continuing until the guard has intervened
        fresh = np.array([ref.state[b].n_int > 0 for b in range(w.batch)])
        hist[t] = np.where(fresh, tf[t], tl[t])
        pm = np.where(fresh, pf[t], pl[t]).astype(np.float32)
        q, kn, vn = synth.host_step(w, pos, seqs)
        # oracle: append, attention, token-level monitor, retained set and compaction
        ref.append(kn, vn)
        out_o, stats_o = ref.attend(q)
        flags_o = np.zeros(w.batch, dtype=np.int32)
        spans_o = np.zeros((w.batch, 2), dtype=np.int32)
        for b in range(w.batch):
            f, sp, _ = oracle.token_detect(hist[:t + 1, b], float(pm[b]), int(ref.len[b]),
                                           prm_o, tp_o, ref.state[b], ts_o[b],
                                           kept=prev_kept[b])
            flags_o[b], spans_o[b] = f, sp
        n_before = ref.len.copy()
        kept_o = ref.prune(flags_o, spans_o)
        # GPU: the same step through the C ABI
        qd, kd, vd = (lg.host_to_device(x, cuda, w.dtype) for x in (q, kn, vn))
        lg.lg_begin_step(cache)
        lg.lg_append(cache, 0, w.L, kd, vd, None, prm_g)
        lg.lg_decode_attend(cache, 0, w.L, qd, w.H_q, g.scale, g.out, g.stats, prm_g.suffix_w, 0,
                            g.max_len, g.ws)
        lg.lg_token_detect_prune(cache, torch.as_tensor(hist[t], device=cuda),
                                 torch.as_tensor(pm, device=cuda), g.state, budget, prm_g, tp_g,
                                 g.flags, g.spans, None, tstate, g.kept_idx, g.kept_count,
                                 g.max_keep, g.max_len)
        torch.cuda.synchronize()
        assert lg.lg_read_device_status(cache) == 0, tag
        out_g = g.out.float().cpu().numpy()   # bf16 outputs, exactly widened
        assert_close(out_g, out_o, rt, ra, tag + " out")
        assert_close(g.stats.cpu().numpy(), stats_o, *STAT_TOL, what=tag + " stats")
        assert np.array_equal(g.flags.cpu().numpy(), flags_o), tag
        assert np.array_equal(g.spans.cpu().numpy(), spans_o), tag
        st = g.state.cpu().numpy().reshape(w.batch, 8)
        kc, ki = g.kept_count.cpu().numpy(), g.kept_idx.cpu().numpy()
        for b in range(w.batch):
            s = ref.state[b]
            assert tuple(st[b, :5]) == (s.t_gen, s.cd, s.level, s.last_trig, s.n_int), (tag, b)
            pruned = bool(flags_o[b]) or n_before[b] > w.budget[b]
            prev_kept[b] = kept_o[b] if pruned else None
            if pruned:
                assert kc[b] == len(kept_o[b]) and np.array_equal(ki[b, :kc[b]], kept_o[b]), \
                    (tag, b)
                prunes += 1
            else:
                assert kc[b] == -1, (tag, b)
        assert np.array_equal(cache.lengths(), ref.len), tag
        if flags_o.any() or (n_before > w.budget).any() or t == STEPS - 1:
            compare_cache(w, ref, cache, ref.len, tag)
        triggers += int(flags_o.sum())
        synth.note_interventions(seqs, pos, flags_o)
        pos = pos + 1
    assert triggers >= 1 and prunes >= 3, (triggers, prunes)
