"""Two independent guarded batches, each with its own cache, workspace, guard state and monitor
state, stepped concurrently on two CUDA streams with their launches interleaved: each must
match its own oracle at every step (attention outputs and statistics within the parity
tolerances; flags, spans, lengths, kept lists and compacted rows exactly).  The library keeps no
state between calls outside the caller's buffers (the pass direction and the chunk counters
live in each call's workspace), so neither batch may see the other."""
import numpy as np
import pytest
import torch

import oracle
import synth
from paper_2604_10044_gb300 import lg
from parity_util import OUT_TOL, STAT_TOL, assert_close, compare_cache

pytestmark = pytest.mark.gpu

STEPS = 10


def test_two_batches_on_two_streams(cuda):
    ws = [synth.make_workload(2, L=2, batch=3, n=700, budget=512, steps=STEPS, tail=(200, 300),
                              periods=(6, 20)),
          synth.make_workload(3, L=2, batch=4, n=900, budget=384, steps=STEPS, periods=(8, 16))]
    streams = [torch.cuda.Stream(device=cuda), torch.cuda.Stream(device=cuda)]
    prm_o, prm_g = oracle.params(), lg.lg_default_params()
    refs, caches, guards, budgets = [], [], [], []
    for w in ws:
        K, V = synth.host_cache(w)
        refs.append(oracle.OracleGuard(w, K.copy(), V.copy(), prm_o))
        cache = lg.Cache.from_host(w, K, V, cuda, params=prm_g)
        caches.append(cache)
        guards.append(lg.Guard(cache, w.H_q, prm_g))
        budgets.append(torch.as_tensor(w.budget.astype(np.int32), device=cuda))
    torch.cuda.synchronize()
    seqs = [w.seqs.copy() for w in ws]
    pos = [w.n0.astype(np.int64) for w in ws]
    triggers = prunes = 0
    for t in range(STEPS):
        host = [synth.host_step(w, pos[i], seqs[i]) for i, w in enumerate(ws)]
        dev = [[lg.host_to_device(x, cuda, w.dtype) for x in host[i]] for i, w in enumerate(ws)]
        torch.cuda.synchronize()
        # both steps enqueued before either is waited for: the two streams run side by side
        for i in range(2):
            q, kn, vn = dev[i]
            guards[i].step(q, kn, vn, budgets[i], stream=streams[i])
        for i, w in enumerate(ws):
            streams[i].synchronize()
            tag = "batch %d step %d" % (i, t)
            r = guards[i].results()
            q, kn, vn = host[i]
            r_ref = refs[i].step(q, kn, vn, pos[i])
            rt, ra = OUT_TOL[w.dtype]
            assert_close(r["out"], r_ref["out"], rt, ra, tag + " out")
            assert_close(r["stats"], r_ref["stats"], *STAT_TOL, what=tag + " stats")
            assert np.array_equal(r["flags"], r_ref["flags"]), tag
            assert np.array_equal(r["spans"], r_ref["spans"]), tag
            assert np.array_equal(r["len"], r_ref["len"]), tag
            for b in range(w.batch):
                kept = r_ref["kept"][b]
                if r["kept_count"][b] >= 0:
                    assert r["kept_count"][b] == len(kept), (tag, b)
                    assert np.array_equal(r["kept_idx"][b, :len(kept)], kept), (tag, b)
                    prunes += 1
            compare_cache(w, refs[i], caches[i], r["len"], tag)
            triggers += int(r["flags"].sum())
            synth.note_interventions(seqs[i], pos[i], r_ref["flags"])
            pos[i] = pos[i] + 1
    assert prunes >= 7, prunes
