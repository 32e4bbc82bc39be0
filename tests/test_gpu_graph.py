"""The guarded step replayed from a CUDA graph gives the same results as eager launches.

Every kernel of the library is launched with programmatic stream serialization, so inside a
captured graph consecutive kernels are joined by programmatic edges and may overlap; each
kernel's griddepcontrol.wait must still order it after its predecessor.  These tests run the
same steps of a seeded workload eagerly and as one graph replay (the way bench.py times them)
and compare the final cache, lengths, guard state and the last step's outputs bit for bit.
"""
import numpy as np
import pytest
import torch

import bench
import synth

pytestmark = pytest.mark.gpu


def _snapshot(b):
    c, g = b.cache, b.guard
    out = {"len": c.len.cpu().numpy().copy(), "k": c.k.cpu(), "v": c.v.cpu(),
           "out": g.out.cpu(), "stats": g.stats.cpu().numpy().copy(),
           "flags_spans": g.flags_spans.cpu().numpy().copy(),
           "status": c.status.cpu().numpy().copy()}
    if b.policy == "loopguard":
        out["state"] = g.state.cpu().numpy().copy()
        out["kept_count"] = g.kept_count.cpu().numpy().copy()
    if b.detector == "token":
        out["tstate"] = b.tstate.cpu().numpy().copy()
    return out


def _valid_rows(x, w, lens):
    """the cache rows in use: [L][H_kv][seq_off_b, seq_off_b + len_b) of every sequence"""
    parts = []
    for b_ in range(w.batch):
        o = int(w.seq_off[b_])
        parts.append(x[:, :, o:o + int(lens[b_])].reshape(-1))
    return torch.cat(parts)


@pytest.mark.parametrize("policy,detector", [("loopguard", "kv"), ("loopguard", "token"),
                                             ("h2o", "kv"), ("streaming", "kv")])
def test_graph_replay_matches_eager(cuda, policy, detector):
    w = synth.make_workload(2, L=2, batch=4, n=1200, budget=768, steps=40, tail=(300, 500),
                            periods=(8, 40))
    K = 24
    side = torch.cuda.Stream(device=cuda)
    with torch.cuda.stream(side):
        b = bench.GpuBench(w, cuda, K, None, policy, detector)
        b.reset()
        for t in range(K):
            b.step(t)
        torch.cuda.synchronize()
        eager = _snapshot(b)
        b.reset()
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=b.stream, capture_error_mode="thread_local"):
            for t in range(K):
                b.step(t)
        b.reset()
        graph.replay()
        torch.cuda.synchronize()
        replay = _snapshot(b)
    assert (eager["status"] == 0).all() and (replay["status"] == 0).all()
    np.testing.assert_array_equal(replay["len"], eager["len"])
    for key in ("stats", "flags_spans", "state", "kept_count", "tstate"):
        if key in eager:
            np.testing.assert_array_equal(replay[key], eager[key], err_msg=key)
    assert torch.equal(replay["out"], eager["out"])
    for key in ("k", "v"):
        assert torch.equal(_valid_rows(replay[key], w, eager["len"]),
                           _valid_rows(eager[key], w, eager["len"])), key
    if policy == "loopguard":
        # the steps pruned (budget events at least), so the replay compacted the cache too
        assert (eager["len"] < w.n0 + K).any()
