"""Attention edge cases through the C ABI against the oracle: empty sequences in a batch (zero
output, m = -inf, l = H = S = 0), one-row sequences, and lengths on either side of a staging
tile (128 rows) and of a chunk (the split-K unit, 768 rows at this shape), in both cache dtypes."""
import numpy as np
import pytest
import torch

import oracle
import synth
from paper_2604_10044_gb300 import lg
from parity_util import OUT_TOL, STAT_TOL, assert_close

pytestmark = pytest.mark.gpu

LENS = [0, 1, 0, 127, 128, 129, 767, 768, 769, 1537, 0, 4097]


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_attend_empty_and_boundary_lengths(cuda, dtype):
    w = synth.make_workload(2, L=2, batch=len(LENS), n=64, budget=64, steps=1,
                            tail=(16, 32), periods=(4, 8))
    w.n0 = np.array(LENS, dtype=np.int32)
    w.budget = np.full(len(LENS), 8192, dtype=np.int32)
    w.cap = None
    w.dtype = dtype
    w.__post_init__()
    K, V = synth.host_cache(w)
    cache = lg.Cache.from_host(w, K, V, cuda)
    max_len = int(w.n0.max())
    q, _, _ = synth.host_step(w, w.n0.astype(np.int64))
    qd = lg.host_to_device(q, cuda, dtype)
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    out = torch.full((w.L, w.batch, w.H_q, w.d), 7.0, dtype=tdt, device=cuda)
    stats = torch.full((w.L, w.batch, w.H_q, 4), 7.0, dtype=torch.float32, device=cuda)
    ws = torch.empty(lg.lg_workspace_size(cache, w.H_q, w.L, max_len, 0) // 4 + 64,
                     dtype=torch.float32, device=cuda)
    scale = 1.0 / np.sqrt(w.d)
    lg.lg_decode_attend(cache, 0, w.L, qd, w.H_q, scale, out, stats, 64, 0, max_len, ws)
    torch.cuda.synchronize()
    assert lg.lg_read_device_status(cache) == 0
    o = lg.device_to_host(out)
    o = (o.astype(np.uint32) << 16).view(np.float32) if dtype == "bf16" else o
    st = stats.cpu().numpy()
    rt, ra = OUT_TOL[dtype]
    for layer in range(w.L):
        for b, n in enumerate(LENS):
            if n == 0:
                assert np.all(o[layer, b] == 0.0), (layer, b)
                assert np.all(st[layer, b, :, 0] == -np.inf), (layer, b)
                assert np.all(st[layer, b, :, 1:] == 0.0), (layer, b)
                continue
            off = int(w.seq_off[b])
            for kvh in range(w.H_kv):
                hs = slice(kvh * w.g, (kvh + 1) * w.g)
                o_ref, s_ref, _ = oracle.attend_group(q[layer, b, hs], K[layer, kvh, off:off + n],
                                                      V[layer, kvh, off:off + n])
                tag = "layer %d seq %d (n=%d) kv-head %d" % (layer, b, n, kvh)
                assert_close(o[layer, b, hs], o_ref, rt, ra, tag + " out")
                assert_close(st[layer, b, hs], s_ref, *STAT_TOL, what=tag + " stats")


def test_pass_direction_changes_no_result(cuda):
    """successive lg_decode_attend calls with one workspace walk the cache in opposite
    directions; the same inputs give bit-identical outputs and statistics, with the H2O score
    accumulation both off and on (ragged lengths, several chunks per group)"""
    w = synth.make_workload(4, L=2, batch=5, len_range=(40, 5000), budget_max=8192, steps=1,
                            onset_max=1, periods=(4, 8))
    K, V = synth.host_cache(w)
    for h2o in (0, 1):
        cache = lg.Cache.from_host(w, K, V, cuda, policy="h2o" if h2o else "loopguard")
        max_len = int(w.n0.max())
        if h2o:
            lg.lg_h2o_reset(cache, max_len)
        q, _, _ = synth.host_step(w, w.n0.astype(np.int64))
        qd = lg.host_to_device(q, cuda, "bf16")
        ws = torch.empty(lg.lg_workspace_size(cache, w.H_q, w.L, max_len, h2o) // 4 + 64,
                         dtype=torch.float32, device=cuda)
        runs = []
        for _ in range(2):
            out = torch.zeros((w.L, w.batch, w.H_q, w.d), dtype=torch.bfloat16, device=cuda)
            stats = torch.zeros((w.L, w.batch, w.H_q, 4), dtype=torch.float32, device=cuda)
            lg.lg_decode_attend(cache, 0, w.L, qd, w.H_q, 1.0 / np.sqrt(w.d), out, stats, 64,
                                h2o, max_len, ws)
            torch.cuda.synchronize()
            assert lg.lg_read_device_status(cache) == 0
            runs.append((out.cpu(), stats.cpu()))
        assert torch.equal(runs[0][0], runs[1][0]), h2o
        assert torch.equal(runs[0][1], runs[1][1]), h2o
