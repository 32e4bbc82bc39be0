"""Device-side error reporting through the sticky status word (no fault, trap or hang):
a sequence at capacity, a length above the call's max_len, and a budget with no room for the
retained set (in the retained-set kernel and in the token-level monitor's) each record their
code, later kernels skip their work, and the host reads the code with lg_read_device_status.
Host-side validation errors return before any launch."""
import numpy as np
import pytest
import torch

import synth
from paper_2604_10044_gb300 import lg

pytestmark = pytest.mark.gpu


def _small(cuda, **over):
    w = synth.make_workload(2, L=2, batch=2, n=300, budget=256, steps=1, tail=(80, 100),
                            periods=(5, 9), **over)
    K, V = synth.host_cache(w)
    cache = lg.Cache.from_host(w, K, V, cuda)
    return w, cache


def test_capacity_exhausted_sets_status(cuda):
    w, cache = _small(cuda)
    cache.len.copy_(cache.cap)                    # every slot in use
    lg.lg_begin_step(cache)
    assert lg.lg_read_device_status(cache) == 4   # LG_ERR_CAPACITY
    before = cache.lengths().copy()
    q, kn, vn = synth.host_step(w, w.n0.astype(np.int64))
    lg.lg_append(cache, 0, w.L, lg.host_to_device(kn, cuda, w.dtype),
                 lg.host_to_device(vn, cuda, w.dtype), None, lg.lg_default_params())
    torch.cuda.synchronize()
    assert np.array_equal(cache.lengths(), before)   # later kernels skipped their work
    assert lg.lg_status_string(4).startswith("sequence length")


def test_max_len_below_a_length_sets_status(cuda):
    w, cache = _small(cuda)
    g = lg.Guard(cache, w.H_q)
    q = torch.zeros((w.L, w.batch, w.H_q, w.d), dtype=torch.bfloat16, device=cuda)
    lg.lg_decode_attend(cache, 0, w.L, q, w.H_q, 0.1, g.out, g.stats, 64, 0, 100, g.ws)
    assert lg.lg_read_device_status(cache) == 4


def test_budget_without_room_sets_status(cuda):
    w, cache = _small(cuda)
    g = lg.Guard(cache, w.H_q)
    budget = torch.full((w.batch,), 60, dtype=torch.int32, device=cuda)   # < anchors + headroom
    lg.lg_prune_compact(cache, None, None, None, budget, g.p, g.kept_idx, g.kept_count,
                        g.max_keep, g.max_len)
    assert lg.lg_read_device_status(cache) == 7   # LG_ERR_BUDGET


def test_token_prune_budget_without_room_sets_status(cuda):
    """lg_token_detect_prune: the token-level monitor's kernel records LG_ERR_BUDGET when the
    budget leaves no room for the retained set, before it writes a kept list or a length, and
    the compaction after it skips its work"""
    w, cache = _small(cuda)
    g = lg.Guard(cache, w.H_q)
    tp = lg.lg_default_token_params()
    tstate = torch.zeros(lg.lg_token_state_size(cache, g.p, tp) // 4, dtype=torch.int32,
                         device=cuda)
    lg.lg_state_init(cache, g.state, 0)
    tok = torch.arange(w.batch, dtype=torch.int32, device=cuda)
    pm = torch.full((w.batch,), 0.5, dtype=torch.float32, device=cuda)
    budget = torch.full((w.batch,), 60, dtype=torch.int32, device=cuda)   # < anchors + headroom
    g.kept_count.fill_(-1)
    before, k0 = cache.lengths().copy(), cache.k.clone()
    lg.lg_token_detect_prune(cache, tok, pm, g.state, budget, g.p, tp, g.flags, g.spans, None,
                             tstate, g.kept_idx, g.kept_count, g.max_keep, g.max_len)
    assert lg.lg_read_device_status(cache) == 7   # LG_ERR_BUDGET
    assert np.array_equal(cache.lengths(), before)
    assert (g.kept_count.cpu() == -1).all()
    assert torch.equal(cache.k, k0)


def test_host_validation_launches_nothing(cuda):
    w, cache = _small(cuda)
    g = lg.Guard(cache, w.H_q)
    q = torch.zeros((w.L, w.batch, w.H_q, w.d), dtype=torch.bfloat16, device=cuda)
    with pytest.raises(lg.LgError) as e:        # workspace too small
        lg.lg_decode_attend(cache, 0, w.L, q, w.H_q, 0.1, g.out, g.stats, 64, 0, g.max_len,
                            g.ws[:16])
    assert e.value.code == 6
    with pytest.raises(lg.LgError) as e:        # misaligned query pointer
        lg.lg_decode_attend(cache, 0, w.L, q.view(-1)[1:], w.H_q, 0.1, g.out, g.stats, 64, 0,
                            g.max_len, g.ws)
    assert e.value.code == 1
    assert lg.lg_read_device_status(cache) == 0


def test_nan_row_propagates_and_votes_off(cuda):
    """a NaN value row gives NaN outputs for the heads that read it; a NaN statistic turns its
    vote off (the detector's NaN policy), without any device error"""
    w, cache = _small(cuda)
    g = lg.Guard(cache, w.H_q)
    cache.v[0, 0, 5, 0] = float("nan")
    q, kn, vn = synth.host_step(w, w.n0.astype(np.int64))
    r = g.step_host(q, kn, vn, w.budget)
    assert np.isnan(r["out"][0, 0, :w.g, 0]).all()          # heads of kv-head 0, sequence 0
    assert np.isfinite(r["out"][0, 1]).all()                 # the other sequence is untouched
    assert np.isfinite(r["stats"][:, 0, :, 2]).all()         # entropy ignores values
