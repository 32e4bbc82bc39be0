"""GPU <-> oracle parity of the token-level monitor (lg_token_detect, Sec. 5.2, Eq. 8, Eq. 9,
App. B.2) feeding the retained set (lg_prune_compact), through the C ABI, step by step on
scripted token streams: a healthy stream, loops of periods 8 (with and without the confidence
signal), 20 and 3, and a noisy small-alphabet stream; two of them under a budget the cache
outgrows (budget cuts change the length the monitor maps spans onto).  Flags, spans, every
diagnostic, the guard state, kept counts and lengths are compared exactly."""
import numpy as np
import pytest
import torch

import oracle
from paper_2604_10044_gb300 import lg

pytestmark = pytest.mark.gpu

STEPS = 620
N0 = 100          # prompt rows in the cache before the first generated token


def _streams(rng):
    healthy = lambda k, base: (np.arange(k) + base).astype(np.int32)
    loop = lambda k, P, base: (np.arange(k) % P + base).astype(np.int32)
    toks, pm = [], []
    # 0: healthy, drawn from a large vocabulary
    toks.append(rng.integers(0, 60_000, STEPS).astype(np.int32))
    pm.append(rng.uniform(0.2, 0.95, STEPS))
    # 1: 300 healthy then a period-8 loop, confident
    toks.append(np.concatenate([healthy(300, 10_000), loop(STEPS - 300, 8, 1)]))
    pm.append(np.where(np.arange(STEPS) >= 300, 0.95, 0.5))
    # 2: the same loop without the confidence signal (diversity + redundancy votes)
    toks.append(np.concatenate([healthy(300, 20_000), loop(STEPS - 300, 8, 1)]))
    pm.append(np.full(STEPS, 0.5))
    # 3: 200 healthy then a period-20 loop, confident
    toks.append(np.concatenate([healthy(200, 30_000), loop(STEPS - 200, 20, 1)]))
    pm.append(np.where(np.arange(STEPS) >= 200, 0.97, 0.4))
    # 4: a short prefix then a period-3 loop (the warmup holds the first trigger back)
    toks.append(np.concatenate([healthy(20, 40_000), loop(STEPS - 20, 3, 1)]))
    pm.append(np.full(STEPS, 0.99))
    # 5: a small alphabet: frequent repeats, no period
    toks.append(rng.integers(0, 6, STEPS).astype(np.int32))
    pm.append(rng.uniform(0.85, 1.0, STEPS))
    # fp32 probabilities: both sides compare the same values
    return np.stack(toks), np.stack(pm).astype(np.float32)


OTHER = (dict(W=300, p_min=2, p_max=50, m_rep=2, l_min=24, stall_len=6, cooldown=16),
         dict(hist=320, cr_every=5, theta_streak=4))


@pytest.mark.parametrize("pass_kept,params,fused", [(True, None, False), (False, None, False),
                                                    (True, OTHER, False), (True, None, True),
                                                    (True, OTHER, True)])
def test_token_monitor_and_prune_match_oracle(cuda, pass_kept, params, fused):
    """pass_kept: the monitor gets the previous prune's retained lists (rows kept in order at
    the tail stay mapped to their tokens), or not (only rows appended since a prune are);
    params: (guard, token) parameter overrides, the same on both sides; fused: one
    lg_token_detect_prune call (the monitor's kernel forms the retained set over the previous
    lists it has just read) in place of lg_token_detect + lg_prune_compact"""
    rng = np.random.default_rng(7)
    toks, pmax = _streams(rng)
    b = toks.shape[0]
    budget_h = np.array([4096, 512, 4096, 512, 4096, 4096], dtype=np.int32)
    cap = np.full(b, N0 + STEPS + 2, dtype=np.int32)
    seq_off = np.concatenate([[0], np.cumsum(cap)[:-1]]).astype(np.int64)
    n0 = np.full(b, N0, dtype=np.int32)
    cache = lg.Cache(1, 1, 128, "f32", seq_off, cap, n0, cuda, "loopguard")
    g_over, t_over = params or ({}, {})
    prm_g, prm_o = lg.lg_default_params(**g_over), oracle.params(**g_over)
    tp_g, tp_o = lg.lg_default_token_params(**t_over), oracle.token_params(**t_over)
    state = torch.zeros((b, lg.STATE_BYTES // 4), dtype=torch.int32, device=cuda)
    lg.lg_state_init(cache, state, 0)
    tstate = torch.zeros(lg.lg_token_state_size(cache, prm_g, tp_g) // 4, dtype=torch.int32,
                         device=cuda)
    flags = torch.zeros(b, dtype=torch.int32, device=cuda)
    spans = torch.zeros((b, 2), dtype=torch.int32, device=cuda)
    diag = torch.zeros((b, 8), dtype=torch.float64, device=cuda)
    budget = torch.as_tensor(budget_h, device=cuda)
    max_keep = int(max(cap.max(), budget_h.max()))   # lg_prune_compact: >= every budget
    kept_idx = torch.zeros((b, max_keep), dtype=torch.int32, device=cuda)
    kept_count = torch.zeros(b, dtype=torch.int32, device=cuda)
    toks_d = torch.as_tensor(toks.T.copy(), device=cuda)       # [steps][b]
    pmax_d = torch.as_tensor(pmax.T.copy(), device=cuda)

    st_o = [oracle.new_state(0) for _ in range(b)]
    ts_o = [oracle.new_token_state() for _ in range(b)]
    n_o = n0.astype(np.int64).copy()
    prev_kept = [None] * b
    triggers = np.zeros(b, dtype=int)
    prunes = 0
    keys = ("ttr", "cr", "streak", "sig1", "sig2", "sig3", "stall", "P")
    for t in range(STEPS):
        lg.lg_begin_step(cache)
        if fused:
            lg.lg_token_detect_prune(cache, toks_d[t], pmax_d[t], state, budget, prm_g, tp_g,
                                     flags, spans, diag, tstate, kept_idx, kept_count, max_keep,
                                     int(cap.max()))
        else:
            lg.lg_token_detect(cache, toks_d[t], pmax_d[t], state, prm_g, tp_g, flags, spans,
                               diag, tstate, kept_idx if pass_kept else None,
                               kept_count if pass_kept else None)
            lg.lg_prune_compact(cache, flags, spans, state, budget, prm_g, kept_idx, kept_count,
                                max_keep, int(cap.max()))
        torch.cuda.synchronize()
        assert lg.lg_read_device_status(cache) == 0, t
        f_g, sp_g, dg_g = flags.cpu().numpy(), spans.cpu().numpy(), diag.cpu().numpy()
        st_g, kc_g, len_g = state.cpu().numpy(), kept_count.cpu().numpy(), cache.len.cpu().numpy()
        for s in range(b):
            n_o[s] += 1
            f, sp, dg = oracle.token_detect(toks[s, :t + 1], float(pmax[s, t]), int(n_o[s]),
                                            prm_o, tp_o, st_o[s], ts_o[s],
                                            kept=prev_kept[s] if pass_kept else None)
            prev_kept[s] = None
            ctx = (t, s, dg, dg_g[s].tolist(), sp, sp_g[s].tolist())
            assert f_g[s] == f and tuple(sp_g[s]) == sp, ctx
            assert [dg[k] for k in keys] == dg_g[s].tolist(), ctx
            so = st_o[s]
            assert st_g[s, :5].tolist() == [so.t_gen, so.cd, so.level, so.last_trig, so.n_int], ctx
            kept = oracle.keep_set(int(n_o[s]), int(budget_h[s]), f, sp, so.level, prm_o)
            if not f and n_o[s] <= budget_h[s]:
                assert kc_g[s] == -1, ctx
            else:
                assert kc_g[s] == len(kept) and np.array_equal(
                    kept_idx[s, :kc_g[s]].cpu().numpy(), kept), ctx
                n_o[s] = len(kept)
                prev_kept[s] = kept
                prunes += 1
            assert len_g[s] == n_o[s], ctx
            triggers[s] += f
    assert lg.lg_read_device_status(cache) == 0
    assert triggers[0] == 0 and triggers[1] >= 1 and triggers[3] >= 1 and triggers[4] >= 2
    assert prunes > triggers.sum()


def test_token_monitor_rejects_short_history(cuda):
    """hist must hold the window and every period test's reads"""
    cap = np.array([64], dtype=np.int32)
    cache = lg.Cache(1, 1, 128, "f32", np.zeros(1, np.int64), cap, np.zeros(1, np.int32), cuda)
    prm = lg.lg_default_params()
    assert lg.lg_token_state_size(cache, prm, lg.lg_default_token_params(hist=200)) == 0
    t = torch.zeros(64, dtype=torch.int32, device=cuda)
    with pytest.raises(lg.LgError):
        lg.lg_token_detect(cache, t, t.float(), t, prm, lg.lg_default_token_params(hist=200),
                           t, t, None, t)
    with pytest.raises(lg.LgError):   # kept lists without their counts
        lg.lg_token_detect(cache, t, t.float(), t, prm, lg.lg_default_token_params(), t, t, None,
                           t, kept_idx=t.view(1, 64), kept_count=None)
