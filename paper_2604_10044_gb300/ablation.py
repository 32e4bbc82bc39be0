"""The guard variants of the paper's ablation (Sec. 6.5, Table 3) run on the GPU path over a
batch of synthetic loop streams (synth.ablation): each step reserves the token's cache row,
runs the token-level monitor with the variant's parameters (none for "no guard") and the
retained set with its compaction, and reports the decisions back to the stream model."""
from __future__ import annotations

import numpy as np
import torch

from . import lg


def run_variant(streams, over, device, budget=1024, stream=None):
    """Run one variant over streams (synth.ablation.LoopStreams, reset here); over: parameter
    overrides, or None for no monitor.  Returns (measures dict, per-step flags [steps][batch])."""
    from synth.ablation import split_params
    streams.reset()
    b, n0, T = streams.batch, streams.n0, streams.steps
    cap = np.full(b, n0 + T + 1, dtype=np.int32)
    seq_off = np.concatenate([[0], np.cumsum(cap)[:-1]]).astype(np.int64)
    cache = lg.Cache(1, 1, 128, "f32", seq_off, cap, np.full(b, n0, dtype=np.int32), device,
                     "loopguard")
    g_over, t_over = split_params(over or {})
    prm = lg.lg_default_params(**g_over)
    tp = lg.lg_default_token_params(**t_over)
    state = torch.zeros((b, lg.STATE_BYTES // 4), dtype=torch.int32, device=device)
    lg.lg_state_init(cache, state, 0, stream)
    tstate = torch.zeros(lg.lg_token_state_size(cache, prm, tp) // 4, dtype=torch.int32,
                         device=device)
    flags = torch.zeros(b, dtype=torch.int32, device=device)
    spans = torch.zeros((b, 2), dtype=torch.int32, device=device)
    budget_d = torch.full((b,), budget, dtype=torch.int32, device=device)
    max_keep = int(max(cap.max(), budget))
    kept_idx = torch.zeros((b, max_keep), dtype=torch.int32, device=device)
    kept_count = torch.zeros(b, dtype=torch.int32, device=device)
    tok_d = torch.zeros(b, dtype=torch.int32, device=device)
    pm_d = torch.zeros(b, dtype=torch.float32, device=device)
    all_flags = np.zeros((T, b), dtype=np.int32)
    for t in range(T):
        tok, pm = streams.step_inputs(t)
        tok_d.copy_(torch.from_numpy(tok))
        pm_d.copy_(torch.from_numpy(pm))
        lg.lg_begin_step(cache, stream)
        if over is not None:
            lg.lg_token_detect_prune(cache, tok_d, pm_d, state, budget_d, prm, tp, flags, spans,
                                     None, tstate, kept_idx, kept_count, max_keep, int(cap.max()),
                                     stream)
        else:
            lg.lg_prune_compact(cache, None, None, None, budget_d, prm, kept_idx, kept_count,
                                max_keep, int(cap.max()), stream)
        f = flags.cpu().numpy() if over is not None else np.zeros(b, dtype=np.int32)
        kc = kept_count.cpu().numpy()
        kept = [None] * b
        pruned = np.flatnonzero(kc >= 0)
        if pruned.size:
            ki = kept_idx[torch.as_tensor(pruned, device=device)].cpu().numpy()
            for r, s in enumerate(pruned):
                kept[s] = ki[r, :kc[s]]
        streams.after_step(t, f, kept)
        all_flags[t] = f
    if lg.lg_read_device_status(cache, stream) != 0:
        raise RuntimeError("device status %d after the ablation run"
                           % lg.lg_read_device_status(cache, stream))
    return streams.measures(), all_flags
