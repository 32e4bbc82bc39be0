"""Token streams and loop labels for the synthetic analog of the paper's ablation (Sec. 6.5,
Table 3): which guard variant breaks planted loops, how often it intervenes, and how many of its
interventions come before the loop begins.  Harness only: no attention, detection or pruning
arithmetic lives here; the caller runs the guard (the GPU path or the oracle) and reports each
step's decisions back.

Model (a reading of the paper's setting; its data and models are not available):
  - healthy text: token ids drawn Zipf(1.1) over a 50 000-token vocabulary (so a 256-token
    window repeats tokens, TTR well below 1), top-1 probability uniform in [0.2, 0.8), with
    benign confident runs (a run of 4..12 steps with p_max in [0.9, 1) starts with
    probability 1/150 at a healthy step) -- the formatting spans that mislead a confidence-only
    trigger;
  - each sequence falls into a loop at a labelled onset (generated tokens), repeating the
    `period` tokens before the onset with p_max 0.95;
  - an intervention at or after the onset breaks the loop when the retained cache keeps fewer
    than `period` rows generated since the onset (the repetitive tail the attention locks
    onto is gone); otherwise the loop goes on, as the paper reports for untargeted pruning.
    A broken loop returns to healthy text to the end of the run.
Measures per variant: loop rate (sequences still looping at T_max), interventions per
sequence, early interventions (before the onset) as a fraction of all interventions.
"""
from __future__ import annotations

import numpy as np

VOCAB = 50_000


class LoopStreams:
    """One batch of sequences: prompt of n0 rows, T steps, per-sequence onset and period."""

    def __init__(self, batch: int, n0: int, steps: int, onset=(800, 1300), periods=(16, 64),
                 seed: int = 11):
        rng = np.random.default_rng(seed)
        self.batch, self.n0, self.steps = batch, n0, steps
        self.onset = rng.integers(onset[0], onset[1] + 1, size=batch)
        self.period = rng.integers(periods[0], periods[1] + 1, size=batch)
        # healthy text of every step, drawn up front (the same for every variant)
        ranks = rng.zipf(1.1, size=(steps, batch))
        self.healthy = ((ranks - 1) % VOCAB).astype(np.int32)
        pm = rng.uniform(0.2, 0.8, size=(steps, batch))
        for b in range(batch):
            t = 0
            while t < steps:
                if rng.random() < 1.0 / 150.0:
                    run = int(rng.integers(4, 13))
                    pm[t:t + run, b] = rng.uniform(0.9, 1.0, size=min(run, steps - t))
                    t += run
                else:
                    t += 1
        self.healthy_pm = pm.astype(np.float32)
        self.reset()

    def reset(self):
        self.broken = np.zeros(self.batch, dtype=bool)
        self.tokens = np.zeros((self.steps, self.batch), dtype=np.int32)
        # generated-token index of every cache row of each sequence (-1 = prompt row)
        self.slot_tok = [list([-1] * self.n0) for _ in range(self.batch)]
        self.interventions = np.zeros(self.batch, dtype=np.int64)
        self.early = np.zeros(self.batch, dtype=np.int64)

    def looping(self, b: int, t: int) -> bool:
        return t >= self.onset[b] and not self.broken[b]

    def step_inputs(self, t: int):
        """this step's token id and top-1 probability of every sequence"""
        tok = self.healthy[t].copy()
        pm = self.healthy_pm[t].copy()
        for b in range(self.batch):
            if self.looping(b, t):
                P, o = int(self.period[b]), int(self.onset[b])
                tok[b] = self.tokens[o - P + (t - o) % P, b]
                pm[b] = np.float32(0.95)
        self.tokens[t] = tok
        for b in range(self.batch):
            self.slot_tok[b].append(t)
        return tok, pm

    def after_step(self, t: int, flags, kept_lists):
        """flags[b]: the guard intervened at step t; kept_lists[b]: the retained slots when the
        cache of b was pruned this step (intervention or budget cut), else None"""
        for b in range(self.batch):
            if kept_lists[b] is not None:
                self.slot_tok[b] = [self.slot_tok[b][j] for j in kept_lists[b]]
            if not flags[b]:
                continue
            self.interventions[b] += 1
            if t < self.onset[b]:
                self.early[b] += 1
            elif not self.broken[b]:
                o = int(self.onset[b])
                loop_rows = sum(1 for g in self.slot_tok[b] if g >= o)
                if loop_rows < int(self.period[b]):
                    self.broken[b] = True

    def measures(self) -> dict:
        n_int = int(self.interventions.sum())
        return {"loop_rate_pct": round(100.0 * float(np.mean(~self.broken)), 2),
                "interventions_per_seq": round(n_int / self.batch, 3),
                "early_pct": round(100.0 * int(self.early.sum()) / n_int, 2) if n_int else None}


# guard variants of the ablation as parameter settings of the token-level monitor
# (None: no monitor, only the budget)
VARIANTS = {
    "no_guard": None,
    # untargeted pruning whenever warmup and cooldown allow: no votes (K = 0), a stall gate that
    # always holds (theta_nov above any novel fraction), and no tail span (the period search is
    # limited to P = 1, which these streams never show), so each prune keeps the recent rows
    "always_on": dict(K=0, theta_nov=2.0, p_min=1, p_max=1),
    # the top-1 confidence streak alone: votes 1 and 2 never fire (TTR and CR are positive),
    # one vote suffices, no gate
    "single_p1": dict(K=1, theta_ttr=0.0, theta_nov=2.0, theta_cr=0.0),
    "full": dict(),
}

TOKEN_PARAM_KEYS = ("cr_every", "theta_streak", "hist", "theta_cr", "theta_conf")


def split_params(over: dict):
    """a variant's overrides as (guard-parameter overrides, token-parameter overrides)"""
    g = {k: v for k, v in over.items() if k not in TOKEN_PARAM_KEYS}
    t = {k: v for k, v in over.items() if k in TOKEN_PARAM_KEYS}
    return g, t
