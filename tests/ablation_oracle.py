"""The ablation variants (synth.ablation) driven by the oracle: the token-level monitor and the
retained set of every sequence, step by step, as the GPU driver runs them."""
import numpy as np

import oracle
from synth.ablation import split_params


def run_variant_oracle(streams, over, budget=1024):
    streams.reset()
    b, n0, T = streams.batch, streams.n0, streams.steps
    g_over, t_over = split_params(over or {})
    prm = oracle.params(**g_over)
    tp = oracle.token_params(**t_over)
    st = [oracle.new_state(0) for _ in range(b)]
    ts = [oracle.new_token_state() for _ in range(b)]
    n = np.full(b, n0, dtype=np.int64)
    prev_kept = [None] * b
    all_flags = np.zeros((T, b), dtype=np.int32)
    for t in range(T):
        tok, pm = streams.step_inputs(t)
        flags = np.zeros(b, dtype=np.int32)
        kept = [None] * b
        for s in range(b):
            n[s] += 1
            f, span, level = 0, (0, 0), 0
            if over is not None:
                f, span, _ = oracle.token_detect(streams.tokens[:t + 1, s], float(pm[s]),
                                                 int(n[s]), prm, tp, st[s], ts[s],
                                                 kept=prev_kept[s])
                level = st[s].level
            if f or n[s] > budget:
                kept[s] = oracle.keep_set(int(n[s]), budget, f, span, level, prm)
                n[s] = len(kept[s])
            prev_kept[s] = kept[s]
            flags[s] = f
        streams.after_step(t, flags, kept)
        all_flags[t] = flags
    return streams.measures(), all_flags
