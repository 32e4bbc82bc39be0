"""The ablation analog (Sec. 6.5, Table 3) driven by the oracle on the CPU, for the full batch of
64 sequences `bench.py --ablation` runs.  The oracle alone gives the reported table (loop rate
%, interventions per sequence, early %): the GPU path's decisions equal the oracle's at every
step (tests/test_gpu_ablation.py), so the figures `bench.py --ablation` prints are these.
Without a guard every loop survives to T_max; the full guard never intervenes before a loop
begins, and the loops it misses are exactly those whose period holds more than 51 distinct
tokens, which keep a window's TTR at or above theta_ttr = 0.2 (distinct / 256) so that only
the confidence vote fires."""
import numpy as np

from ablation_oracle import run_variant_oracle
from synth.ablation import VARIANTS, LoopStreams


def test_the_reported_table_is_the_oracles():
    s = LoopStreams(64, 3853, 2500)
    want = {"no_guard": (100.0, 0.0, None), "always_on": (21.88, 74.0, 42.48),
            "single_p1": (0.0, 12.109, 38.45), "full": (7.81, 0.922, 0.0)}
    for name, (rate, per_seq, early) in want.items():
        m, _ = run_variant_oracle(s, VARIANTS[name])
        assert (m["loop_rate_pct"], m["interventions_per_seq"], m["early_pct"]) == \
            (rate, per_seq, early), name
    # after the full guard (the last variant run): its misses are the >51-distinct loops
    distinct = np.array([len(set(s.tokens[int(s.onset[b]) - int(s.period[b]):int(s.onset[b]),
                                          b].tolist())) for b in range(64)])
    missed = ~s.broken
    assert np.array_equal(missed, distinct > 51)
    assert 0 < missed.sum() < 64
