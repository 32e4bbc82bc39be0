"""The ablation analog (Sec. 6.5, Table 3) driven by the oracle on the CPU, for the full batch of
64 sequences `bench.py --ablation` runs: without a guard every loop survives to T_max; the full
guard never intervenes before a loop begins, and the loops it misses are exactly those whose
period holds more than 51 distinct tokens, which keep a window's TTR at or above theta_ttr = 0.2
(distinct / 256) so that only the confidence vote fires."""
import numpy as np

from ablation_oracle import run_variant_oracle
from synth.ablation import VARIANTS, LoopStreams


def test_no_guard_and_full_guard():
    s = LoopStreams(64, 3853, 2500)
    m, flags = run_variant_oracle(s, VARIANTS["no_guard"])
    assert m["loop_rate_pct"] == 100.0 and m["interventions_per_seq"] == 0.0
    m, flags = run_variant_oracle(s, VARIANTS["full"])
    assert m["early_pct"] == 0.0
    distinct = np.array([len(set(s.tokens[int(s.onset[b]) - int(s.period[b]):int(s.onset[b]),
                                          b].tolist())) for b in range(64)])
    missed = ~s.broken
    assert np.array_equal(missed, distinct > 51)
    assert 0 < missed.sum() < 64
