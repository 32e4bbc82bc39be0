"""The guard variants of the ablation analog (Sec. 6.5, Table 3; synth.ablation) on the GPU path
(paper_2604_10044_gb300.ablation) against the same variants driven by the oracle, on a reduced
batch and on the full batch `bench.py --ablation` runs: identical interventions at every step,
identical measures."""
import numpy as np
import pytest

import synth.ablation as A
from ablation_oracle import run_variant_oracle
from paper_2604_10044_gb300.ablation import run_variant

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("variant", list(A.VARIANTS))
def test_ablation_variant_matches_oracle(cuda, variant):
    streams = A.LoopStreams(8, 1500, 1400, onset=(300, 600), periods=(8, 60), seed=5)
    over = A.VARIANTS[variant]
    m_g, f_g = run_variant(streams, over, cuda)
    m_o, f_o = run_variant_oracle(streams, over)
    bad = np.argwhere(f_g != f_o)
    assert bad.size == 0, (variant, bad[:5].tolist())
    assert m_g == m_o, (variant, m_g, m_o)


def test_full_ablation_batch_matches_oracle(cuda):
    """the batch bench.py --ablation reports (64 sequences, a 3853-token prompt, B = 1024, 2500
    steps): every variant's interventions at every step and its measures equal the oracle's, so
    the printed table is the oracle's"""
    streams = A.LoopStreams(64, 3853, 2500)
    for variant, over in A.VARIANTS.items():
        m_g, f_g = run_variant(streams, over, cuda)
        m_o, f_o = run_variant_oracle(streams, over)
        bad = np.argwhere(f_g != f_o)
        assert bad.size == 0, (variant, bad[:5].tolist())
        assert m_g == m_o, (variant, m_g, m_o)
