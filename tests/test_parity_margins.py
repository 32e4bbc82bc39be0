"""The GPU parity runs compare the guard's decisions bit for bit, float votes included: that is
sound only if no step's mean entropy or suffix lift lands next to its threshold, where fp32
statistics on the GPU and fp64 ones in the oracle could take different sides.  This runs the
oracle alone over the loop-guard workloads of tests/test_gpu_parity.py and the full-size
multi-step one of tests/test_gpu_fullsize.py (the same seeds, shapes and step counts) and checks that every step keeps both means at least 1 % from theta_ent and
theta_lift (the tie band of the statistics' tolerance is 1e-4)."""
import numpy as np
import pytest

import oracle
import synth

def _dtype_case(dtype, d):
    w = synth.make_workload(2, L=2, batch=2, n=500, budget=384, steps=3, tail=(150, 200),
                            periods=(5, 12), H_q=8, H_kv=4)
    w.dtype, w.d = dtype, d
    w.__post_init__()
    return w


CASES = [
    ("tiny", lambda: synth.make_workload(1), {}),
    ("llama-small", lambda: synth.make_workload(2, L=2, batch=4, n=1200, budget=768, steps=40,
                                                tail=(300, 500), periods=(8, 40)), {}),
    ("per-layer", lambda: synth.make_workload(2, L=3, batch=2, n=700, budget=512, steps=6,
                                              tail=(200, 300), periods=(10, 30)), {}),
    ("sinks-gqa6", lambda: synth.make_workload(3, L=2, batch=5, n=1500, budget=512, steps=12,
                                               periods=(8, 24)), {}),
    ("ragged", lambda: synth.make_workload(4, L=2, batch=6, len_range=(40, 3000),
                                           budget_max=1024, steps=24, onset_max=4,
                                           periods=(4, 8)), {}),
    ("gqa8-short", lambda: synth.make_workload(5, L=1, batch=3, n=33, budget=512, steps=3,
                                               tail=16, period=4), {}),
    ("gqa8", lambda: synth.make_workload(5, L=2, batch=2, n=640, budget=384, steps=4, tail=200,
                                         period=8), {}),
    ("paper-shaped", lambda: synth.make_workload(6, L=2, onset=(90, 110), steps=200), {}),
    ("params-wide", lambda: synth.make_workload(2, L=2, batch=4, n=1200, budget=768, steps=40,
                                                tail=(300, 500), periods=(8, 40)),
     dict(W=400, p_min=3, p_max=40, m_rep=2, l_min=16, stall_len=6, K=1)),
    ("params-narrow", lambda: synth.make_workload(2, L=2, batch=4, n=1200, budget=768, steps=40,
                                                  tail=(300, 500), periods=(8, 40)),
     dict(W=100, p_max=60, K=3, theta_lift=1.5, cooldown=8, t_min=10, retrig_window=20)),
    ("params-700", lambda: synth.make_workload(2, L=2, batch=4, n=1200, budget=768, steps=40,
                                               tail=(300, 500), periods=(8, 40)),
     dict(W=700, p_max=100)),
    ("six-kv-heads", lambda: synth.make_workload(2, L=2, batch=4, n=1200, budget=768, steps=40,
                                                 tail=(300, 500), periods=(8, 40), H_q=12,
                                                 H_kv=6), {}),
    # test_gpu_fullsize.py::test_llama8b_full_size_four_steps (about 25 s here)
    ("llama-full-size", lambda: synth.make_workload(2, steps=4), {}),
] + [("%s-d%d" % (dt, d), (lambda dt=dt, d=d: _dtype_case(dt, d)), {})
     for dt, d in (("f32", 128), ("bf16", 64), ("f32", 64))]


@pytest.mark.parametrize("name,make,over", CASES, ids=[c[0] for c in CASES])
def test_parity_workloads_stay_clear_of_the_float_thresholds(name, make, over):
    w = make()
    K, V = synth.host_cache(w)
    prm = oracle.params(**over)
    g = oracle.OracleGuard(w, K, V, prm)
    seqs, pos = w.seqs.copy(), w.n0.astype(np.int64)
    closest = 1.0
    for _ in range(w.steps):
        q, kn, vn = synth.host_step(w, pos, seqs)
        r = g.step(q, kn, vn, pos)
        for d in r["diags"]:
            if d is not None:
                closest = min(closest, abs(d["ebar"] - prm.theta_ent) / prm.theta_ent,
                              abs(d["lbar"] - prm.theta_lift) / prm.theta_lift)
        synth.note_interventions(seqs, pos, r["flags"])
        pos = pos + 1
    assert closest >= 0.01, (name, closest)
