"""GPU <-> oracle parity through the C ABI on seeded workloads.

Small cases follow the structure of the five benchmark workloads at sizes the oracle finishes
in seconds, every step compared in full (outputs, statistics, flags, spans, kept lists,
compacted caches).  Shapes span several staging tiles, several CTA chunks and ragged tails.
"""
import numpy as np
import pytest
import torch

import synth
from parity_util import run_h2o, run_loopguard, run_streaming

pytestmark = pytest.mark.gpu


def test_tiny_single_layer_guard(cuda):
    """workload 1 exactly as specified: 1 layer, 8/8 heads, d=64, fp32, n=512, B=256"""
    w = synth.make_workload(1)
    c = run_loopguard(w, cuda)
    assert c["triggers"] == 1 and c["prunes"] == 1


def test_llama_shaped_small_multistep(cuda):
    """workload 2 structure (GQA 4, bf16, d=128, half the sequences looping) at 2 layers,
    n=1200, B=768: budget events on step 1, loop triggers, cooldown and re-triggers"""
    w = synth.make_workload(2, L=2, batch=4, n=1200, budget=768, steps=40, tail=(300, 500),
                            periods=(8, 40))
    c = run_loopguard(w, cuda)
    assert c["triggers"] >= 1 and c["prunes"] >= 4


@pytest.mark.parametrize("per_call", [1, 2])
def test_per_layer_calls_match(cuda, per_call):
    """the same workload with lg_decode_attend called per layer, or per two layers (calls of 2
    and 1 layers on one workspace: a different group count per call)"""
    w = synth.make_workload(2, L=3, batch=2, n=700, budget=512, steps=6, tail=(200, 300),
                            periods=(10, 30))
    run_loopguard(w, cuda, n_layers_per_call=per_call)


def test_separate_detect_and_prune_calls(cuda):
    """lg_detect then lg_prune_compact (the retained set in its own kernel) on the workload 2
    structure: the same results as the fused call"""
    w = synth.make_workload(2, L=2, batch=4, n=1200, budget=768, steps=40, tail=(300, 500),
                            periods=(8, 40))
    c = run_loopguard(w, cuda, fused_prune=False)
    assert c["triggers"] >= 1 and c["prunes"] >= 4


def test_small_model_sinks_gqa6(cuda):
    """workload 3 structure: 12/2 heads (GQA 6), attention sinks x8, loops after 75% of n"""
    w = synth.make_workload(3, L=2, batch=5, n=1500, budget=512, steps=12, periods=(8, 24))
    c = run_loopguard(w, cuda)
    assert c["prunes"] >= 5


def test_ragged_batch(cuda):
    """workload 4 structure: log-uniform lengths, budget min(n + 256, B_max), late loop onset"""
    w = synth.make_workload(4, L=2, batch=6, len_range=(40, 3000), budget_max=1024, steps=24,
                            onset_max=4, periods=(4, 8))
    run_loopguard(w, cuda)


def test_gqa8_and_short_rows(cuda):
    """workload 5 structure (64/8 heads -> GQA 8) with short sequences: lengths below one
    staging tile and one row over a tile boundary"""
    w = synth.make_workload(5, L=1, batch=3, n=33, budget=512, steps=3, tail=16, period=4)
    run_loopguard(w, cuda)
    w = synth.make_workload(5, L=2, batch=2, n=640, budget=384, steps=4, tail=200, period=8)
    run_loopguard(w, cuda)


@pytest.mark.parametrize("dtype,d", [("f32", 128), ("bf16", 64), ("f32", 64)])
def test_other_dtypes_and_head_dims(cuda, dtype, d):
    w = synth.make_workload(2, L=2, batch=2, n=500, budget=384, steps=3, tail=(150, 200),
                            periods=(5, 12), H_q=8, H_kv=4)
    w.dtype, w.d = dtype, d
    w.__post_init__()
    run_loopguard(w, cuda)


@pytest.mark.parametrize("H_q,H_kv,d", [(8, 8, 128), (6, 2, 128), (10, 2, 128), (7, 1, 128),
                                        (20, 4, 64)])
def test_every_gqa_group(cuda, H_q, H_kv, d):
    """the tensor-core pass at the GQA groups the benchmark shapes do not reach (g = 1, 3, 5,
    7; odd groups store their logits one by one and pad the MMA columns differently) on the
    guarded path, budget cuts and loops included"""
    w = synth.make_workload(2, L=2, batch=3, n=600, budget=384, steps=4, tail=(150, 250),
                            periods=(5, 16), H_q=H_q, H_kv=H_kv)
    w.d = d
    w.__post_init__()
    run_loopguard(w, cuda)


@pytest.mark.parametrize("H_q,H_kv", [(2, 2), (4, 2), (6, 2), (16, 2)])
def test_h2o_every_load_width(cuda, H_q, H_kv):
    """the H2O score update at g = 1, 2, 3, 8: logits read one, two, one and four at a time"""
    w = synth.make_workload(2, L=2, batch=3, n=400, budget=256, steps=4, H_q=H_q, H_kv=H_kv,
                            tail=(100, 150), periods=(6, 20))
    assert run_h2o(w, cuda) >= 3 * 4


def test_h2o_comparator(cuda):
    """H2O path: first cut from n > B + 1 to B (radix select + ordered gather), then one
    swap-remove per step"""
    w = synth.make_workload(2, L=2, batch=3, n=400, budget=256, steps=5, H_q=8, H_kv=2,
                            tail=(100, 150), periods=(6, 20))
    assert run_h2o(w, cuda) >= 3 * 5


def test_h2o_ragged(cuda):
    w = synth.make_workload(4, L=1, batch=5, len_range=(100, 1500), budget_max=512, steps=4,
                            periods=(4, 8), onset_max=2)
    run_h2o(w, cuda)


def test_device_generator_matches_host(cuda):
    """the device twin of the workload generator returns the host twin's bits"""
    w = synth.make_workload(3, L=2, batch=3, n=300, budget=128, steps=2, periods=(8, 16))
    K, V = synth.host_cache(w)
    dt = torch.bfloat16
    Kd = torch.zeros((w.L, w.H_kv, w.S_total, w.d), dtype=dt, device=cuda)
    Vd = torch.zeros_like(Kd)
    seqs = synth.seqs_tensor(w.seqs, cuda)
    off = torch.as_tensor(w.seq_off, device=cuda)
    n0 = torch.as_tensor(w.n0, device=cuda)
    s = torch.cuda.current_stream().cuda_stream
    synth.dev_fill_cache(w, Kd, Vd, seqs, off, n0, int(w.n0.max()), s)
    torch.cuda.synchronize()
    from paper_2604_10044_gb300.lg import device_to_host
    assert np.array_equal(device_to_host(Kd), K) and np.array_equal(device_to_host(Vd), V)
    pos = w.n0.astype(np.int64) + 5
    q, kn, vn = synth.host_step(w, pos)
    qd = torch.zeros((w.L, w.batch, w.H_q, w.d), dtype=dt, device=cuda)
    kd = torch.zeros((w.L, w.batch, w.H_kv, w.d), dtype=dt, device=cuda)
    vd = torch.zeros_like(kd)
    synth.dev_step(w, seqs, torch.as_tensor(pos, device=cuda), qd, kd, vd, s)
    torch.cuda.synchronize()
    assert np.array_equal(device_to_host(qd), q)
    assert np.array_equal(device_to_host(kd), kn) and np.array_equal(device_to_host(vd), vn)


def test_streaming_comparator(cuda):
    """StreamingLLM path: first cut from n > B + 1 to sinks + window, then one oldest-row
    eviction per step, ragged lengths"""
    w = synth.make_workload(4, L=2, batch=4, len_range=(100, 900), budget_max=384, steps=4,
                            periods=(4, 8), onset_max=2)
    run_streaming(w, cuda)


def test_streaming_window_wraps(cuda):
    """StreamingLLM over 150 steps with a 64-row budget (4 sinks + a 60-row window): the window's
    slots are refilled in ring order and wrap twice; every step's rows and positions match the
    oracle's oldest-row eviction"""
    w = synth.make_workload(4, L=1, batch=3, len_range=(100, 300), budget_max=64, steps=150,
                            periods=(4, 8), onset_max=2)
    run_streaming(w, cuda)


@pytest.mark.parametrize("policy", ["h2o", "streaming"])
def test_comparators_at_the_paper_shape(cuda, policy):
    """H2O and StreamingLLM at the paper's setting with all 28 layers (16/8 heads, the 3853-row
    prompt, B = 1024): the first cut to the budget, then 80 steps of one eviction each (H2O's
    one-pass choice of the lowest score, StreamingLLM's slot of the window's oldest row),
    every step's outputs, statistics, rows and positions against the oracle"""
    w = synth.make_workload(6, steps=80)
    if policy == "h2o":
        run_h2o(w, cuda)
    else:
        run_streaming(w, cuda)


def test_paper_shaped_guard(cuda):
    """workload 6 structure (the paper's setting: 16/8 heads, one 3853-token prompt, B=1024):
    the first budget cut from 3854 rows, periodic budget cuts every B - T_keep steps, and a
    planted loop that triggers, at 2 layers and an early onset"""
    w = synth.make_workload(6, L=2, onset=(90, 110), steps=200)
    c = run_loopguard(w, cuda)
    assert c["triggers"] >= 1 and c["prunes"] >= 3


@pytest.mark.parametrize("over", [
    # a window wider than one thread stride, periods from 3 (compared directly), 2 repeats,
    # a 6-row stall, one vote
    dict(W=400, p_min=3, p_max=40, m_rep=2, l_min=16, stall_len=6, K=1),
    # a narrow window, all three votes, a short cooldown and warmup
    dict(W=100, p_max=60, K=3, theta_lift=1.5, cooldown=8, t_min=10, retrig_window=20),
    # a window wider than the detect CTA (512 threads): several rounds of comparisons and of
    # the latest-match scan
    dict(W=700, p_max=100),
])
def test_nondefault_guard_params(cuda, over):
    """the same pipeline under other monitor constants: both sides take the same parameters"""
    w = synth.make_workload(2, L=2, batch=4, n=1200, budget=768, steps=40, tail=(300, 500),
                            periods=(8, 40))
    run_loopguard(w, cuda, params=over)


def test_sketch_rows_of_six_chunks(cuda):
    """6 kv-heads of d = 128: a sketch row of 24 words is 6 16-byte chunks, not a power of two,
    so the loop-onset test compares the new row a row per thread instead of a chunk per lane"""
    w = synth.make_workload(2, L=2, batch=4, n=1200, budget=768, steps=40, tail=(300, 500),
                            periods=(8, 40), H_q=12, H_kv=6)
    c = run_loopguard(w, cuda)
    assert c["triggers"] >= 1 and c["prunes"] >= 4
