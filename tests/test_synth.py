"""Self-tests of the seeded workload generator (harness, not the method): determinism,
moments of the normals, bf16 rounding against torch, the planted loop structure and the
workload shapes of the five benchmark configurations."""
import numpy as np
import pytest

import synth


def test_normals_moments_and_determinism():
    z = synth.host_normals(1, synth_role := 1, 0, 0, 0, 0, 200000)
    assert abs(z.mean()) < 0.01 and abs(z.std() - 1.0) < 0.01
    assert np.abs(z).max() <= 2 * np.sqrt(3) + 1e-6         # Irwin-Hall(4) support
    z2 = synth.host_normals(1, synth_role, 0, 0, 0, 0, 200000)
    assert np.array_equal(z, z2)
    z3 = synth.host_normals(2, synth_role, 0, 0, 0, 0, 1000)
    assert not np.array_equal(z[:1000], z3)


def test_bf16_rounding_matches_torch():
    import torch
    w = synth.make_workload(2, L=1, batch=1, n=64, budget=64, steps=1)
    rows = synth.host_rows(w, 0, 0, 0, 0, 0, 64)
    w32 = synth.make_workload(2, L=1, batch=1, n=64, budget=64, steps=1)
    w32.dtype = "f32"
    rows32 = synth.host_rows(w32, 0, 0, 0, 0, 0, 64)
    t = torch.from_numpy(rows32).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(rows, t)


def test_planted_loop_structure():
    w = synth.make_workload(1)
    s = w.seqs[0]
    start, P = int(s["start"]), int(s["period"])
    assert (start, P) == (512 - 192, 24)
    K, V = synth.host_cache(w)
    for p in range(start, 512):
        src = start - P + (p - start) % P
        dk = np.abs(K[0, :, p] - K[0, :, src])
        assert dk.max() < 0.6 and dk.mean() < 0.15           # sigma = 0.1 noise
    # rows before the loop are independent draws
    assert np.abs(K[0, :, 100] - K[0, :, 124]).mean() > 0.5
    # fresh_from turns the rows loop-free again
    seqs = w.seqs.copy()
    seqs["fresh_from"][0] = 400
    r = synth.host_rows(w, 0, 0, 0, 0, 400, 1, seqs)
    assert np.abs(r[0] - K[0, 0, 400]).mean() > 0.5


def test_query_targets_repeated_key():
    """zstar queries give every copy of the repeated key a logit near zstar = 12"""
    w = synth.make_workload(2, L=1, batch=2, n=1024, budget=512, steps=1, tail=(512, 512),
                            periods=(32, 32))
    b = int(np.flatnonzero(w.seqs["looping"])[0])
    K, V = synth.host_cache(w)
    pos = w.n0.astype(np.int64)
    q, kn, vn = synth.host_step(w, pos)
    wid = lambda a: (a.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    s = w.seqs[b]
    src = int(s["start"]) - int(s["period"]) + (1024 - int(s["start"])) % int(s["period"])
    for h in range(w.H_q):
        kvh = h // w.g
        logit = wid(q[0, b, h]) @ wid(K[0, kvh, w.seq_off[b] + src]) / np.sqrt(128)
        assert abs(logit - 12.0) < 0.5


@pytest.mark.parametrize("i", [1, 2, 3, 4, 5])
def test_workload_shapes(i):
    w = synth.make_workload(i)
    expect = {1: (1, 8, 8, 64, "f32", 1), 2: (32, 32, 8, 128, "bf16", 8),
              3: (28, 12, 2, 128, "bf16", 32), 4: (32, 32, 8, 128, "bf16", 64),
              5: (32, 64, 8, 128, "bf16", 16)}[i]
    assert (w.L, w.H_q, w.H_kv, w.d, w.dtype, w.batch) == expect
    frac = {1: 1.0, 2: 0.5, 3: 0.6, 4: 0.3, 5: 0.5}[i]
    assert w.seqs["looping"].sum() == round(frac * w.batch)
    if i == 4:
        assert w.n0.min() >= 1024 and w.n0.max() <= 65536
        assert np.array_equal(w.budget, np.minimum(w.n0 + 256, 16384))
    assert np.all(w.cap >= np.maximum(w.n0, w.budget) + 1)


def test_paper_shaped_workload():
    """workload 6: the Qwen3-1.7B shape, one 3853-token prompt, B = 1024, T_max = 2500, a loop
    whose onset is 800-1300 generated tokens in, with a period of 16-64"""
    w = synth.make_workload(6)
    assert (w.L, w.H_q, w.H_kv, w.d, w.dtype, w.batch) == (28, 16, 8, 128, "bf16", 1)
    assert w.n0.tolist() == [3853] and w.budget.tolist() == [1024] and w.steps == 2500
    s = w.seqs[0]
    assert s["looping"] == 1 and 800 <= s["start"] - 3853 <= 1300 and 16 <= s["period"] <= 64


@pytest.mark.parametrize("i", [2, 3, 4, 5])
def test_loop_plans_follow_the_recipe(i):
    """the planted loops of each full-size workload: periods, tails, starts and onsets drawn from
    the stated ranges (workload 2: P 16-128, tail 1024-3072; 3: P 8-64, start in
    [3n/4, n - 4P]; 4: P 16-64, onset 0-200 steps after the prompt; 5: P 32, tail 16384)"""
    w = synth.make_workload(i)
    for b in np.flatnonzero(w.seqs["looping"]):
        s, n = w.seqs[b], int(w.n0[b])
        P, start = int(s["period"]), int(s["start"])
        if i == 2:
            assert 16 <= P <= 128 and 1024 <= n - start <= 3072
        elif i == 3:
            assert 8 <= P <= 64 and 3 * n // 4 <= start <= max(3 * n // 4, n - 4 * P)
        elif i == 4:
            assert 16 <= P <= 64 and 0 <= start - n <= 200
        else:
            assert P == 32 and n - start == 16384
    if i == 3:
        assert w.n_sink == 4 and w.sink_factor == 8.0
