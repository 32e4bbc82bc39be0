"""GPU <-> oracle parity at the benchmark workloads' full sizes, in bench.py's launch
configuration (one lg_decode_attend call over all layers, max_len = capacity).

The device cache comes from the device generator, the oracle's rows from the host generator
(bit-identical by construction and by test_gpu_parity::test_device_generator_matches_host).
  attention: sampled (layer, sequence, kv-head) groups, every head of the group, one by one;
  detect:    every sequence, on seeded per-head statistics (so the oracle does not need the
             full-size attention) and each side's own sketches of the guard layer;
  prune:     every sequence's kept list, the compacted bytes of sampled streams, and the
             moved sketches of one pruned sequence.
The Llama-3-8B-shaped workload also runs four whole steps at full size, the attention's own
statistics driving the loop-onset test, every output and the whole cache compared each step.
"""
import math

import numpy as np
import pytest
import torch

import oracle
import synth
from paper_2604_10044_gb300 import lg
from parity_util import OUT_TOL, STAT_TOL, assert_close, run_loopguard

pytestmark = pytest.mark.gpu


def _rng_groups(w, k, seed):
    rng = np.random.default_rng(seed)
    groups = {(w.L - 1, 0, w.H_kv - 1)}
    while len(groups) < k:
        groups.add((int(rng.integers(w.L)), int(rng.integers(w.batch)), int(rng.integers(w.H_kv))))
    return sorted(groups)


def _seeded_stats(w, n, seed):
    """per (layer, sequence, head) statistics with sequence-level means well away from the
    vote thresholds: mean H / ln n in {0.4, 0.9}, mean S n / W_s in {1.0, 3.0}"""
    rng = np.random.default_rng(seed)
    st = np.zeros((w.L, w.batch, w.H_q, 4), dtype=np.float32)
    for b in range(w.batch):
        e = 0.4 if rng.random() < 0.6 else 0.9
        lam = 3.0 if rng.random() < 0.5 else 1.0
        ws = min(64, int(n[b]))
        jit = rng.uniform(0.9, 1.1, size=(w.L, w.H_q))
        st[:, b, :, 0] = 5.0
        st[:, b, :, 1] = 100.0
        st[:, b, :, 2] = e * math.log(n[b]) * jit
        st[:, b, :, 3] = np.minimum(lam * ws / n[b] * jit, 1.0)
    return st


def _guard_sketch_rows(w, b, lo, hi, seqs, v_new_row):
    """oracle sketches of rows [lo, hi) of sequence b (hi - 1 is the appended row)"""
    nrow = hi - 1 - lo
    V = np.stack([synth.host_rows(w, 1, 0, h, b, lo, nrow, seqs) for h in range(w.H_kv)], 1)
    rows = np.concatenate([V, v_new_row[None]], 0)  # [rows][H_kv][d]
    return np.stack([oracle.sketch(np.ascontiguousarray(r)) for r in rows])


def _oracle_detect(w, b, nb, B, st_seed, v_new_row, prm):
    """the oracle's test on sketches of the rows it reads: the window and the period tests
    need the last 512 rows; only a trigger with a tail period reads back to n - B/2 - P*"""
    for back in (700, B // 2 + 700):
        lo = max(0, nb - back)
        sk = np.zeros((nb, w.H_kv * w.d // 32), dtype=np.uint32)
        sk[lo:] = _guard_sketch_rows(w, b, lo, nb, w.seqs, v_new_row)
        st = oracle.new_state()
        f, sp, dg = oracle.detect(st_seed[:, b].astype(np.float64), sk, B, prm, st)
        if not (f and dg["P"] > 0) or lo == 0:
            break
    return f, sp, dg, st


def run_full_size(w, device, n_groups=4, n_streams=3, seed=0):
    import gc
    gc.collect()
    torch.cuda.empty_cache()
    need = w.kv_bytes() + (2 << 30)
    free, _ = torch.cuda.mem_get_info(device)
    if free < need:
        pytest.skip("needs %.1f GB of free device memory, %.1f GB free" % (need / 1e9, free / 1e9))
    s = torch.cuda.current_stream().cuda_stream
    cache = lg.Cache(w.L, w.H_kv, w.d, w.dtype, w.seq_off, w.cap, w.n0, device, "loopguard")
    seqs_d = synth.seqs_tensor(w.seqs, device)
    off_d = torch.as_tensor(w.seq_off, device=device)
    n0_d = torch.as_tensor(w.n0, device=device)
    synth.dev_fill_cache(w, cache.k, cache.v, seqs_d, off_d, n0_d, int(w.n0.max()), s)
    prm_g = lg.lg_default_params()
    prm_o = oracle.params()
    lg.lg_sketch_build(cache, prm_g, int(w.n0.max()))
    guard = lg.Guard(cache, w.H_q, prm_g)
    pos = w.n0.astype(np.int64)
    q, kn, vn = synth.host_step(w, pos)
    dt = w.dtype
    lg.lg_begin_step(cache)
    lg.lg_append(cache, 0, w.L, lg.host_to_device(kn, device, dt), lg.host_to_device(vn, device, dt),
                 None, prm_g)
    lg.lg_decode_attend(cache, 0, w.L, lg.host_to_device(q, device, dt), w.H_q, guard.scale,
                        guard.out, guard.stats, prm_g.suffix_w, 0, guard.max_len, guard.ws)
    torch.cuda.synchronize()
    assert lg.lg_read_device_status(cache) == 0
    out = lg.device_to_host(guard.out)
    out = (out.astype(np.uint32) << 16).view(np.float32) if dt == "bf16" else out
    stats = guard.stats.cpu().numpy()
    n = w.n0 + 1
    # attention on sampled groups
    rt, ra = OUT_TOL[dt]
    for (layer, b, kvh) in _rng_groups(w, n_groups, seed):
        K = np.concatenate([synth.host_rows(w, 0, layer, kvh, b, 0, int(w.n0[b])),
                            kn[layer, b, kvh][None]])
        V = np.concatenate([synth.host_rows(w, 1, layer, kvh, b, 0, int(w.n0[b])),
                            vn[layer, b, kvh][None]])
        hs = slice(kvh * w.g, (kvh + 1) * w.g)
        o_ref, s_ref, _ = oracle.attend_group(q[layer, b, hs], K, V)
        tag = "layer %d seq %d kv-head %d" % (layer, b, kvh)
        assert_close(out[layer, b, hs], o_ref, rt, ra, tag + " out")
        assert_close(stats[layer, b, hs], s_ref, *STAT_TOL, what=tag + " stats")
    # detect on seeded statistics; every sequence
    st_seed = _seeded_stats(w, n, seed)
    guard.stats.copy_(torch.from_numpy(st_seed).to(device))
    budget_d = torch.as_tensor(w.budget.astype(np.int32), device=device)
    lg.lg_detect(cache, guard.stats, w.H_q, guard.state, budget_d, prm_g, guard.flags,
                 guard.spans, guard.diag, guard.dstate)
    lg.lg_prune_compact(cache, guard.flags, guard.spans, guard.state, budget_d, prm_g,
                        guard.kept_idx, guard.kept_count, guard.max_keep, guard.max_len)
    torch.cuda.synchronize()
    assert lg.lg_read_device_status(cache) == 0
    flags = guard.flags.cpu().numpy()
    spans = guard.spans.cpu().numpy()
    kc = guard.kept_count.cpu().numpy()
    ki = guard.kept_idx.cpu().numpy()
    pruned = 0
    for b in range(w.batch):
        nb, B = int(n[b]), int(w.budget[b])
        f, sp, dg, st = _oracle_detect(w, b, nb, B, st_seed, vn[0, b], prm_o)
        assert flags[b] == f and tuple(spans[b]) == sp, (b, flags[b], f, spans[b], sp, dg)
        kept = oracle.keep_set(nb, B, f, sp, st.level, prm_o)
        if kc[b] < 0:
            assert np.array_equal(kept, np.arange(nb)), b
            continue
        pruned += 1
        assert kc[b] == len(kept) and np.array_equal(ki[b, :len(kept)], kept), b
    # compacted bytes: sampled streams, and the sketches of every pruned sequence
    rng = np.random.default_rng(seed + 1)
    for _ in range(n_streams):
        b = int(rng.integers(w.batch))
        if kc[b] < 0:
            continue
        layer, kvh = int(rng.integers(w.L)), int(rng.integers(w.H_kv))
        kept = ki[b, :kc[b]]
        for is_v, T in ((0, cache.k), (1, cache.v)):
            ref = np.concatenate([synth.host_rows(w, is_v, layer, kvh, b, 0, int(w.n0[b])),
                                  (vn if is_v else kn)[layer, b, kvh][None]])[kept]
            o = int(w.seq_off[b])
            got = lg.device_to_host(T[layer, kvh, o:o + kc[b]])
            assert np.array_equal(got, ref), (b, layer, kvh, is_v)
    # sketches moved with their rows: first 64 and last 512 kept slots of one pruned sequence
    b = int(np.flatnonzero(kc >= 0)[0])
    kept = ki[b, :kc[b]]
    sel = np.unique(np.concatenate([np.arange(min(64, len(kept))),
                                    np.arange(max(0, len(kept) - 512), len(kept))]))
    sk_g = cache.sketch.cpu().numpy().view(np.uint32)[int(w.seq_off[b]) + sel]
    for r, j in enumerate(sel):
        pos_j = int(kept[j])
        if pos_j == int(w.n0[b]):
            row = vn[0, b]
        else:
            row = np.stack([synth.host_rows(w, 1, 0, h, b, pos_j, 1)[0] for h in range(w.H_kv)])
        assert np.array_equal(sk_g[r], oracle.sketch(np.ascontiguousarray(row))), (b, j)
    return pruned


def test_llama_decode_full_size(cuda):
    """workload 2: 32 layers, 32/8 heads, b=8, n=8192, B=4096 (8.7 GB of K/V)"""
    w = synth.make_workload(2)
    assert run_full_size(w, cuda) == w.batch          # every sequence is over budget


def test_small_model_long_context_full_size(cuda):
    """workload 3: 28 layers, 12/2 heads (GQA 6), sinks, b=32, n=32768, B=8192 (30 GB)"""
    w = synth.make_workload(3)
    assert run_full_size(w, cuda, n_groups=3) == w.batch


def test_ragged_serving_full_size(cuda):
    """workload 4: b=64, n log-uniform in [1024, 65536], B=min(n+256, 16384) (~130 GB)"""
    w = synth.make_workload(4)
    over = int(np.sum(w.n0 + 1 > w.budget))
    assert run_full_size(w, cuda, n_groups=3) >= over


def test_bandwidth_sweep_full_size(cuda):
    """workload 5: 32 layers, 64/8 heads (GQA 8), b=16, n=131072, B=32768 (275 GB)"""
    w = synth.make_workload(5)
    assert run_full_size(w, cuda, n_groups=2, n_streams=2) == w.batch


def test_paper_shaped_full_size(cuda):
    """workload 6: the paper's setting at full size (28 layers, 16/8 heads, the 3853-row prompt,
    B=1024): the first step's attention, detection on seeded statistics and the budget cut"""
    w = synth.make_workload(6)
    assert run_full_size(w, cuda, n_groups=4, n_streams=3) == w.batch


def test_llama8b_full_size_four_steps(cuda):
    """workload 2 at full size (32 layers, 32/8 heads, 8 sequences of 8192 rows, B = 4096) for
    four guarded steps through the whole path and the oracle side by side: outputs and
    statistics of every head within tolerance, the votes taken on the attention's own
    statistics, flags, spans, kept lists, guard state and every cached byte bit for bit (the
    first step triggers on the looping sequences and cuts every sequence to the budget)"""
    w = synth.make_workload(2, steps=4)
    free, _ = torch.cuda.mem_get_info(cuda)
    if free < w.kv_bytes() + (4 << 30):
        pytest.skip("needs %.1f GB of free device memory" % ((w.kv_bytes() + (4 << 30)) / 1e9))
    c = run_loopguard(w, cuda, steps=4)
    assert c["steps"] == 4 and c["triggers"] >= 1 and c["prunes"] >= w.batch, c
