"""The retained set I_keep (Sec. 5.3, Eq. 10, Eq. 11) on the GPU against the oracle over a
sweep of lengths, budgets, triggers, spans and aggressiveness levels, through both calls that
form it (lg_prune_compact, and lg_detect_prune's fused kernel is covered by the pipeline
parity tests).  K rows carry their own slot index, so the compacted cache is checked too."""
import numpy as np
import pytest
import torch

import oracle
from paper_2604_10044_gb300 import lg

pytestmark = pytest.mark.gpu


def _cases(seed, count):
    rng = np.random.default_rng(seed)
    cases = []
    for k in range(count):
        B = int(rng.choice([160, 256, 384, 512, 1000, 1024, 4096]))
        kind = k % 6
        if kind == 0:
            n = int(rng.integers(0, 40))                    # at most the anchors
        elif kind == 1:
            n = int(rng.integers(B - 8, B + 2))             # around the budget
        else:
            n = int(rng.integers(B + 1, 4 * B))
        flag = int(rng.random() < 0.6)
        R = B // 2
        lo_w = max(32, n - R)
        u = rng.random()
        if u < 0.2:
            span = (0, 0)                                   # trigger without a tail period
        elif u < 0.4:
            a = min(int(rng.integers(0, max(1, lo_w))), n)  # reaches below W^recent
            span = (a, int(rng.integers(a, n + 1)))
        elif u < 0.6:
            a = min(int(rng.integers(lo_w, max(lo_w + 1, n))), n)   # ends at n
            span = (a, n)
        else:
            a = min(int(rng.integers(lo_w, max(lo_w + 1, n))), n)
            span = (a, int(rng.integers(a, n + 1)))         # inside, may leave rows above
        level = int(rng.integers(0, 4))
        cases.append((n, B, flag, span, level))
    return cases


@pytest.mark.parametrize("seed", [0, 1])
def test_keep_set_sweep(cuda, seed):
    prm_o = oracle.params()
    prm_g = lg.lg_default_params()
    cases = _cases(seed, 96)
    b = len(cases)
    n0 = np.array([c[0] for c in cases], dtype=np.int32)
    cap = np.maximum(n0, 1)
    seq_off = np.zeros(b, dtype=np.int64)
    seq_off[1:] = np.cumsum(cap.astype(np.int64))[:-1]
    S = int(cap.sum())
    d = 128  # H_kv * d a multiple of 128 (whole 16-byte sketch chunks)
    k = torch.zeros((1, 1, S, d), dtype=torch.float32, device=cuda)
    for s in range(b):
        k[0, 0, seq_off[s]:seq_off[s] + n0[s], 0] = torch.arange(int(n0[s]), dtype=torch.float32,
                                                                 device=cuda)
    cache = lg.Cache(1, 1, d, "f32", seq_off, cap, n0, cuda, "loopguard", k=k)
    budget = torch.as_tensor(np.array([c[1] for c in cases], dtype=np.int32), device=cuda)
    flags = torch.as_tensor(np.array([c[2] for c in cases], dtype=np.int32), device=cuda)
    spans = torch.as_tensor(np.array([c[3] for c in cases], dtype=np.int32), device=cuda)
    state = torch.zeros((b, lg.STATE_BYTES // 4), dtype=torch.int32, device=cuda)
    state[:, 2] = torch.as_tensor(np.array([c[4] for c in cases], dtype=np.int32), device=cuda)
    max_keep = int(max(c[1] for c in cases))
    kept_idx = torch.full((b, max_keep), -7, dtype=torch.int32, device=cuda)
    kept_count = torch.zeros(b, dtype=torch.int32, device=cuda)
    lg.lg_prune_compact(cache, flags, spans, state, budget, prm_g, kept_idx, kept_count,
                        max_keep, int(cap.max()))
    torch.cuda.synchronize()
    assert lg.lg_read_device_status(cache) == 0
    kc = kept_count.cpu().numpy()
    ki = kept_idx.cpu().numpy()
    lens = cache.len.cpu().numpy()
    K = k[0, 0, :, 0].cpu().numpy()
    for s, (n, B, flag, span, level) in enumerate(cases):
        ref = oracle.keep_set(n, B, flag, span, level, prm_o)
        ctx = (s, n, B, flag, span, level)
        if not flag and n <= B:
            assert kc[s] == -1 and lens[s] == n, ctx
            continue
        assert kc[s] == len(ref) and lens[s] == len(ref), (ctx, kc[s], len(ref))
        assert np.array_equal(ki[s, :kc[s]], ref), ctx
        o = int(seq_off[s])
        assert np.array_equal(K[o:o + kc[s]], ref.astype(np.float32)), ctx


def test_compaction_mixed_dense_and_sparse_tiles(cuda):
    """in-place compaction (Sec. 5.3's index-gather) of whole bf16 rows with random bits, over
    kept lists that mix dense stretches (slots a few rows below their sources, a barrier every
    tile), the sparse lattice of long caches (barrier-free for many tiles) and spans of 40, 63,
    64 and 65 rows (one tile is 64 rows of 256 bytes): every retained K, V and sketch byte
    equals the oracle's gather of the original cache, bit for bit"""
    prm_o = oracle.params()
    prm_g = lg.lg_default_params()
    cases = [(131073, 32768, 0, (0, 0), 0), (131073, 32768, 1, (114689, 131073), 0),
             (8193, 4096, 0, (0, 0), 0), (5000, 4096, 1, (4900, 4940), 0),
             (5000, 4096, 1, (4800, 4863), 0), (5000, 4096, 1, (4800, 4864), 1),
             (5000, 4096, 1, (4800, 4865), 2), (4097, 4096, 0, (0, 0), 0),
             (32769, 8192, 1, (32000, 32600), 1), (20000, 16384, 1, (19000, 19990), 3),
             (3000, 1024, 1, (2990, 3000), 0), (700, 640, 0, (0, 0), 0)]
    b = len(cases)
    L, H_kv, d = 2, 2, 128
    n0 = np.array([c[0] for c in cases], dtype=np.int32)
    cap = n0 + 1
    seq_off = np.zeros(b, dtype=np.int64)
    seq_off[1:] = np.cumsum(cap.astype(np.int64))[:-1]
    S = int(cap.sum())
    g = torch.Generator(device=cuda).manual_seed(5)
    bits = lambda *shape: torch.randint(-32768, 32768, shape, dtype=torch.int32, device=cuda,
                                        generator=g)
    k = bits(L, H_kv, S, d).to(torch.int16).view(torch.bfloat16)
    v = bits(L, H_kv, S, d).to(torch.int16).view(torch.bfloat16)
    cache = lg.Cache(L, H_kv, d, "bf16", seq_off, cap, n0, cuda, "loopguard", k=k, v=v)
    cache.sketch.copy_(bits(S, H_kv * d // 32))
    K0, V0 = cache.to_host()
    SK0 = cache.sketch.cpu().numpy()
    budget = torch.as_tensor(np.array([c[1] for c in cases], dtype=np.int32), device=cuda)
    flags = torch.as_tensor(np.array([c[2] for c in cases], dtype=np.int32), device=cuda)
    spans = torch.as_tensor(np.array([c[3] for c in cases], dtype=np.int32), device=cuda)
    state = torch.zeros((b, lg.STATE_BYTES // 4), dtype=torch.int32, device=cuda)
    state[:, 2] = torch.as_tensor(np.array([c[4] for c in cases], dtype=np.int32), device=cuda)
    max_keep = int(max(c[1] for c in cases))
    kept_idx = torch.full((b, max_keep), -7, dtype=torch.int32, device=cuda)
    kept_count = torch.zeros(b, dtype=torch.int32, device=cuda)
    lg.lg_prune_compact(cache, flags, spans, state, budget, prm_g, kept_idx, kept_count,
                        max_keep, int(cap.max()))
    torch.cuda.synchronize()
    assert lg.lg_read_device_status(cache) == 0
    kc = kept_count.cpu().numpy()
    ki = kept_idx.cpu().numpy()
    K1, V1 = cache.to_host()
    SK1 = cache.sketch.cpu().numpy()
    for s, (n, B, flag, span, level) in enumerate(cases):
        ref = oracle.keep_set(n, B, flag, span, level, prm_o)
        assert kc[s] == len(ref) and np.array_equal(ki[s, :kc[s]], ref), s
        o, m = int(seq_off[s]), len(ref)
        for A0, A1 in ((K0, K1), (V0, V1)):
            want = A0[:, :, o:o + n].copy()
            for layer in range(L):
                for h in range(H_kv):
                    oracle.compact_rows(want[layer, h], ref)
            assert np.array_equal(A1[:, :, o:o + m], want[:, :, :m]), s
        want = SK0[o:o + n].copy()
        oracle.compact_rows(want, ref)
        assert np.array_equal(SK1[o:o + m], want[:m]), s
