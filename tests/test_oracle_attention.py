"""Pins of the oracle's attention and statistics (Sec. 3.1, Eq. 1) against closed forms.

Each case is built so that the result is known without running any attention code:
identical keys (uniform softmax), a two-level cache whose logits are exactly 0 or z,
constant values, and a one-hot query-to-kv-head map.  A dropped term, a wrong sign, a
transposed operand or a wrong GQA index fails at least one of them.
"""
import math

import numpy as np
import pytest

import oracle


def bf16_bits(x):
    """round-to-nearest-even float32 -> bf16 bits, independent of the generator"""
    import torch
    t = torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16)


def test_softmax_rows_sum_to_one():
    rng = np.random.default_rng(0)
    q = rng.standard_normal((4, 64)).astype(np.float32)
    K = rng.standard_normal((37, 64)).astype(np.float32)
    V = rng.standard_normal((37, 64)).astype(np.float32)
    out, stats, alpha = oracle.attend_group(q, K, V, want_alpha=True)
    assert np.all(np.abs(alpha.sum(axis=1) - 1.0) <= 1e-12)
    assert np.all(alpha > 0)
    # H in [0, ln n], S in [0, 1], l = sum exp(s - m) >= 1 (the max term is 1)
    n = 37
    assert np.all((stats[:, 2] >= 0) & (stats[:, 2] <= math.log(n) + 1e-12))
    assert np.all((stats[:, 3] >= 0) & (stats[:, 3] <= 1 + 1e-12))
    assert np.all(stats[:, 1] >= 1.0)


@pytest.mark.parametrize("n,suffix_w", [(1, 64), (5, 64), (100, 64), (100, 256), (300, 64)])
def test_identical_keys_uniform(n, suffix_w):
    """identical keys: alpha = 1/n, H = ln n, S = W_s/n with W_s = min(suffix_w, n), m = s"""
    rng = np.random.default_rng(1)
    d = 64
    k = rng.standard_normal(d).astype(np.float32)
    K = np.tile(k, (n, 1))
    V = rng.standard_normal((n, d)).astype(np.float32)
    q = rng.standard_normal((2, d)).astype(np.float32)
    out, stats, alpha = oracle.attend_group(q, K, V, suffix_w=suffix_w, want_alpha=True)
    Ws = min(suffix_w, n)
    s_expect = (q.astype(np.float64) @ k.astype(np.float64)) / 8.0
    np.testing.assert_allclose(alpha, 1.0 / n, rtol=1e-12)
    np.testing.assert_allclose(stats[:, 0], s_expect, rtol=1e-12)
    np.testing.assert_allclose(stats[:, 1], n, rtol=1e-12)
    np.testing.assert_allclose(stats[:, 2], math.log(n), rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(stats[:, 3], Ws / n, rtol=1e-12)
    # out = mean of the value rows
    np.testing.assert_allclose(out, np.tile(V.astype(np.float64).mean(0), (2, 1)), rtol=1e-10,
                               atol=1e-12)
    # suffix lift S * n / W_s = 1 for uniform attention
    np.testing.assert_allclose(stats[:, 3] * n / Ws, 1.0, rtol=1e-12)


@pytest.mark.parametrize("n,r,z", [(64, 1, 3.0), (200, 7, 2.5), (200, 7, -1.5), (513, 50, 8.0)])
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_two_level_cache_closed_form(n, r, z, dtype):
    """r hot keys with logit exactly z (the last r rows) and n - r cold keys with logit 0.

    q = 8 e_0, scale 1/8, hot keys have k_0 = z, cold keys k_0 = 0 (other components are
    random and meet a zero query component).  Closed forms with E = r e^z + n - r:
      alpha_hot = e^z / E, alpha_cold = 1 / E, H = ln E - r z e^z / E,
      S (last W_s >= r rows) = (r e^z + W_s - r) / E, m = max(z, 0), l = E e^{-m},
      out = alpha_hot * r * a + alpha_cold * (n - r) * b   (V rows a for hot, b for cold)."""
    rng = np.random.default_rng(2)
    d = 64
    K = rng.standard_normal((n, d)).astype(np.float32)
    K[:, 0] = 0.0
    K[n - r:, 0] = z
    q = np.zeros((1, d), dtype=np.float32)
    q[0, 0] = 8.0
    a = np.full(d, 0.75, dtype=np.float32)
    bv = np.full(d, -0.25, dtype=np.float32)
    V = np.tile(bv, (n, 1))
    V[n - r:] = a
    if dtype == "bf16":
        # every value above is exactly representable in bf16 except the random padding
        K, V, q = bf16_bits(K), bf16_bits(V), bf16_bits(q)
    Ws = 64
    out, stats, alpha = oracle.attend_group(q, K, V, scale=1.0 / 8.0, suffix_w=Ws,
                                            want_alpha=True)
    E = r * math.exp(z) + n - r
    m = max(z, 0.0)
    np.testing.assert_allclose(alpha[0, n - r:], math.exp(z) / E, rtol=1e-12)
    np.testing.assert_allclose(alpha[0, :n - r], 1.0 / E, rtol=1e-12)
    np.testing.assert_allclose(stats[0, 0], m, rtol=1e-15)
    np.testing.assert_allclose(stats[0, 1], E * math.exp(-m), rtol=1e-12)
    H = math.log(E) - r * z * math.exp(z) / E
    np.testing.assert_allclose(stats[0, 2], H, rtol=1e-10, atol=1e-12)
    S = (r * math.exp(z) + min(Ws, n) - r) / E
    np.testing.assert_allclose(stats[0, 3], S, rtol=1e-12)
    expect = math.exp(z) / E * r * 0.75 + 1.0 / E * (n - r) * (-0.25)
    np.testing.assert_allclose(out[0], expect, rtol=1e-10, atol=1e-12)


def test_constant_values_give_constant_output():
    rng = np.random.default_rng(3)
    q = rng.standard_normal((3, 128)).astype(np.float32)
    K = rng.standard_normal((77, 128)).astype(np.float32)
    V = np.full((77, 128), 1.375, dtype=np.float32)
    out, _, _ = oracle.attend_group(bf16_bits(q), bf16_bits(K), bf16_bits(V))
    np.testing.assert_allclose(out, 1.375, rtol=1e-13)


def test_one_hot_attention_picks_value_row():
    """one key with a logit far above the others: out is that row's value (bf16 widened)"""
    rng = np.random.default_rng(4)
    d, n = 128, 50
    K = (rng.standard_normal((n, d)) * 0.01).astype(np.float32)
    K[17, :] = 1.0
    q = np.full((1, d), 4.0, dtype=np.float32)       # logit of row 17 = 4*128/sqrt(128) = 45
    V = rng.standard_normal((n, d)).astype(np.float32)
    Vb = bf16_bits(V)
    out, stats, _ = oracle.attend_group(bf16_bits(q), bf16_bits(K), Vb)
    v17 = (Vb[17].astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    np.testing.assert_allclose(out[0], v17, rtol=1e-12, atol=1e-12)
    assert stats[0, 2] < 1e-12


def test_gqa_group_mapping_and_h2o_invariant():
    """attend_all maps query head h to kv-head h // g; with V constant per kv-head the
    outputs reveal the map.  The accumulated H2O score gains exactly g per row set."""
    import synth
    w = synth.make_workload(2, L=2, batch=2, n=96, budget=64, steps=1, H_q=6, H_kv=2,
                            tail=(40, 48), periods=(8, 8))
    rng = np.random.default_rng(5)
    K = bf16_bits(rng.standard_normal((w.L, w.H_kv, w.S_total, w.d)))
    Vf = np.zeros((w.L, w.H_kv, w.S_total, w.d), dtype=np.float32)
    for layer in range(w.L):
        for kvh in range(w.H_kv):
            Vf[layer, kvh] = 10 * layer + kvh + 0.5
    V = bf16_bits(Vf)
    q = bf16_bits(rng.standard_normal((w.L, w.batch, w.H_q, w.d)))
    g = oracle.OracleGuard(w, K, V, policy="h2o")
    out, stats = g.attend(q)
    for layer in range(w.L):
        for b in range(w.batch):
            for h in range(w.H_q):
                np.testing.assert_allclose(out[layer, b, h], 10 * layer + h // w.g + 0.5,
                                           rtol=1e-12)
    for layer in range(w.L):
        for kvh in range(w.H_kv):
            for b in range(w.batch):
                o = w.seq_off[b]
                tot = g.h2o[layer, kvh, o:o + w.n0[b]].sum()
                np.testing.assert_allclose(tot, w.g, rtol=1e-12)
