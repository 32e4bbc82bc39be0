"""The oracle's whole decode step on the tiny single-layer workload (1 layer, 8/8 heads, d=64,
fp32, n=512, B=256, a 24-row block repeated over the last 192 positions).

Everything asserted follows from the construction, not from a previous run:
  after the append n = 513; R = B/2 = 128, so W^recent = [385, 513);
  the loop covers [320, 513), so every row of W^recent matches the row 24 earlier and the
  smallest verified period is 24; I_bad = W^recent and C_recent is empty;
  history outside W^recent is [32, 385): 353 rows > B_sparse = 256 - 64 - 32 - 64 = 96,
  so the sparse part is the lattice 32 + floor(353 j / 96), j < 96, and |I_keep| = 128.
"""
import numpy as np

import oracle
import synth


def test_tiny_guard_step():
    w = synth.make_workload(1)
    K, V = synth.host_cache(w)
    g = oracle.OracleGuard(w, K.copy(), V.copy())
    pos = w.n0.astype(np.int64)
    q, kn, vn = synth.host_step(w, pos)
    r = g.step(q, kn, vn, pos)
    assert r["flags"][0] == 1
    assert int(r["diags"][0]["P"]) == 24
    assert tuple(r["spans"][0]) == (385, 513)
    expect = np.concatenate([np.arange(32), 32 + (np.arange(96) * 353) // 96])
    assert np.array_equal(r["kept"][0], expect)
    assert r["len"][0] == 128
    # the compacted cache is the ordered gather of the appended cache
    full = np.concatenate([K[0, :, :512], kn[0, 0][:, None, :]], axis=1)
    assert np.array_equal(g.K[0, :, :128], full[:, expect])
    assert g.state[0].cd == 32 and g.state[0].n_int == 1 and g.state[0].t_gen == 65
