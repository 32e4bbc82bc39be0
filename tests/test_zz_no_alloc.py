"""lg_decode_attend_noalloc, the attend entry point for callers that cannot allocate device
memory (a plugin inside a framework that owns all device allocations, or a loop that cannot
take cudaMalloc's implicit synchronisation).  Its scratch is a static array of the library.

Checked through the C ABI against lg_decode_attend with a caller workspace, on two calls in a
row (the second reuses the array the first left behind), within the parity tests' tolerances.
This file is collected last so that a run stopping at the first failure has run every other
test first; it also passes alone in a fresh process.
"""
import numpy as np
import pytest
import torch

import synth
from paper_2604_10044_gb300 import lg

pytestmark = pytest.mark.gpu

OUT_RTOL, OUT_ATOL = 2e-2, 1e-3     # bf16 attention output
STAT_RTOL, STAT_ATOL = 1e-4, 1e-6   # fp32 statistics


def _close(a, b, rtol, atol):
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    return bool(np.all(np.abs(a - b) <= atol + rtol * np.abs(b)))


def test_noalloc_matches_workspace_call_twice(cuda):
    w = synth.make_workload(2, L=3, batch=3, n=1500, budget=1024, steps=2, tail=(300, 400),
                            periods=(10, 30))
    K, V = synth.host_cache(w)
    cache = lg.Cache.from_host(w, K, V, cuda)
    max_len = int(w.n0.max())
    qs = []
    for k in range(2):
        q, _, _ = synth.host_step(w, w.n0.astype(np.int64) + k)
        qs.append(lg.host_to_device(q, cuda, w.dtype))
    ws_bytes = lg.lg_workspace_size(cache, w.H_q, w.L, max_len, 0)
    assert 0 < ws_bytes <= lg.NOALLOC_SCRATCH_BYTES
    ws = torch.empty(ws_bytes // 4 + 64, dtype=torch.float32, device=cuda)
    scale = 1.0 / np.sqrt(w.d)
    for k in range(2):
        out_a = torch.zeros((w.L, w.batch, w.H_q, w.d), dtype=torch.bfloat16, device=cuda)
        st_a = torch.zeros((w.L, w.batch, w.H_q, 4), dtype=torch.float32, device=cuda)
        out_b, st_b = torch.zeros_like(out_a), torch.zeros_like(st_a)
        lg.lg_decode_attend(cache, 0, w.L, qs[k], w.H_q, scale, out_a, st_a, 64, 0, max_len, ws)
        lg.lg_decode_attend_noalloc(cache, 0, w.L, qs[k], w.H_q, scale, out_b, st_b, 64, 0,
                                    max_len)
        torch.cuda.synchronize()
        assert lg.lg_read_device_status(cache) == 0
        assert _close(out_b.float().cpu(), out_a.float().cpu(), OUT_RTOL, OUT_ATOL), k
        assert _close(st_b.cpu(), st_a.cpu(), STAT_RTOL, STAT_ATOL), k


def test_noalloc_rejects_oversized_request(cuda):
    """a call whose workspace exceeds the static scratch returns LG_ERR_WORKSPACE"""
    w = synth.make_workload(2, L=1, batch=1, n=64, budget=64, steps=1)
    K, V = synth.host_cache(w)
    cache = lg.Cache.from_host(w, K, V, cuda)
    big = 1 << 24   # max_len so large that the split-K partials exceed 32 MiB
    assert lg.lg_workspace_size(cache, w.H_q, 1, big, 0) > lg.NOALLOC_SCRATCH_BYTES
    q = torch.zeros((1, 1, w.H_q, w.d), dtype=torch.bfloat16, device=cuda)
    out = torch.zeros_like(q)
    st = torch.zeros((1, 1, w.H_q, 4), dtype=torch.float32, device=cuda)
    with pytest.raises(lg.LgError) as e:
        lg.lg_decode_attend_noalloc(cache, 0, 1, q, w.H_q, 0.1, out, st, 64, 0, big)
    assert e.value.code == 6
