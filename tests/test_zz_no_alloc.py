"""lg_decode_attend_noalloc, the attend entry point for callers that cannot allocate device
memory (a plugin inside a framework that owns all device allocations, or a loop that cannot
take cudaMalloc's implicit synchronisation).  Its scratch is a static array of the library.

Checked through the C ABI on two calls in a row (the second reuses the array the first left
behind), within the parity tests' tolerances, against both the CPU oracle (attention, Eq. 1,
with its statistics) and lg_decode_attend with a caller workspace:
  - the bf16 tensor-core path (GQA 4, three layers in one call);
  - the fp32 path at head_dim 64 (a partial kernel and a merge kernel, both on the array);
  - the H2O accumulation (the logits kept in the array between the pass and the score
    update): accumulated scores within 1e-4 relative of the oracle's after each call.
This file is collected last so that a run stopping at the first failure has run every other
test first; it also passes alone in a fresh process.
"""
import numpy as np
import pytest
import torch

import oracle
import synth
from paper_2604_10044_gb300 import lg

from parity_util import OUT_TOL, STAT_TOL, assert_close

pytestmark = pytest.mark.gpu

H2O_TOL = (1e-4, 1e-6)   # accumulated H2O scores (fp32 sums of attention weights)


def _two_calls(w, cuda, policy, accumulate_h2o):
    """two attention calls with different queries through both entry points; each result is
    compared with the oracle, and the no-alloc one with the workspace one"""
    K, V = synth.host_cache(w)
    ref = oracle.OracleGuard(w, K.copy(), V.copy(), policy=policy)
    cache_a = lg.Cache.from_host(w, K, V, cuda, policy=policy)   # workspace call
    cache_b = lg.Cache.from_host(w, K, V, cuda, policy=policy)   # no-alloc call
    max_len = int(w.n0.max())
    ws_bytes = lg.lg_workspace_size(cache_a, w.H_q, w.L, max_len, accumulate_h2o)
    assert 0 < ws_bytes <= lg.NOALLOC_SCRATCH_BYTES
    ws = torch.empty(ws_bytes // 4 + 64, dtype=torch.float32, device=cuda)
    tdt = torch.bfloat16 if w.dtype == "bf16" else torch.float32
    scale = 1.0 / np.sqrt(w.d)
    rt, ra = OUT_TOL[w.dtype]
    for k in range(2):
        q, _, _ = synth.host_step(w, w.n0.astype(np.int64) + k)
        qd = lg.host_to_device(q, cuda, w.dtype)
        out_a = torch.zeros((w.L, w.batch, w.H_q, w.d), dtype=tdt, device=cuda)
        st_a = torch.zeros((w.L, w.batch, w.H_q, 4), dtype=torch.float32, device=cuda)
        out_b, st_b = torch.full_like(out_a, 7.0), torch.full_like(st_a, 7.0)
        lg.lg_decode_attend(cache_a, 0, w.L, qd, w.H_q, scale, out_a, st_a, 64, accumulate_h2o,
                            max_len, ws)
        lg.lg_decode_attend_noalloc(cache_b, 0, w.L, qd, w.H_q, scale, out_b, st_b, 64,
                                    accumulate_h2o, max_len)
        torch.cuda.synchronize()
        assert lg.lg_read_device_status(cache_a) == 0 and lg.lg_read_device_status(cache_b) == 0
        out_ref, st_ref = ref.attend(q)
        tag = "%s call %d" % (w.name, k)
        got_b = out_b.float().cpu().numpy()
        assert_close(got_b, out_ref, rt, ra, tag + " out vs oracle")
        assert_close(st_b.cpu().numpy(), st_ref, *STAT_TOL, what=tag + " stats vs oracle")
        assert_close(got_b, out_a.float().cpu().numpy(), rt, ra, tag + " out vs workspace call")
        assert_close(st_b.cpu().numpy(), st_a.cpu().numpy(), *STAT_TOL,
                     what=tag + " stats vs workspace call")
        if accumulate_h2o:
            sb = cache_b.h2o.cpu().numpy()
            sa = cache_a.h2o.cpu().numpy()
            for b in range(w.batch):
                o, n = int(w.seq_off[b]), int(w.n0[b])
                assert_close(sb[:, :, o:o + n], ref.h2o[:, :, o:o + n], *H2O_TOL,
                             what=tag + " H2O scores vs oracle, seq %d" % b)
                assert_close(sb[:, :, o:o + n], sa[:, :, o:o + n], *H2O_TOL,
                             what=tag + " H2O scores vs workspace call, seq %d" % b)


def test_noalloc_bf16_twice(cuda):
    w = synth.make_workload(2, L=3, batch=3, n=1500, budget=1024, steps=2, tail=(300, 400),
                            periods=(10, 30))
    _two_calls(w, cuda, "loopguard", 0)


def test_noalloc_fp32_head_dim_64_twice(cuda):
    w = synth.make_workload(1, n=700, loop_len=192, budget=512)
    _two_calls(w, cuda, "loopguard", 0)


def test_noalloc_h2o_accumulation_twice(cuda):
    w = synth.make_workload(2, L=2, batch=2, n=1200, budget=1024, steps=2, tail=(200, 300),
                            periods=(10, 30), H_kv=2, H_q=8)
    _two_calls(w, cuda, "h2o", 1)


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
