"""CPU-side checks of the C ABI library: it loads without a GPU, exports every function
include/lg.h declares, fills the default parameters and rejects bad arguments on the host
before launching anything."""
import ctypes
import os
import re

import pytest

from paper_2604_10044_gb300 import lg

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared():
    src = open(os.path.join(ROOT, "include", "lg.h")).read()
    return sorted(set(re.findall(r"^LG_API [^(]*?\b(lg_\w+)\(", src, flags=re.M)))


def test_every_declared_symbol_is_exported():
    names = declared()
    assert len(names) == 21
    assert sorted(lg.exported_symbols()) == names
    L = lg.lib()
    for n in names:
        assert hasattr(L, n), n


def test_defaults_and_status_strings():
    p = lg.lg_default_params()
    assert (p.W, p.K, p.t_min, p.cooldown, p.n_anchor, p.stall_len) == (256, 2, 64, 32, 32, 4)
    assert p.theta_ttr == 0.2 and p.theta_nov == 0.02
    assert lg.lg_status_string(0) == "ok"
    assert "budget" in lg.lg_status_string(7)


def test_host_validation_rejects_before_launch():
    """null cache pointers and unsupported shapes are refused on the host (no GPU touched)"""
    c = lg.LgCache()
    L = lg.lib()
    assert L.lg_begin_step(ctypes.byref(c), None) == 1
    # fake non-null, aligned device pointers: validation stops on the head_dim first
    fake = 1 << 20
    c = lg.LgCache(k=fake, v=fake, dtype=0, L=1, H_kv=8, d=96, batch=1, S_total=10, seq_off=fake,
                   cap=fake, len=fake, sketch=fake, dev_status=fake)
    assert L.lg_begin_step(ctypes.byref(c), None) == 2
    c.d = 128
    c.k = fake + 8                                   # misaligned cache pointer
    assert L.lg_begin_step(ctypes.byref(c), None) == 1
    c.k = fake
    p = lg.lg_default_params()
    # GQA group of 9 is unsupported; workspace missing is reported before any launch
    assert L.lg_decode_attend(ctypes.byref(c), 0, 1, fake, 72, 0.1, fake, fake, 64, 0, 10,
                              None, 0, None) == 2
    assert L.lg_decode_attend(ctypes.byref(c), 0, 1, fake, 32, 0.1, fake, fake, 64, 0, 10,
                              None, 0, None) == 6
    assert L.lg_decode_attend(ctypes.byref(c), 0, 2, fake, 32, 0.1, fake, fake, 64, 0, 10,
                              fake, 1 << 30, None) == 1   # layers out of range
    p.p_max = 0
    assert L.lg_detect(ctypes.byref(c), fake, 32, fake, fake, ctypes.byref(p), fake, fake,
                       None, fake, None) == 1
    p.p_max = 128
    assert L.lg_detect_state_size(ctypes.byref(c), ctypes.byref(p)) == 4 * (130 + c.S_total)
    ws = L.lg_workspace_size(ctypes.byref(c), 32, 1, 1000, 0)
    assert ws > 0 and ws % 256 == 0


def test_every_status_code_has_its_own_message():
    """each lg_status value lg.h declares maps to a distinct message; anything else is unknown"""
    src = open(os.path.join(ROOT, "include", "lg.h")).read()
    block = src[src.index("typedef enum {"):src.index("} lg_status;")]
    codes = [int(v) for v in re.findall(r"LG_\w+ = (\d+)", block)]
    assert codes == list(range(len(codes)))
    msgs = [lg.lg_status_string(c) for c in codes]
    assert len(set(msgs)) == len(codes) and "unknown status" not in msgs
    assert lg.lg_status_string(len(codes)) == "unknown status"
    assert lg.lg_status_string(-1) == "unknown status"


def _fake_cache(**over):
    fake = 1 << 20
    c = lg.LgCache(k=fake, v=fake, dtype=0, L=2, H_kv=8, d=128, batch=1, S_total=64,
                   seq_off=fake, cap=fake, len=fake, sketch=fake, dev_status=fake)
    for k, v in over.items():
        setattr(c, k, v)
    return c


def test_each_call_validates_its_arguments_on_the_host():
    """every refusal below happens before any launch (the pointers are never dereferenced on the
    host, and no GPU is present): the code returned is the one lg.h documents"""
    L = lg.lib()
    F = 1 << 20
    p = lg.lg_default_params()
    tp = lg.lg_default_token_params()
    c = _fake_cache()
    by = ctypes.byref
    cases = [
        # the cache itself
        ("dtype", lambda: L.lg_begin_step(by(_fake_cache(dtype=5)), None), 2),
        ("sketch rows of whole chunks", lambda: L.lg_begin_step(by(_fake_cache(H_kv=1, d=64)), None), 2),
        ("h2o without pos", lambda: L.lg_begin_step(by(_fake_cache(h2o=F)), None), 1),
        ("no sequences", lambda: L.lg_begin_step(by(_fake_cache(batch=0)), None), 1),
        # lg_append
        ("append layer range", lambda: L.lg_append(by(c), 1, 2, F, F, None, by(p), None), 1),
        ("append misaligned rows", lambda: L.lg_append(by(c), 0, 1, F + 4, F, None, by(p), None), 1),
        ("append positions", lambda: L.lg_append(by(_fake_cache(h2o=F, pos=F)), 0, 1, F, F, None,
                                                 by(p), None), 1),
        # lg_decode_attend
        ("H_q not a multiple", lambda: L.lg_decode_attend(by(c), 0, 1, F, 30, 0.1, F, F, 64, 0,
                                                          10, F, 1 << 30, None), 1),
        ("suffix width", lambda: L.lg_decode_attend(by(c), 0, 1, F, 32, 0.1, F, F, 0, 0, 10, F,
                                                    1 << 30, None), 1),
        ("scale NaN", lambda: L.lg_decode_attend(by(c), 0, 1, F, 32, float("nan"), F, F, 64, 0,
                                                 10, F, 1 << 30, None), 1),
        ("scale 0", lambda: L.lg_decode_attend(by(c), 0, 1, F, 32, 0.0, F, F, 64, 0, 10, F,
                                               1 << 30, None), 1),
        ("h2o scores missing", lambda: L.lg_decode_attend(by(c), 0, 1, F, 32, 0.1, F, F, 64, 1,
                                                          10, F, 1 << 30, None), 1),
        ("workspace alignment", lambda: L.lg_decode_attend(by(c), 0, 1, F, 32, 0.1, F, F, 64, 0,
                                                           10, F + 16, 1 << 30, None), 6),
        ("stats alignment", lambda: L.lg_decode_attend(by(c), 0, 1, F, 32, 0.1, F, F + 4, 64, 0,
                                                       10, F, 1 << 30, None), 1),
    ]
    for name, over in (("tau_ham", dict(tau_ham=1.5)), ("W", dict(W=0)), ("K", dict(K=4)),
                       ("periods", dict(p_min=5, p_max=4)), ("level_max", dict(level_max=31))):
        bad = lg.lg_default_params(**over)
        cases.append(("params " + name,
                      lambda bad=bad: L.lg_detect(by(c), F, 32, F, F, by(bad), F, F, None, F,
                                                  None), 1))
    wide = lg.lg_default_params(W=4000, p_max=128)
    cases += [
        ("detect H_q", lambda: L.lg_detect(by(c), F, 30, F, F, by(p), F, F, None, F, None), 1),
        ("detect state alignment", lambda: L.lg_detect(by(c), F, 32, F + 8, F, by(p), F, F, None,
                                                       F, None), 1),
        ("detect window beyond shared memory", lambda: L.lg_detect(by(c), F, 32, F, F, by(wide),
                                                                   F, F, None, F, None), 2),
        ("detect_prune kept list", lambda: L.lg_detect_prune(by(c), F, 32, F, F, by(p), F, F,
                                                             None, F, None, F, 10, 10, None), 1),
        ("prune_compact max_keep", lambda: L.lg_prune_compact(by(c), F, F, F, F, by(p), F, F, 0,
                                                              10, None), 1),
        ("prune_compact flags without spans", lambda: L.lg_prune_compact(by(c), F, None, F, F,
                                                                         by(p), F, F, 10, 10,
                                                                         None), 1),
        ("token state alignment", lambda: L.lg_token_detect(by(c), F, F, None, None, 0, F + 8,
                                                            by(p), by(tp), F, F, None, F, None),
         1),
        ("token kept lists paired", lambda: L.lg_token_detect(by(c), F, F, F, None, 4, F, by(p),
                                                              by(tp), F, F, None, F, None), 1),
        ("token_prune kept lists", lambda: L.lg_token_detect_prune(by(c), F, F, F, F, by(p),
                                                                   by(tp), F, F, None, F, None,
                                                                   F, 10, 10, None), 1),
        ("token_prune budget", lambda: L.lg_token_detect_prune(by(c), F, F, F, None, by(p),
                                                               by(tp), F, F, None, F, F, F, 10,
                                                               10, None), 1),
        ("token_prune max_keep", lambda: L.lg_token_detect_prune(by(c), F, F, F, F, by(p), by(tp),
                                                                 F, F, None, F, F, F, 0, 10,
                                                                 None), 1),
        ("h2o evict without scores", lambda: L.lg_h2o_evict(by(c), F, F, 10, None), 1),
        ("streaming sinks", lambda: L.lg_streaming_evict(by(_fake_cache(h2o=F, pos=F)), F, F, -1,
                                                         10, None), 1),
        ("status without a host word", lambda: L.lg_read_device_status(by(c), None, None), 1),
    ]
    bad_tp = lg.lg_default_token_params(cr_every=0)
    cases.append(("token params", lambda: L.lg_token_detect(by(c), F, F, None, None, 0, F, by(p),
                                                            by(bad_tp), F, F, None, F, None), 1))
    for name, call, code in cases:
        assert call() == code, name
