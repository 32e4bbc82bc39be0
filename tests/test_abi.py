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
    assert len(names) == 20
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
