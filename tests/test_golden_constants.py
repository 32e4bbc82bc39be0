"""The constants the paper prints (tests/golden/paper_constants.txt, each with its section) are
the defaults of the library (lg_default_params, lg_default_token_params), of the oracle, and
the budget and generation cap of the paper-shaped workload."""
import os

import oracle
import synth
from paper_2604_10044_gb300 import lg

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "paper_constants.txt")


def paper_constants():
    out = {}
    for line in open(GOLDEN):
        line = line.split("#", 1)[0].strip()
        if not line:
            continue
        name, value, cite = line.split(None, 2)
        assert cite.startswith(("Sec.", "App.")), line
        out[name] = float(value)
    return out


GUARD = ("W", "K", "n_anchor", "theta_ttr", "theta_nov", "stall_len", "t_min", "cooldown")
TOKEN = ("theta_cr", "theta_conf", "theta_streak")


def test_fixture_lists_every_constant_once():
    c = paper_constants()
    assert set(GUARD + TOKEN + ("budget", "T_max")) == set(c)


def test_library_defaults_are_the_papers():
    c = paper_constants()
    p = lg.lg_default_params()
    for name in GUARD:
        v = getattr(p, name)
        assert v == (c[name] if isinstance(v, float) else int(c[name])), name
    tp = lg.lg_default_token_params()
    for name in TOKEN:
        assert getattr(tp, name) == (c[name] if name != "theta_streak" else int(c[name])), name


def test_oracle_defaults_are_the_papers():
    c = paper_constants()
    p = oracle.params()
    for name in GUARD:
        assert getattr(p, name) == c[name], name
    for name in TOKEN:
        assert oracle.TOKEN_DEFAULTS[name] == c[name], name


def test_paper_shaped_workload_uses_the_papers_budget_and_cap():
    c = paper_constants()
    w = synth.make_workload(6)
    assert (w.budget == c["budget"]).all()
    assert w.steps == c["T_max"]
