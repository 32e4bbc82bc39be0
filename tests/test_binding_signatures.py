"""The Python binding against the C declarations of include/lg.h, without a GPU: every declared
function has a wrapper of the same name in the binding, and the ctypes signature the binding
gives the shared library has exactly as many arguments as the declaration."""
import inspect
import os
import re

from paper_2604_10044_gb300 import lg

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declarations():
    """{name: number of parameters} of every LG_API function in include/lg.h"""
    src = open(os.path.join(ROOT, "include", "lg.h")).read()
    src = re.sub(r"/\*.*?\*/", " ", src, flags=re.S)
    src = re.sub(r"//[^\n]*", " ", src)
    out = {}
    for m in re.finditer(r"^LG_API [^(]*?\b(lg_\w+)\(([^)]*)\)\s*;", src, flags=re.M):
        params = m.group(2).strip()
        out[m.group(1)] = 0 if params in ("", "void") else params.count(",") + 1
    return out


def test_every_declaration_has_a_wrapper():
    decl = declarations()
    assert len(decl) == 21
    for name in decl:
        assert callable(getattr(lg, name, None)), name


def test_ctypes_signatures_match_the_header():
    L = lg.lib()
    for name, n in declarations().items():
        assert len(getattr(L, name).argtypes) == n, (name, n, getattr(L, name).argtypes)


def test_wrappers_take_the_stream_last_and_optional():
    """every wrapper of a call that takes a cudaStream_t ends with stream=None (the current
    stream when omitted)"""
    src = open(os.path.join(ROOT, "include", "lg.h")).read()
    for name in declarations():
        m = re.search(r"\b%s\(([^)]*)\)" % name, src)
        if "cudaStream_t" not in m.group(1):
            continue
        params = list(inspect.signature(getattr(lg, name)).parameters.values())
        assert params[-1].name == "stream" and params[-1].default is None, name
