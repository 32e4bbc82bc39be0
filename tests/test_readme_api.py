"""The decode-loop example in README.md names only functions and Guard/Cache attributes that the
Python binding has, with the binding's argument counts (checked without a GPU)."""
import inspect
import os
import re

from paper_2604_10044_gb300 import lg

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _example():
    text = open(os.path.join(ROOT, "README.md")).read()
    blocks = re.findall(r"```python\n(.*?)```", text, flags=re.S)
    assert blocks, "README has no python example"
    return blocks[0]


def _calls(src):
    """(name, number of positional arguments) of every lg.<function>(...) call"""
    out = []
    for m in re.finditer(r"\blg\.(\w+)\(", src):
        depth, i, args, start = 1, m.end(), 0, m.end()
        while depth:
            ch = src[i]
            if ch in "([{":
                depth += 1
            elif ch in ")]}":
                depth -= 1
            elif ch == "," and depth == 1:
                args += 1
            i += 1
        body = src[start:i - 1].strip()
        out.append((m.group(1), args + 1 if body else 0, body))
    return out


def test_readme_calls_exist_with_their_arity():
    for name, nargs, body in _calls(_example()):
        fn = getattr(lg, name)
        if inspect.isclass(fn):
            continue
        params = inspect.signature(fn).parameters.values()
        required = sum(p.default is inspect.Parameter.empty for p in params)
        n_kw = body.count("=") - body.count("==")
        assert required <= nargs <= len(params), (name, nargs, required)
        assert nargs - n_kw <= len(params), name


def test_readme_guard_attributes_exist():
    src = _example()
    used = set(re.findall(r"\bg\.(\w+)", src))
    guard_src = inspect.getsource(lg.Guard)
    for a in used:
        assert re.search(r"self\.%s\b" % a, guard_src), a
