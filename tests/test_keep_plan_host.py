"""The retained set the guard kernels write (keep_plan and keep_row in csrc/lg_keep.cuh, slot j
of I_keep as a function of j, Sec. 5.3, Eq. 10, Eq. 11), compiled for the host from the kernel's
own source text, against the oracle's I_keep (anchors, the sparse lattice, the tail-cleaned
recent rows, marked and collected) on a few thousand random prune events: triggered or over
budget, spans below, across and inside the recent window, every level."""
import os
import re
import shutil
import subprocess
import tempfile

import numpy as np
import pytest

import oracle

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "paper_2604_10044_gb300", "csrc", "lg_keep.cuh")
CUDA_INC = "/usr/local/cuda/include"


def _block(text, start_pat):
    m = re.search(start_pat, text, flags=re.M)
    assert m, start_pat
    i = text.index("{", m.start())
    depth = 0
    for j in range(i, len(text)):
        depth += {"{": 1, "}": -1}.get(text[j], 0)
        if depth == 0:
            end = j + 1
            if text[end:end + 1] == ";":
                end += 1
            return text[m.start():end]
    raise AssertionError("unbalanced " + start_pat)


HARNESS = r'''
#include <cstdint>
#include <cstdio>
#include "lg.h"
#define __device__
#define __forceinline__ inline
static inline int max(int a, int b) { return a > b ? a : b; }
static inline int min(int a, int b) { return a < b ? a : b; }
%(code)s
int main() {
  lg_guard_params p;
  lg_default_params_host(&p);
  int n, B, flag, lo, hi, level;
  while (std::scanf("%%d %%d %%d %%d %%d %%d", &n, &B, &flag, &lo, &hi, &level) == 6) {
    KeepPlan k;
    if (!keep_plan(n, B, flag, lo, hi, level, p, k)) { std::printf("-1\n"); continue; }
    std::printf("%%d", k.count);
    for (int j = 0; j < k.count; ++j) std::printf(" %%d", keep_row(k, j));
    std::printf("\n");
  }
  return 0;
}
'''


def _cases(rng, count):
    out = []
    while len(out) < count:
        B = int(rng.choice([64, 96, 128, 256, 1000, 1024, 2048]))
        n = int(rng.integers(1, 3 * B))
        flag = int(rng.random() < 0.6)
        if not flag and n <= B:
            continue                      # no prune: the kernel only marks the sequence
        lo = int(rng.integers(0, n + 1))
        hi = int(rng.integers(lo, n + 1))
        out.append((n, B, flag, lo, hi, int(rng.integers(0, 4))))
    return out


def test_kernel_keep_plan_matches_the_oracle():
    if shutil.which("g++") is None or not os.path.exists(os.path.join(CUDA_INC, "cuda_runtime.h")):
        pytest.skip("needs g++ and the CUDA headers")
    text = open(SRC).read()
    code = (_block(text, r"^struct KeepPlan \{") + "\n" +
            _block(text, r"^__device__ __forceinline__ bool keep_plan\(") + "\n" +
            _block(text, r"^__device__ __forceinline__ int keep_row\("))
    prm = oracle.params()
    # the library's defaults, the same values as the oracle's (pinned against the paper by
    # tests/test_golden_constants.py), for the fields keep_plan reads
    defaults = ("static void lg_default_params_host(lg_guard_params *p) {\n"
                "  *p = lg_guard_params{};\n"
                "  p->n_anchor = %d; p->headroom = %d;\n}\n" % (prm.n_anchor, prm.headroom))
    src = HARNESS % dict(code=defaults + code)
    rng = np.random.default_rng(21)
    cases = _cases(rng, 3000)
    with tempfile.TemporaryDirectory() as d:
        cpp, exe = os.path.join(d, "keep.cpp"), os.path.join(d, "keep")
        open(cpp, "w").write(src)
        subprocess.run(["g++", "-O2", "-std=c++17", "-I", os.path.join(ROOT, "include"),
                        "-I", CUDA_INC, cpp, "-o", exe], check=True)
        inp = "\n".join(" ".join(map(str, c)) for c in cases) + "\n"
        r = subprocess.run([exe], input=inp, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0
    lines = r.stdout.splitlines()
    assert len(lines) == len(cases)
    for (n, B, flag, lo, hi, level), line in zip(cases, lines):
        got = np.array(line.split()[1:], dtype=np.int64)
        want = oracle.keep_set(n, B, flag, (lo, hi), level, prm)
        assert int(line.split()[0]) == len(want), (n, B, flag, lo, hi, level)
        assert np.array_equal(got, want), (n, B, flag, lo, hi, level)
