"""The detect kernel's vote helpers (paper_2604_10044_gb300/csrc/lg_votes.cuh), compiled from the
same source for the host, agree with the fp64 quotient decisions they stand for
(tests/vote_helpers_check.cpp): every count of windows of up to 300 rows against thresholds on,
next to and between the quotients, and sums on both sides of each bound."""
import os
import shutil
import subprocess
import tempfile

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _cuda_include():
    for d in (os.environ.get("CUDA_HOME", ""), "/usr/local/cuda"):
        if d and os.path.exists(os.path.join(d, "include", "vector_types.h")):
            return os.path.join(d, "include")
    return None


def test_vote_helpers_match_the_quotients():
    inc = _cuda_include()
    if shutil.which("g++") is None or inc is None:
        pytest.skip("needs g++ and the CUDA headers")
    with tempfile.TemporaryDirectory() as d:
        exe = os.path.join(d, "vote_check")
        subprocess.run(["g++", "-O2", "-std=c++17", "-ffp-contract=off",
                        "-I", os.path.join(ROOT, "paper_2604_10044_gb300", "csrc"), "-I", inc,
                        os.path.join(ROOT, "tests", "vote_helpers_check.cpp"), "-o", exe],
                       check=True)
        r = subprocess.run([exe], capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stdout
    assert "mismatches 0" in r.stdout
