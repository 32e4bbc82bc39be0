"""bench.py end to end on a small case: one JSON line with every key of the measurement
contract (metric, value, unit, steps, warm-up, ms_per_step, the roofline object with its bound,
achieved rate, peak, fraction and traffic, the end-to-end object with the bytes it copies, the
SM clocks seen during the timed region, the launches counted), and the reference arm's line on
the same config."""
import json
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _line(*args):
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), *args], cwd=ROOT,
                       capture_output=True, text=True, timeout=900)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, r.stdout[-2000:]
    return json.loads(lines[0])


def test_bench_line_keeps_the_contract():
    args = ["--workload", "2", "--batch", "2", "--steps", "6", "--warmup", "3"]
    d = _line(*args, "--no-cpu-baseline")
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
              "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config", "roofline",
              "e2e", "clocks", "gpu_launches"):
        assert k in d, k
    assert d["n_gpus"] == 1 and d["steps"] == 6 and d["warmup"] == 3
    assert d["value"] > 0 and d["ms_per_step"] > 0 and d["higher_is_better"] is True
    assert d["scaling"] == "weak" and d["dtype"] == "bf16" and d["vs_baseline"] is None
    assert d["config"]["workload"].startswith("Llama-3-8B")
    r = d["roofline"]
    assert r["bound"] == "hbm" and r["unit"] == "GB/s"
    assert r["achieved"] > 0 and r["peak"] > 0 and abs(r["frac"] - r["achieved"] / r["peak"]) < 1e-3
    assert "traffic" in r and 0 < r["frac_of_read_peak"] < 2
    e = d["e2e"]
    assert e["value"] > 0 and e["h2d_bytes_per_step"] > 0 and e["d2h_bytes_per_step"] > 0
    c = d["clocks"]
    assert c["sm_mhz"] > 0 and c["sm_max_mhz"] > 0 and isinstance(c["reasons"], list)
    # six library launches and one harness launch a step on this path
    assert d["gpu_launches"] == 7 * 6


@pytest.mark.parametrize("extra", [["--detector", "kv"], ["--detector", "token"],
                                   ["--fresh-each-step"]])
def test_reference_line_is_on_the_same_config(extra):
    """the reference arm times the GPU arm's batch (--batch), detector (--detector) and steps
    (--fresh-each-step)"""
    args = ["--workload", "2", "--batch", "2", "--steps", "4", "--warmup", "3", *extra]
    d = _line(*args, "--no-cpu-baseline")
    r = _line(*args, "--impl", "reference")
    assert r["impl"] == "reference" and r["metric"] == d["metric"] and r["unit"] == d["unit"]
    assert r["config"] == d["config"] and r["higher_is_better"] is True
    assert r["value"] > 0 and r["cpu_baseline"]["kind"] == "oracle"
    assert r["e2e"]["h2d_bytes_per_step"] == 0 and r["e2e"]["d2h_bytes_per_step"] == 0
    assert "of 2" in r["cpu_baseline"]["sample"]   # sequence 0 of the GPU arm's 2
    assert ("each from a fresh cache" in r["cpu_baseline"]["sample"]) == \
        ("--fresh-each-step" in extra)
