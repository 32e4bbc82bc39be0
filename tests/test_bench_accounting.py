"""The algorithmic byte counts behind bench.py's bandwidth and roofline figures, on the CPU:
attention bytes against the K+V size of the Llama-3-8B-shaped workload (8193 rows of 32
layers x 8 kv-heads x d = 128 in bf16, K and V: 8.59 GB per step), compaction bytes against
hand-counted moved rows, and the committed DRAM-traffic summary's gate on the kernel source."""
import json
import os

import numpy as np

import bench
import synth


def test_attend_bytes_match_the_cache_size():
    w = synth.make_workload(2)
    n_rows = np.full(w.batch, 8193)
    kv = 8 * 8193 * 32 * 8 * 2 * 128 * 2           # sequences x rows x layers x heads x K,V x d x bf16
    qo = 2 * 32 * 8 * 32 * 128 * 2 + 32 * 8 * 32 * 16  # q in, out back (bf16), {m, l, H, S} fp32
    assert bench.attend_bytes(w, n_rows) == kv + qo
    assert abs(kv / 1e9 - 8.59) < 0.01
    # the H2O path adds the logits (written and read back, 4 bytes per query head) and the
    # score read-modify-write (8 bytes) per (layer, kv-head, row)
    rows = 32 * 8 * 8 * 8193
    assert bench.attend_bytes(w, n_rows, h2o=True) == kv + qo + (8 * w.g + 8) * rows


def test_compact_bytes_count_moved_rows_only():
    w = synth.make_workload(2, L=2, batch=3, n=64, budget=64, steps=1, tail=(16, 32),
                            periods=(4, 8))
    kept_idx = np.zeros((3, 10), dtype=np.int32)
    kept_count = np.array([-1, 6, 4], dtype=np.int32)
    kept_idx[1, :6] = [0, 1, 2, 5, 7, 9]     # slots 3, 4, 5 take rows 5, 7, 9: three moved rows
    kept_idx[2, :4] = [0, 1, 2, 3]           # nothing moves
    row = 2 * w.L * w.H_kv * w.d * 2 + w.H_kv * w.d // 8  # K and V of every layer, plus the sketch
    assert bench.compact_bytes(w, kept_count, kept_idx) == 2 * 3 * row


def test_traffic_summary_is_gated_on_the_kernel_source():
    assert bench.traffic_from_profile("0" * 64) is None
    path = os.path.join(bench.ROOT, "profiles", "attend_mma_traffic.txt")
    with open(path) as f:
        d = json.load(f)
    # a full-size launch reads each K/V row once: its DRAM bytes are its algorithmic bytes
    # less at most what L2 can hold of the previous pass (129 MB), plus the partials written
    assert d["alg_bytes"] - 129e6 <= d["dram_bytes"] <= 1.02 * d["alg_bytes"]
    assert d["dram_bytes"] == d["dram_bytes_read"] + d["dram_bytes_write"]
    # the algorithmic bytes of the captured launch, as bench.py counts them
    w = synth.make_workload(d["workload"])
    assert w.batch == d["batch"] and d["rows"] % (w.L * w.H_kv) == 0
    qo = bench.attend_bytes(w, np.zeros(w.batch, dtype=np.int64))
    assert d["alg_bytes"] == qo + 2 * w.d * w.esize * d["rows"]
    got = bench.traffic_from_profile(d["source_sha256"])
    assert got is not None and got["dram_bytes"] == d["dram_bytes"]


def test_traffic_gate_ignores_comments_not_code():
    src = 'int a = 1;  // rows\n/* chunks\n   per CTA */\nconst char *s = "// kept";\n'
    same = 'int a = 1;\nconst char *s = "// kept";  /* a new comment */\n'
    assert bench.code_only(src) == bench.code_only(same)
    assert bench.code_only(src) != bench.code_only(src.replace("a = 1", "a = 2"))
    assert '"// kept"' in bench.code_only(src)
