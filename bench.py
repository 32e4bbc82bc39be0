#!/usr/bin/env python3
"""Benchmark of the LoopGuard decode path on GB300: guarded decode steps/s.

Workload (default): the bandwidth sweep, the largest of the five -- 32 layers, 64 query / 8 KV
heads, head_dim 128, bf16, 16 sequences of 131072 cached tokens (275 GB of K/V), budget 32768,
half the sequences carrying a planted period-32 tail of 16384 tokens.  Synthetic seeded inputs
(the paper's LoopBench prompts and model weights are not available); every step reads tens of
GB of K/V, far more than the 129 MB L2.  --workload 1..6 selects the others (2 = the
Llama-3-8B-shaped decode batch, 6 = the paper's own setting).

One step = one guarded decode step of the whole batch through the C ABI, every kernel of
the path included: reserve the slot, append the new K/V rows of all layers (+ sketch),
decode attention over the cache fused with the per-head statistics (Eq. 1), the loop-onset
test (Eq. 8, Eq. 9), the retained set and in-place compaction (Eq. 10, Eq. 11).  A harness
kernel selects each sequence's next inputs (loop continuation, or loop-free after the guard
intervened) from buffers generated before timing.  The timed steps start from the freshly
generated cache, so step 1 carries the budget event of every sequence (131073 -> 32704 rows
on the default workload) and the later steps read the retained rows.

Prints one JSON line.  --impl reference times the CPU oracle instead, on a bounded sample of
the same timed run (the same sample as the GPU line's cpu_baseline).
"""
import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import synth  # noqa: E402

METRIC = "guarded decode steps/s (attend+stats, detect, prune/compact) and achieved HBM GB/s"
UNIT = "steps/s"
L2_BYTES = 129e6
EV_EVERY = 8  # timing events on every 8th timed step,
EV_SAMPLES = 40  # or on about 40 steps of a longer run (each sampled step loses its overlap)
DEFAULT_STEPS = 400
DEFAULT_STEPS_W5 = 20   # about 0.25 s of GPU time from the fresh 275 GB cache
ORACLE_TARGET_S = 20.0  # CPU seconds the oracle's timed sample may take, about (a cap)
# (row, kv-head) reads of the oracle's sample over its K steps: the sampled layer count follows
# from the workload and K alone, so both oracle figures time the same sample (about 11 s on the
# 16 Grace cores at the default line: 10 of 32 layers of sequence 0)
ORACLE_SAMPLE_ROW_HEADS = 6.0e7


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=0,
                    help="timed steps (default: %d on the bandwidth sweep, %d on the others)"
                         % (DEFAULT_STEPS_W5, DEFAULT_STEPS))
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    ap.add_argument("--workload", type=int, default=5)
    ap.add_argument("--layers-per-call", type=int, default=0,
                    help="layers per lg_decode_attend call (0 = all layers in one call)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-clocks", action="store_true")
    ap.add_argument("--batch", type=int, default=0,
                    help="override the workload's batch (smaller cases for profiling)")
    ap.add_argument("--policy", default="loopguard",
                    choices=["loopguard", "h2o", "streaming", "full"],
                    help="cache policy of the timed steps: LoopGuard, or a comparator on the "
                         "same inputs: H2O (accumulated-score eviction), StreamingLLM "
                         "(attention sinks + sliding window) or the full cache (no eviction)")
    ap.add_argument("--fresh-each-step", action="store_true",
                    help="time every step from a freshly generated cache (the first decode "
                         "step: attention over the full prefill and the budget prune)")
    ap.add_argument("--detector", default="kv", choices=["kv", "token"],
                    help="loop-onset test of the LoopGuard policy: over attention statistics and "
                         "V-row sketches (lg_detect_prune), or over the generated token ids and "
                         "top-1 probabilities (lg_token_detect_prune)")
    ap.add_argument("--ablation", action="store_true",
                    help="run the synthetic analog of the paper's ablation (no guard, always-on "
                         "pruning, the confidence streak alone, the full guard) on the GPU path and "
                         "print its measures instead of the step benchmark")
    ap.add_argument("--eager", action="store_true",
                    help="time the steps as eager launches instead of one CUDA graph replay")
    ap.add_argument("--oracle-one-thread", action="store_true", help=argparse.SUPPRESS)
    ap.add_argument("--profile-steps", type=int, default=0,
                    help="run this many steps untimed and exit (for ncu launch lists)")
    args = ap.parse_args()
    if not args.steps:
        args.steps = DEFAULT_STEPS_W5 if args.workload == 5 else DEFAULT_STEPS
    return args


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


def read_peak(dev, gib=4, reps=10):
    """read-only HBM bandwidth of this GPU, measured in this run: three read-only passes over
    gib GiB (synth: 16-byte evict-first loads from registers; 1-D bulk copies of 16 KB into
    shared memory, 3 CTAs per SM; of 32 KB, one CTA per SM), each the best of `reps` timed
    passes alternating between two such buffers (so that no pass starts on rows the previous
    one left in L2), CUDA events on the launching stream.  Returns (best GB/s, {probe: GB/s})."""
    import torch
    n = gib << 30
    bufs = [torch.zeros(n, dtype=torch.uint8, device=dev) for _ in range(2)]
    sink = torch.zeros(1, dtype=torch.int32, device=dev)
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    st = torch.cuda.current_stream(dev)
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    probes = {
        "loads_16B": lambda buf: synth.dev_read_stream(buf, sink, 4 * sms, st.cuda_stream),
        "bulk_16KB": lambda buf: synth.dev_read_bulk(buf, 16384, sink, err, 3 * sms,
                                                     st.cuda_stream),
        "bulk_32KB": lambda buf: synth.dev_read_bulk(buf, 32768, sink, err, sms,
                                                     st.cuda_stream)}
    res = {}
    for name, run in probes.items():
        run(bufs[1])  # warm-up (loads the kernel)
        best = float("inf")
        for r in range(reps):
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(st)
            run(bufs[r % 2])
            b.record(st)
            b.synchronize()
            best = min(best, a.elapsed_time(b))
        res[name] = round(n / (best * 1e-3) / 1e9, 1)
    if int(err.item()):
        raise RuntimeError("a read-bandwidth probe timed out on a wait")
    del bufs
    torch.cuda.empty_cache()
    return max(res.values()), res


def l2_note(w):
    """the K/V bytes a step reads against the 129 MB L2, from the workload's shape alone (the
    same words in both arms): the first step reads every cached row; once the cache is within
    budget a step reads at least the anchors and the sparse lattice of each sequence
    (T_keep - B/4 rows, T_keep = B - min(64, B/4)) and at most its budget"""
    row = 2 * w.L * w.H_kv * w.d * w.esize  # K+V of one cached token over all layers
    first = row * int(np.sum(w.n0.astype(np.int64) + 1))
    tk = w.budget - np.minimum(64, w.budget // 4)
    lo = row * int(np.sum(np.where(w.n0 > w.budget, tk - w.budget // 4, w.n0)))
    hi = row * int(np.sum(np.minimum(w.n0.astype(np.int64) + 1, w.budget + 1)))
    if lo > L2_BYTES:
        return ("inputs larger than L2: the first step reads %.1f GB of K/V, later steps "
                "%.1f-%.1f GB (cache %.1f GB per GPU)" % (first / 1e9, lo / 1e9, hi / 1e9,
                                                         w.kv_bytes() / 1e9))
    return ("no flush between steps: a step within budget reads %.0f-%.0f MB of K/V, near or "
            "below the 129 MB L2, so bandwidth figures include L2 hits (cache %.0f MB per GPU)"
            % (lo / 1e6, hi / 1e6, w.kv_bytes() / 1e6))


def run_config(w, args, ws):
    """the config dict of both arms' lines (the workload and what the timed steps are)"""
    return dict(w.describe(), decode_steps=args.steps, l2=l2_note(w), policy=args.policy,
                timed_steps="each from a fresh cache" if args.fresh_each_step
                else "consecutive decode steps from a fresh cache",
                detector="token ids and p_max (lg_token_detect_prune)"
                if args.detector == "token" else "attention statistics and V-row sketches",
                parallelism="dp%d (independent batches, no collective)" % ws,
                tokens_per_step=w.batch * ws)


# ------------------------------------------------------------------ distributed plumbing

def dist_setup():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("gloo")
    return ws, rank, local


def barrier(ws):
    if ws > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x, ws):
    if ws == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(x, ws):
    if ws == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(t.item())


# ------------------------------------------------------------------ clocks during the timed region

class Clocks:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index, enabled=True):
        """the raw samples go to $LG_CLOCKS_DIR (default: the system temporary directory)"""
        self.proc = None
        self.path = os.path.join(os.environ.get("LG_CLOCKS_DIR") or tempfile.gettempdir(),
                                 "clocks_bench_%d.csv" % gpu_index)
        if not enabled:
            return
        os.makedirs(os.path.dirname(self.path), exist_ok=True)
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(gpu_index), "--query-gpu=" + self.FIELDS,
                 "--format=csv,noheader,nounits", "-lms", "50"], stdout=self.f,
                stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.f.close()
        sm, mx, reasons = [], 0.0, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    mx = max(mx, float(parts[2]))
                except ValueError:
                    continue
                for n, v in zip(names, parts[5:9]):
                    if v.lower() == "active":
                        reasons.add(n)
        if not sm:
            return {"samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


# ------------------------------------------------------------------ GPU arm

class GpuBench:
    """Device buffers, the per-step input variants and one guarded step on the C ABI."""

    def __init__(self, w, dev, total_steps, layers_per_call, policy="loopguard", detector="kv"):
        import torch
        from paper_2604_10044_gb300 import lg
        self.torch, self.lg = torch, lg
        self.detector = detector
        self.w, self.dev = w, dev
        self.policy = policy
        self.stream = torch.cuda.current_stream()
        self.s = self.stream.cuda_stream
        self.cache = lg.Cache(w.L, w.H_kv, w.d, w.dtype, w.seq_off, w.cap, w.n0, dev, policy)
        self.nl = layers_per_call if layers_per_call else w.L
        self.guard = lg.Guard(self.cache, w.H_q, n_layers_per_call=self.nl, policy=policy)
        # token positions of every step's new row (the same under either policy)
        self.pos32 = torch.as_tensor(
            (w.n0[None, :].astype(np.int64) + np.arange(max(total_steps, 1))[:, None]).astype(
                np.int32), device=dev)
        self.p = self.guard.p
        self.off_d = torch.as_tensor(w.seq_off, device=dev)
        self.n0_d = torch.as_tensor(w.n0, device=dev)
        self.budget_d = torch.as_tensor(w.budget.astype(np.int32), device=dev)
        self.seqs_d = synth.seqs_tensor(w.seqs, dev)
        bf = torch.bfloat16 if w.dtype == "bf16" else torch.float32
        S, L, b = total_steps, w.L, w.batch
        # both input variants of every step (A = loop continues, B = loop-free), packed per
        # step in one slab [q_A q_B k_A k_B v_A v_B] so that a step's inputs are one copy
        nq, nk = L * b * w.H_q * w.d, L * b * w.H_kv * w.d
        self.inp = torch.empty((S, 2 * nq + 4 * nk), dtype=bf, device=dev)
        cut = lambda o, n, h: self.inp[:, o:o + n].view(S, L, b, h, w.d)
        self.qA, self.qB = cut(0, nq, w.H_q), cut(nq, nq, w.H_q)
        self.kA, self.kB = cut(2 * nq, nk, w.H_kv), cut(2 * nq + nk, nk, w.H_kv)
        self.vA, self.vB = cut(2 * nq + 2 * nk, nk, w.H_kv), cut(2 * nq + 3 * nk, nk, w.H_kv)
        pos = torch.empty(b, dtype=torch.int64, device=dev)
        for t in range(S):
            pos.copy_(self.n0_d.to(torch.int64) + t)
            synth.dev_step(w, self.seqs_d, pos, self.qA[t], self.kA[t], self.vA[t], self.s, mode=2)
            synth.dev_step(w, self.seqs_d, pos, self.qB[t], self.kB[t], self.vB[t], self.s, mode=1)
        self.q = torch.empty((L, b, w.H_q, w.d), dtype=bf, device=dev)
        self.kn = torch.empty((L, b, w.H_kv, w.d), dtype=bf, device=dev)
        self.vn = torch.empty_like(self.kn)
        self.esz = 2 if w.dtype == "bf16" else 4
        e = self.esz
        # each sequence's inputs turn loop-free once the guard has intervened on it (its
        # state's intervention count); under the comparator policies loops persist
        self.gstate = self.guard.state if policy == "loopguard" else None
        self.sel = synth.Select3(w, self.gstate, lg.STATE_BYTES // 4, lg.STATE_WORD_N_INT,
                                 (self.q, self.kn, self.vn),
                                 (w.H_q * w.d * e, w.H_kv * w.d * e, w.H_kv * w.d * e))
        if detector == "token":
            # generated token ids and top-1 probabilities of every step, both variants
            tl, tf, pl, pf = synth.token_streams(w, S)
            self.tokA, self.tokB = (torch.as_tensor(x, device=dev) for x in (tl, tf))
            self.pmA, self.pmB = (torch.as_tensor(x, device=dev) for x in (pl, pf))
            self.tok = torch.zeros(b, dtype=torch.int32, device=dev)
            self.pm = torch.zeros(b, dtype=torch.float32, device=dev)
            self.tp = lg.lg_default_token_params()
            self.tstate = torch.zeros(lg.lg_token_state_size(self.cache, self.guard.p, self.tp) // 4,
                                      dtype=torch.int32, device=dev)
        torch.cuda.synchronize()

    def reset(self):
        """fresh cache of the workload, guard state and sequence modes (untimed)"""
        torch, w, lg = self.torch, self.w, self.lg
        self.cache.len.copy_(self.n0_d)
        synth.dev_fill_cache(w, self.cache.k, self.cache.v, self.seqs_d.copy_(
            synth.seqs_tensor(w.seqs, self.dev)), self.off_d, self.n0_d, int(w.n0.max()), self.s)
        if self.policy in ("h2o", "streaming", "full"):
            lg.lg_h2o_reset(self.cache, int(w.n0.max()))
        else:
            lg.lg_sketch_build(self.cache, self.p, int(w.n0.max()))
        # the token monitor counts generated tokens from 0; the KV-space test counts the
        # prompt as seen (its window starts full)
        lg.lg_state_init(self.cache, self.guard.state, 0 if self.detector == "token" else 64)
        self.guard.dstate.zero_()
        if self.detector == "token":
            self.tstate.zero_()
        self.cache.status.zero_()
        torch.cuda.synchronize()

    def use_stage(self, on=True):
        """read every step's inputs from one fixed device slab (filled by the caller before each
        step, as a serving loop fills its input buffers) instead of the step's own slab, so that
        one captured graph serves every step; the slab packs both input variants and, for the
        token-level detector, both token and p_max variants as raw bytes"""
        torch, w = self.torch, self.w
        self.stage = None
        if not on:
            return
        L, b, d = w.L, w.batch, w.d
        nq, nk = L * b * w.H_q * d, L * b * w.H_kv * d
        inp_bytes = self.inp[0].numel() * self.inp.element_size()
        tok_bytes = 16 * b if self.detector == "token" else 0
        self.stage = torch.empty(inp_bytes + tok_bytes, dtype=torch.uint8, device=self.dev)
        sin = self.stage[:inp_bytes].view(self.inp.dtype)
        cut = lambda o, n, h: sin[o:o + n].view(L, b, h, d)
        self.st_A = (cut(0, nq, w.H_q), cut(2 * nq, nk, w.H_kv), cut(2 * nq + 2 * nk, nk, w.H_kv))
        self.st_B = (cut(nq, nq, w.H_q), cut(2 * nq + nk, nk, w.H_kv),
                     cut(2 * nq + 3 * nk, nk, w.H_kv))
        if tok_bytes:
            ti = self.stage[inp_bytes:inp_bytes + 8 * b].view(torch.int32)
            tp = self.stage[inp_bytes + 8 * b:].view(torch.float32)
            self.st_tok = (ti[:b], ti[b:], tp[:b], tp[b:])

    def stage_host(self, K):
        """the K steps' staged inputs in pinned host memory, [K][stage bytes]"""
        torch = self.torch
        rows = [self.inp[:K].cpu().view(torch.uint8).reshape(K, -1)]
        if self.detector == "token":
            rows += [torch.cat([self.tokA[:K], self.tokB[:K]], 1).cpu().view(torch.uint8),
                     torch.cat([self.pmA[:K], self.pmB[:K]], 1).cpu().view(torch.uint8)]
        return torch.cat(rows, 1).contiguous().pin_memory()

    def select_inputs(self, t):
        """the step's q, k_new, v_new (and, for the token-level monitor, its token id and top-1
        probability) in one launch, each sequence's variant chosen by its guard state"""
        staged = getattr(self, "stage", None) is not None
        tokens = None
        if self.detector == "token" and self.policy == "loopguard":
            tl, tf, pl, pf = (self.st_tok if staged else
                              (self.tokA[t], self.tokB[t], self.pmA[t], self.pmB[t]))
            tokens = (tl, tf, pl, pf, self.tok, self.pm)
        if staged:
            self.sel(self.st_A, self.st_B, self.s, tokens)
            return
        self.sel((self.qA[t], self.kA[t], self.vA[t]), (self.qB[t], self.kB[t], self.vB[t]),
                 self.s, tokens)

    def step(self, t, ev=None, split=False):
        """one guarded decode step; ev = (a0, a1, p0, p1) events around attend and the guard
        (a1 -> p1); split: the loop-onset test and the compaction as separate calls
        (lg_detect or lg_token_detect, then lg_prune_compact: the same results) with p0 between
        them"""
        lg, c, g, p, w = self.lg, self.cache, self.guard, self.p, self.w
        h2o = self.policy == "h2o"
        guard_path = self.policy == "loopguard"
        pos_t = None if guard_path else self.pos32[t]
        self.select_inputs(t)
        lg.lg_begin_step(c, self.s)
        lg.lg_append(c, 0, w.L, self.kn, self.vn, pos_t, p, self.s)
        if ev:
            ev[0].record(self.stream)
        for l0 in range(0, w.L, self.nl):
            nl = min(self.nl, w.L - l0)   # the last call takes what is left
            lg.lg_decode_attend(c, l0, nl, self.q[l0:l0 + nl], w.H_q, g.scale, g.out[l0:l0 + nl],
                                g.stats[l0:l0 + nl], p.suffix_w, 1 if h2o else 0, g.max_len,
                                g.ws, self.s)
        if ev:
            ev[1].record(self.stream)
        token = guard_path and self.detector == "token"
        if token and not split:
            # the token-level monitor on the step's token and top-1 probability (picked with the
            # step's inputs), its retained set, then the compaction
            lg.lg_token_detect_prune(c, self.tok, self.pm, g.state, self.budget_d, p, self.tp,
                                     g.flags, g.spans, None, self.tstate, g.kept_idx,
                                     g.kept_count, g.max_keep, g.max_len, self.s)
        elif token:
            lg.lg_token_detect(c, self.tok, self.pm, g.state, p, self.tp, g.flags, g.spans,
                               None, self.tstate, g.kept_idx, g.kept_count, self.s)
        elif guard_path and not split:
            # loop-onset test and retained set in one kernel, then the compaction
            lg.lg_detect_prune(c, g.stats, w.H_q, g.state, self.budget_d, p, g.flags, g.spans,
                               None, g.dstate, g.kept_idx, g.kept_count, g.max_keep, g.max_len,
                               self.s)
        elif guard_path:
            lg.lg_detect(c, g.stats, w.H_q, g.state, self.budget_d, p, g.flags, g.spans, None,
                         g.dstate, self.s)
        if ev:
            ev[2].record(self.stream)
        if guard_path and split:
            lg.lg_prune_compact(c, g.flags, g.spans, g.state, self.budget_d, p, g.kept_idx,
                                g.kept_count, g.max_keep, g.max_len, self.s)
        elif h2o:
            lg.lg_h2o_evict(c, self.budget_d, pos_t, g.max_len, self.s)
        elif self.policy == "streaming":
            lg.lg_streaming_evict(c, self.budget_d, pos_t, lg.N_SINK, g.max_len, self.s)
        if ev:
            ev[3].record(self.stream)

    # launches of this repository's kernels per step (harness + path)
    def launches_per_step(self):
        calls = math.ceil(self.w.L / self.nl)
        # per call on the tensor-core path: the counter reset and the pass (it merges its own
        # partials); a partial pass and a merge on the fp32 path; H2O adds the score update
        attend = 2 + (1 if self.policy == "h2o" else 0)
        path = 1 + 1 + attend * calls               # begin, append (+sketch), attend
        harness = 1                                 # the step's inputs
        if self.policy in ("h2o", "streaming"):     # evict, lengths
            path += 2
        elif self.policy == "loopguard" and self.detector == "token":
            path += 2                               # token monitor + keep, compact
        elif self.policy == "loopguard":
            path += 2                               # detect + keep, compact
        return path, harness

    def replay_log(self, K, fresh=False):
        """replay the timed trajectory (the decisions are deterministic, so they are the
        timed run's), recording per-step lengths and kept lists, with the guard split into
        lg_detect and lg_prune_compact and events around the compaction; returns
        (lens, kept, compaction ms per step)"""
        torch = self.torch
        # one untimed step of the split guard first: the timed run launches the fused call
        # only, and the first launch of a kernel also loads it (lazy module loading)
        self.reset()
        self.step(0, None, split=True)
        self.reset()
        lens, kept, evs = [], [], []
        for t in range(K):
            if fresh:
                self.reset()
            lens.append(self.cache.len.clone())
            ev = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
            self.step(0 if fresh else t, ev, split=True)
            evs.append(ev)
            if self.policy != "loopguard":
                kept.append((None, None))
                continue
            kc = self.guard.kept_count.clone()
            kept.append((kc, self.guard.kept_idx.clone() if int((kc >= 0).sum()) else None))
        torch.cuda.synchronize()
        return lens, kept, [e[2].elapsed_time(e[3]) for e in evs]


def attend_bytes(w, n_rows, h2o=False):
    """algorithmic bytes of attend+stats for one step: K and V rows once per kv-head and
    layer, queries, outputs and statistics; on the H2O path also the logits written and read
    back (4 g bytes each) and the score read-modify-write (8 bytes) per (layer, kv-head, row)"""
    esz = 2 if w.dtype == "bf16" else 4
    rows = w.L * w.H_kv * int(np.sum(n_rows))
    kv = 2 * w.d * esz * rows
    qo = 2 * w.L * w.batch * w.H_q * w.d * esz + w.L * w.batch * w.H_q * 16
    extra = (8 * w.g + 8) * rows if h2o else 0
    return kv + qo + extra


def compact_bytes(w, kept_count, kept_idx):
    """algorithmic bytes of one prune: every moved row of K and V (all layers and kv-heads) and
    of the sketches read once and written once"""
    esz = 2 if w.dtype == "bf16" else 4
    total = 0
    for b in range(w.batch):
        c = int(kept_count[b])
        if c < 0:
            continue
        k = kept_idx[b, :c]
        moved = int(np.sum(k != np.arange(c)))
        total += 2 * moved * (2 * w.L * w.H_kv * w.d * esz + w.H_kv * w.d // 8)
    return total


def traffic_from_profile(kernel_src_hash):
    """DRAM bytes per attend launch from the committed ncu summary, if it was taken on the
    current kernel source; else None"""
    path = os.path.join(ROOT, "profiles", "attend_mma_traffic.txt")
    if not os.path.exists(path):
        return None
    with open(path) as f:
        d = json.load(f)
    if d.get("source_sha256") != kernel_src_hash:
        return None
    return d


def code_only(src):
    """C/C++/CUDA source without its comments, runs of white space as one space: an edit of a
    comment or of the layout leaves it unchanged, any edit of the code does not"""
    out, i, n = [], 0, len(src)
    while i < n:
        c = src[i]
        if c == '"' or c == "'":                      # a literal, copied whole
            j = i + 1
            while j < n and src[j] != c:
                j += 2 if src[j] == "\\" else 1
            out.append(src[i:j + 1])
            i = j + 1
        elif src.startswith("//", i):
            j = src.find("\n", i)
            i = n if j < 0 else j
        elif src.startswith("/*", i):
            j = src.find("*/", i + 2)
            out.append(" ")
            i = n if j < 0 else j + 2
        else:
            out.append(c)
            i += 1
    return " ".join("".join(out).split())


def source_hash():
    """sha256 of the attention kernel's code (comments and layout excluded): the committed
    DRAM-traffic summary holds the value for the code it was captured on"""
    import hashlib
    h = hashlib.sha256()
    for f in ("lg_attend_mma.cu", "lg_common.cuh"):
        with open(os.path.join(ROOT, "paper_2604_10044_gb300", "csrc", f)) as fh:
            h.update(code_only(fh.read()).encode())
    return h.hexdigest()


def gpu_workload(args, rank=0):
    """the GPU arm's workload: rank r > 0 draws its own batch (seed 1000 + r); the capacity
    covers every step of the run under any policy (the full cache never evicts)"""
    over = {"steps": max(args.steps, args.warmup, args.profile_steps, 1)}
    if rank:
        over["seed"] = 1000 + rank
    if args.batch:
        over["batch"] = args.batch
    return synth.make_workload(args.workload, **over)


def run_gpu(args, ws, rank, local):
    import torch
    assert torch.cuda.is_available(), "the gb300 arm needs a CUDA device"
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    K, W = args.steps, args.warmup
    w = gpu_workload(args, rank)
    if args.profile_steps:
        # untimed steps inside an NVTX range "steps" (ncu --nvtx-include "steps/")
        bench = GpuBench(w, dev, args.profile_steps, args.layers_per_call, args.policy,
                         args.detector)
        bench.reset()
        rows = []
        torch.cuda.nvtx.range_push("steps")
        for t in range(args.profile_steps):
            rows.append(w.L * w.H_kv * int((bench.cache.len.cpu() + 1).sum()))
            bench.step(t)
        torch.cuda.synchronize()
        torch.cuda.nvtx.range_pop()
        # K/V rows each step's attention launch reads (for the DRAM-traffic summary)
        print(json.dumps({"workload": args.workload, "batch": w.batch,
                          "attend_rows_per_launch": rows,
                          "attend_alg_bytes_per_launch": [
                              attend_bytes(w, np.full(w.batch, 0)) + 2 * w.d * w.esize * r
                              for r in rows]}), flush=True)
        return None
    # the read-only bandwidth denominator, measured before the cache takes the memory
    rpeak, rprobes = read_peak(dev)
    fresh = args.fresh_each_step
    # every launch of the run goes to one side stream (stream capture needs a non-default one)
    side = torch.cuda.Stream(device=dev)
    torch.cuda.set_stream(side)
    bench = GpuBench(w, dev, 1 if fresh else max(K, W, 1), args.layers_per_call, args.policy,
                     args.detector)

    # warm-up on the trajectory's first W steps, then a fresh cache for the timed run
    bench.reset()
    for t in range(W):
        if fresh:
            bench.reset()
        bench.step(0 if fresh else t)
    torch.cuda.synchronize()
    start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    graph = None
    eager_ms = None
    # steps whose attention pass and guard are bracketed by timing events inside the timed
    # region: every EV_EVERY-th step (an event between two kernels ends their programmatic
    # launch overlap, so events on every step would slow the steps they time)
    # (starting at step every/2, so that the first step's one-off budget cut of every sequence,
    # one step in K of the timed region, does not weigh as one in K/every of the sample)
    every = 1 if fresh else max(min(EV_EVERY, max(1, K // 4)), K // EV_SAMPLES)
    sampled = set(range(every // 2, K, every))
    ev_note = ("every step" if every == 1 else
               "every %dth step of the timed region from step %d (%d of %d), events around the "
               "attention pass and the guard" % (every, every // 2, len(sampled), K))
    if not fresh and not args.eager:
        # the same K steps timed eagerly first (reported beside the graph figure), then
        # captured once as a CUDA graph whose single replay is the timed region; events
        # recorded as graph nodes time each part of every step
        bench.reset()
        barrier(ws)
        torch.cuda.synchronize()
        start.record(bench.stream)
        for t in range(K):
            bench.step(t)
        stop.record(bench.stream)
        torch.cuda.synchronize()
        eager_ms = max_over_ranks(start.elapsed_time(stop), ws)
        evs = [[torch.cuda.Event(enable_timing=True, external=True) for _ in range(4)]
               if t in sampled else None for t in range(K)]
        for e in evs:
            for x in e or ():
                x.record(bench.stream)
        bench.reset()
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=bench.stream, capture_error_mode="thread_local"):
            for t in range(K):
                bench.step(t, evs[t])
        graph.replay()                        # untimed: uploads the graph
        torch.cuda.synchronize()
        if bench.lg.lg_read_device_status(bench.cache) != 0:
            raise RuntimeError("device status %d after the graph warm-up replay"
                               % bench.lg.lg_read_device_status(bench.cache))
    else:
        evs = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] if t in sampled else None
               for t in range(K)]
    bench.reset()
    clocks = Clocks(local, enabled=not args.no_clocks)
    barrier(ws)
    torch.cuda.synchronize()
    if graph is not None:
        start.record(bench.stream)
        graph.replay()
        stop.record(bench.stream)
        torch.cuda.synchronize()
        ms_local = start.elapsed_time(stop)
    elif fresh:
        # every step from a freshly generated cache; only the steps are timed
        ms_local = 0.0
        for t in range(K):
            if t:
                bench.reset()
            start.record(bench.stream)
            bench.step(0, evs[t])
            stop.record(bench.stream)
            torch.cuda.synchronize()
            ms_local += start.elapsed_time(stop)
    else:
        start.record(bench.stream)
        for t in range(K):
            bench.step(t, evs[t])
        stop.record(bench.stream)
        torch.cuda.synchronize()
        ms_local = start.elapsed_time(stop)
    barrier(ws)
    clk = clocks.stop()
    status = bench.lg.lg_read_device_status(bench.cache)
    if status != 0:
        raise RuntimeError("device status %d after the timed run" % status)
    ms = max_over_ranks(ms_local, ws)
    sampled = sorted(sampled)
    attend_ms = [evs[t][0].elapsed_time(evs[t][1]) for t in sampled]
    guard_ms = [evs[t][1].elapsed_time(evs[t][3]) for t in sampled]

    # algorithmic bytes of the same trajectory (deterministic replay, not the timed region)
    lens, kept, prune_ms = bench.replay_log(K, fresh)
    a_bytes, c_bytes, c_ms = [], [], []
    for t in range(K):
        n_rows = lens[t].cpu().numpy() + 1
        a_bytes.append(attend_bytes(w, n_rows, args.policy == "h2o"))
        kc, ki = kept[t]
        if kc is None:
            continue
        kc = kc.cpu().numpy()
        if ki is not None:
            c_bytes.append(compact_bytes(w, kc, ki.cpu().numpy()))
            c_ms.append(prune_ms[t])
    hbm_peak, peak_kind = peaks()
    attend_gbs = sum(a_bytes[t] for t in sampled) / (sum(attend_ms) * 1e-3) / 1e9
    compact_gbs = (sum(c_bytes) / (sum(c_ms) * 1e-3) / 1e9) if c_ms else None

    e2e = e2e_eager = None
    if not args.no_e2e and not fresh and args.policy == "loopguard":
        e2e, e2e_eager = run_e2e(bench, K, ws, graphs=not args.eager)

    value = sum_over_ranks(K, ws) / (ms * 1e-3)
    step_read = sum(a_bytes) / max(1, len(a_bytes))
    path_l, harness_l = bench.launches_per_step()
    # DRAM bytes of one attention launch of the sampled steps, from the committed capture of
    # this workload on the current kernel code (scaled by the rows a launch reads: the sampled
    # steps' lengths differ from the captured launch's by a few rows); else null
    prof = traffic_from_profile(source_hash())
    traffic, traffic_note = None, "no DRAM capture of this workload on the current kernel code"
    sampled_rows = [w.L * w.H_kv * int(np.sum(lens[t].cpu().numpy() + 1)) for t in sampled]
    if (prof and bench.nl == w.L and prof.get("workload") == args.workload
            and prof.get("batch") == w.batch and args.policy == "loopguard"):
        rows = sum(sampled_rows) / len(sampled_rows)
        traffic = int(prof["dram_bytes"] * rows / prof["rows"])
        traffic_note = ("ncu dram__bytes_read.sum + dram__bytes_write.sum of the attention launch "
                        "of %s (profiles/attend_mma_traffic.txt), scaled by %.6f for the rows "
                        "of the sampled steps" % (prof["launch"], rows / prof["rows"]))
    line = {
        "metric": METRIC, "value": round(value, 3), "unit": UNIT, "n_gpus": ws, "steps": K,
        "warmup": W, "ms_per_step": round(ms / K, 4), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": w.dtype, "data": "synthetic",
        "config": run_config(w, args, ws),
        "launch": {"mode": "eager" if graph is None else
                   "one CUDA graph replay of the K steps (captured before timing)",
                   "layers_per_attend_call": bench.nl},
        "kv_read_GB_per_step": round(step_read / 1e9, 3),
        "roofline": {"bound": "hbm", "achieved": round(attend_gbs, 1), "peak": hbm_peak,
                     "unit": "GB/s", "frac": round(attend_gbs / hbm_peak, 4),
                     "traffic": traffic, "traffic_note": traffic_note,
                     "alg_bytes_per_launch": int(sum(a_bytes[t] for t in sampled) / len(sampled)),
                     "kernel": "lg_decode_attend (tensor-core pass with its split-K merge), all "
                               "%d layers per call" % w.L if bench.nl == w.L
                               else "lg_decode_attend",
                     "peak_kind": peak_kind + " copy bandwidth (MEASURED_PEAKS.json)",
                     "read_peak": round(rpeak, 1),
                     "frac_of_read_peak": round(attend_gbs / rpeak, 4),
                     "read_peak_kind": "the fastest of three read-only passes over 4 GiB, "
                                       "measured in this run (best of 10 each, CUDA events)",
                     "read_probes_GB_per_s": rprobes},
        "kernels": {
            "attend_stats": {"GB_per_s": round(attend_gbs, 1),
                             "frac_of_%s_peak" % peak_kind: round(attend_gbs / hbm_peak, 4),
                             "frac_of_8TBs_nominal": round(attend_gbs / 8000.0, 4),
                             "frac_of_read_peak": round(attend_gbs / rpeak, 4),
                             "ms_per_step": round(sum(attend_ms) / len(sampled), 4),
                             "timed_steps": ev_note},
            "prune_compact": {"GB_per_s": round(compact_gbs, 1) if compact_gbs else None,
                              "frac_of_%s_peak" % peak_kind:
                                  round(compact_gbs / hbm_peak, 4) if compact_gbs else None,
                              "frac_of_8TBs_nominal":
                                  round(compact_gbs / 8000.0, 4) if compact_gbs else None,
                              "events": len(c_ms),
                              "ms_per_event": round(sum(c_ms) / len(c_ms), 4) if c_ms else None,
                              "moved_bytes_per_event": int(sum(c_bytes) / len(c_bytes))
                              if c_bytes else 0},
            # the guard's kernels on the sampled steps; with programmatic launch the kernels of
            # a step overlap, so the step time is below the sum of its parts
            "guard_ms_per_step": round(sum(guard_ms) / len(sampled), 4)},
        "eager_ms_per_step": round(eager_ms / K, 4) if eager_ms is not None else None,
        "gpu_launches": (path_l + harness_l) * K,
        "gpu_launches_detail": {"path_per_step": path_l, "harness_per_step": harness_l},
        "clocks": clk,
    }
    if e2e:
        line["e2e"] = e2e
        line["e2e_eager"] = {"value": e2e_eager, "unit": UNIT}
    return line, w


def run_e2e(bench, K, ws, graphs=True):
    """the same steps through the C ABI with host buffers: every step copies its inputs from
    pinned host memory into the step's input slab on the device (one copy), runs the guarded
    step and reads the outputs back (attention output, flags, spans, lengths), and the host
    waits for them before the next step.  graphs: the step's calls and the gathering of its
    results are captured once as one CUDA graph over the fixed slab (as a serving loop
    captures its decode step) and replayed every step, the copies around it stream copies;
    else the calls are launched eagerly.  Returns (line dict, eager steps/s)."""
    torch = bench.torch
    w = bench.w
    g = bench.guard
    bench.use_stage(True)
    stage_h = bench.stage_host(K)  # both input variants of every step, filled before timing
    out_h = torch.empty(g.out.shape, dtype=g.out.dtype).pin_memory()
    fs_h = torch.empty(3 * w.batch, dtype=torch.int32).pin_memory()
    len_h = torch.empty(w.batch, dtype=torch.int32).pin_memory()
    # graphed steps gather the outputs, flags, spans and lengths into one buffer on the device
    # (inside the step's graph), read back with one copy
    out_bytes = g.out.numel() * g.out.element_size()
    pack_d = torch.empty(out_bytes + 16 * w.batch, dtype=torch.uint8, device=bench.dev)
    pack_h = torch.empty(pack_d.numel(), dtype=torch.uint8).pin_memory()
    pack_out = pack_d[:out_bytes].view(g.out.dtype).view(g.out.shape)
    pack_fs = pack_d[out_bytes:out_bytes + 12 * w.batch].view(torch.int32)
    pack_len = pack_d[out_bytes + 12 * w.batch:].view(torch.int32)

    def pack():
        pack_out.copy_(g.out)
        pack_fs.copy_(g.flags_spans)
        pack_len.copy_(bench.cache.len)

    def copy_in(t):
        bench.stage.copy_(stage_h[t], non_blocking=True)

    def copy_out():
        out_h.copy_(g.out, non_blocking=True)
        fs_h.copy_(g.flags_spans, non_blocking=True)
        len_h.copy_(bench.cache.len, non_blocking=True)

    def enqueue(t):
        copy_in(t)
        bench.step(t)
        copy_out()

    def timed(run_step):
        bench.reset()
        barrier(ws)
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        for t in range(K):
            run_step(t)
            bench.stream.synchronize()
        return max_over_ranks(time.perf_counter() - t0, ws)

    dt_eager = timed(enqueue)
    dt_graph = None
    if graphs:
        # one graph for every step: it reads the fixed input slab (the copies into it and out
        # of the gathered results stay stream copies; as graph nodes, copies from pinned host
        # memory ran several times slower on this system)
        gr = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gr, stream=bench.stream, capture_error_mode="thread_local"):
            bench.step(0)
            pack()
        bench.reset()
        copy_in(0)
        gr.replay()  # untimed: the first launch of a graph uploads it
        torch.cuda.synchronize()

        def graphed(t):
            copy_in(t)
            gr.replay()
            pack_h.copy_(pack_d, non_blocking=True)
        dt_graph = timed(graphed)
    bench.use_stage(False)
    h2d = stage_h[0].numel()
    d2h = out_h.numel() * out_h.element_size() + (fs_h.numel() + len_h.numel()) * 4
    rate = lambda d: round(sum_over_ranks(K, ws) / d, 3) if d else None
    # the faster of the two ways a serving loop can drive the calls (both reported)
    use_graph = dt_graph is not None and dt_graph < dt_eager
    line = {"value": rate(dt_graph if use_graph else dt_eager), "unit": UNIT,
            "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
            "launch": "a stream copy in, the step's kernels and the gathering of its results as "
                      "one CUDA graph (the same for every step), a stream copy out; host waits "
                      "for each step" if use_graph
                      else "eager calls, host waits for each step",
            "steps_per_s_eager": rate(dt_eager), "steps_per_s_graphed_kernels": rate(dt_graph),
            "note": "inputs of both sequence modes (loop continues / loop-free) copied every "
                    "step; outputs, flags, spans and lengths read back every step; the faster "
                    "of the two launch modes"}
    return line, rate(dt_eager)


# ------------------------------------------------------------------ CPU oracle arm

def oracle_sample_workload(w, n_seq):
    """the first n_seq sequences of workload w (same rows: the generator keys on the index)"""
    sub = synth.Workload(name=w.name, L=w.L, H_q=w.H_q, H_kv=w.H_kv, d=w.d, dtype=w.dtype,
                         batch=n_seq, n0=w.n0[:n_seq], budget=w.budget[:n_seq], steps=w.steps,
                         seed=w.seed, seqs=w.seqs[:n_seq].copy(), head_scale=w.head_scale,
                         n_sink=w.n_sink, sink_factor=w.sink_factor, sigma=w.sigma,
                         query_mode=w.query_mode, zstar=w.zstar, q_noise=w.q_noise)
    return sub


def time_oracle(w, n_seq, n_layers, steps, warm=0, policy="loopguard", detector="kv",
                fresh=False):
    """the oracle (as it stands) running `steps` guarded decode steps of the first n_seq
    sequences restricted to the first n_layers layers, from a fresh cache (after `warm`
    warm-up steps, themselves from a fresh cache); detector "token": the token-level monitor
    on the generated-token streams in place of the KV-space test, as on the GPU arm (tokens
    counted from 0, each sequence's loop-free tokens once the guard has intervened on it);
    fresh: every timed step from a fresh cache (the first step, as --fresh-each-step times it).
    Returns (seconds per step, threads)"""
    import oracle
    sub = oracle_sample_workload(w, n_seq)
    sub.L = n_layers
    K, V = synth.host_cache(sub)
    token = policy == "loopguard" and detector == "token"

    def run(n):
        g = oracle.OracleGuard(sub, K.copy(), V.copy(), policy=policy,
                               t_gen0=0 if token else 64)
        seqs = sub.seqs.copy()
        pos = sub.n0.astype(np.int64)
        if token:
            tl, tf, pl, pf = synth.token_streams(sub, n)
            tp = oracle.token_params()
            ts = [oracle.new_token_state() for _ in range(sub.batch)]
            hist = np.zeros((n, sub.batch), dtype=np.int32)
            prev_kept = [None] * sub.batch
        times = []
        for t in range(n):
            q, kn, vn = synth.host_step(sub, pos, seqs)
            t0 = time.perf_counter()
            if token:
                g.append(kn, vn)
                g.attend(q)
                flags = np.zeros(sub.batch, dtype=np.int32)
                spans = np.zeros((sub.batch, 2), dtype=np.int32)
                for b in range(sub.batch):
                    fresh = g.state[b].n_int > 0
                    hist[t, b] = tf[t, b] if fresh else tl[t, b]
                    pm = float(pf[t, b] if fresh else pl[t, b])
                    flags[b], spans[b], _ = oracle.token_detect(
                        hist[:t + 1, b], pm, int(g.len[b]), g.prm, tp, g.state[b], ts[b],
                        kept=prev_kept[b])
                n_before = g.len.copy()
                kept = g.prune(flags, spans)
                prev_kept = [kept[b] if flags[b] or n_before[b] > sub.budget[b] else None
                             for b in range(sub.batch)]
                r = {"flags": flags}
            else:
                r = g.step(q, kn, vn, pos)
            times.append(time.perf_counter() - t0)
            if policy == "loopguard":
                synth.note_interventions(seqs, pos, r["flags"])
            pos = pos + 1
        return times, getattr(g, "threads", 1)

    if warm:
        run(warm)          # warm-up steps; the timed steps start again from the fresh cache
    if fresh:
        times, threads = [], 1
        for _ in range(steps):
            t, threads = run(1)
            times += t
        return times, threads
    return run(steps)


def oracle_sample(w, K, W, policy="loopguard", target_s=ORACLE_TARGET_S, max_layers=None,
                  detector="kv", fresh=False):
    """The oracle on a bounded sample of the GPU arm's timed run: sequence 0 of the batch and its
    first n_layers layers, W warm-up steps, then the same K consecutive guarded decode steps from
    a fresh cache (the first carries the budget cut, as on the GPU).  n_layers follows from the
    sample's work (ORACLE_SAMPLE_ROW_HEADS), capped by a one-layer timing run so that the K timed
    steps take at most about 2 target_s on a slow host.  Both oracle figures
    of bench.py (the GPU line's cpu_baseline and the --impl reference line) are this sample.
    Returns a dict: value (batch steps/s, the sample scaled by sequences and layers), the
    measured seconds, the scale and a description."""
    if max_layers == 1:
        n_layers = 1
    else:
        # from the sample's work: sequence 0 reads its n0 + 1 rows on the first step and at most
        # its budget's on every later one, once per kv-head and layer
        n0, B = int(w.n0[0]), int(w.budget[0])
        per_layer = ((n0 + 1) * K if fresh else (n0 + 1) + (K - 1) * min(n0 + 1, B)) * w.H_kv
        n_layers = int(min(max_layers or w.L, max(1, round(ORACLE_SAMPLE_ROW_HEADS / per_layer))))
        # a cap from a one-layer timing run, for a host much slower than the one the work figure
        # was set on (one layer on few cores overstates a layer's share, so this rarely binds)
        cal = min(K, 3)
        t_cal, _ = time_oracle(w, 1, 1, cal, policy=policy, detector=detector, fresh=fresh)
        t_layer = t_cal[0] + (K - 1) * (float(np.mean(t_cal[1:])) if cal > 1 else t_cal[0])
        n_layers = int(max(1, min(n_layers, (2 * target_s) // max(t_layer, 1e-6))))
    times, threads = time_oracle(w, 1, n_layers, K, warm=W, policy=policy, detector=detector,
                                 fresh=fresh)
    sec = sum(times)
    scale = (1.0 / w.batch) * (n_layers / w.L)   # batch steps per sampled step
    return {"value": K * scale / sec, "sec": sec, "steps": K, "scale": scale,
            "threads": threads, "n_layers": n_layers,
            "sample": "%s (after %d warm-up step(s)), of sequence 0 of %d and its layers 0..%d "
                      "of %d; value = steps x %.6f batch steps per sampled step / %.2f s" % (
                          "%d first guarded decode steps, each from a fresh cache" % K if fresh
                          else "the first %d guarded decode steps of the GPU arm's timed "
                               "trajectory, from its fresh cache" % K,
                          W, w.batch, n_layers - 1, w.L, scale, sec)}


def cpu_baseline(w, args):
    """the oracle on the host cores: the bounded sample of oracle_sample, as batch steps/s; and
    beside it the same trajectory's first steps on one thread (one layer, at most 2 steps, in a
    fresh interpreter: the oracle takes its thread count when it loads)"""
    o = oracle_sample(w, args.steps, args.warmup, args.policy, detector=args.detector,
                      fresh=args.fresh_each_step)
    line = {"value": round(o["value"], 6), "unit": UNIT, "cores": o["threads"],
            "kind": "oracle", "affinity_cores": len(os.sched_getaffinity(0)),
            "sample": o["sample"], "sample_scale": o["scale"],
            "ms_per_sample_step": round(o["sec"] / o["steps"] * 1e3, 3)}
    try:
        env = dict(os.environ, OMP_NUM_THREADS="1")
        cmd = [sys.executable, os.path.abspath(__file__), "--oracle-one-thread",
               "--workload", str(args.workload), "--steps", str(min(args.steps, 2)),
               "--policy", args.policy, "--detector", args.detector]
        if args.batch:
            cmd += ["--batch", str(args.batch)]
        if args.fresh_each_step:
            cmd += ["--fresh-each-step"]
        r = subprocess.run(cmd, env=env, capture_output=True, text=True, timeout=600)
        one = json.loads(r.stdout.strip().splitlines()[-1])
        line["single_thread"] = {"value": round(one["value"], 6), "unit": UNIT,
                                 "cores": one["threads"], "sample": one["sample"]}
    except Exception as e:  # a reported extra: its failure leaves the main figure
        line["single_thread"] = {"value": None, "error": str(e)[:200]}
    return line


def run_reference(args, ws, rank):
    """--impl reference: the CPU oracle on the host cores, on the same bounded sample of the
    same timed run as the GPU line's cpu_baseline (oracle_sample): W warm-up steps, then K
    timed steps from a fresh cache.  ms_per_step is the measured time of one sampled step;
    value = sample_scale x 1000 / ms_per_step batch steps/s."""
    if rank != 0:
        return
    K, W = args.steps, args.warmup
    w = gpu_workload(args, rank)   # rank 0's batch: the GPU arm's, --batch included
    o = oracle_sample(w, K, W, args.policy, detector=args.detector, fresh=args.fresh_each_step)
    value = o["value"]
    line = {"impl": "reference", "metric": METRIC, "value": round(value, 6), "unit": UNIT,
            "n_gpus": ws, "steps": K, "warmup": W,
            "ms_per_step": round(o["sec"] / K * 1e3, 3), "sample_scale": o["scale"],
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": run_config(w, args, ws),
            "cpu_baseline": {"value": round(value, 6), "unit": UNIT, "cores": o["threads"],
                             "kind": "oracle", "affinity_cores": len(os.sched_getaffinity(0)),
                             "sample": o["sample"], "sample_scale": o["scale"]},
            "e2e": {"value": round(value, 6), "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def run_ablation(args, local):
    """the ablation analog (synth.ablation) at the paper's setting: B = 1024, a 3853-token
    prompt, T_max = 2500, loops starting at 800-1300 generated tokens with periods 16..64"""
    import torch
    import synth.ablation as A
    from paper_2604_10044_gb300.ablation import run_variant
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    streams = A.LoopStreams(args.batch or 64, 3853, 2500)
    res = {}
    for name, over in A.VARIANTS.items():
        t0 = time.perf_counter()
        m, _ = run_variant(streams, over, dev)
        m["wall_s"] = round(time.perf_counter() - t0, 2)
        res[name] = m
    print(json.dumps({
        "metric": "synthetic ablation of the guard variants (Table 3 analog)",
        "unit": "loop rate %, interventions per sequence, early interventions %",
        "variants": res, "data": "synthetic",
        "config": {"sequences": streams.batch, "prompt": 3853, "budget": 1024,
                   "steps": streams.steps, "onset": "U{800..1300}", "period": "U{16..64}",
                   "detector": "token-level monitor and retained set (lg_token_detect_prune)"}}),
        flush=True)


def main():
    args = parse()
    if args.oracle_one_thread:
        # internal: the oracle's sample on this process's threads (one, from the environment)
        w = gpu_workload(args)
        o = oracle_sample(w, args.steps, 0, args.policy, target_s=0.0, max_layers=1,
                          detector=args.detector, fresh=args.fresh_each_step)
        print(json.dumps({"value": o["value"], "threads": o["threads"], "sample": o["sample"]}),
              flush=True)
        return
    ws, rank, local = dist_setup()
    if args.ablation:
        if rank == 0:
            run_ablation(args, local)
        return
    if ws != args.gpus:
        raise SystemExit("--gpus %d but WORLD_SIZE=%d" % (args.gpus, ws))
    if args.impl == "reference":
        run_reference(args, ws, rank)
        return
    res = run_gpu(args, ws, rank, local)
    if res is None:
        return
    line, w = res
    if rank == 0:
        if ws == 1 and not args.no_cpu_baseline:
            line["cpu_baseline"] = cpu_baseline(w, args)
        print(json.dumps(line), flush=True)


if __name__ == "__main__":
    main()
