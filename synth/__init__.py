"""Seeded synthetic workloads for the LoopGuard decode path (harness only).

The guard runs on K/V caches, queries and appended rows that a language model
would produce; none is available here, so this module draws them from a
counter-based generator.  It serves both sides of every parity test: the host
generator (``libsynth_host.so``) and the device generator (``libsynth_dev.so``)
compile the same recipe (``csrc/synth_core.h``) and return the same bits.  The
module holds none of the guard's arithmetic (no attention, statistics,
detection or pruning): only hashing, normals, loop planting and rounding.

Workloads follow the paper's setting (long-context decode under a fixed KV
budget, Sec. 6.1) at the five benchmark shapes:

  1  tiny single-layer guard, fp32, literal planted loop of a 24-row block x8
  2  Llama-3-8B-shaped decode, 32 layers, 32/8 heads, bf16, b=8, n=8192, B=4096
  3  small-model long context, 28 layers, 12/2 heads, b=32, n=32768, B=8192, sinks
  4  ragged serving batch, b=64, n log-uniform in [1024, 65536], B=min(n+256, 16384)
  5  bandwidth sweep, 32 layers, 64/8 heads, b=16, n=131072, B=32768
  6  the paper's setting: Qwen3-1.7B shape, one 3853-token prompt, B=1024, T_max 2500

``make_workload(i, **overrides)`` returns one of them; overrides shrink a
workload for tests while keeping its structure.
"""
from __future__ import annotations

import ctypes
import math
import os
from dataclasses import dataclass, field

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
HOST_LIB = os.path.join(_HERE, "libsynth_host.so")
DEV_LIB = os.path.join(_HERE, "libsynth_dev.so")

NEVER = 0x7FFFFFFF
BF16, F32 = 0, 1
Q_ZSTAR, Q_LITERAL = 0, 1
M64 = (1 << 64) - 1


class SynWorkload(ctypes.Structure):
    _fields_ = [
        ("seed", ctypes.c_uint64),
        ("L", ctypes.c_int32), ("H_q", ctypes.c_int32), ("H_kv", ctypes.c_int32),
        ("d", ctypes.c_int32), ("dtype", ctypes.c_int32),
        ("head_scale", ctypes.c_int32), ("n_sink", ctypes.c_int32),
        ("sink_factor", ctypes.c_float), ("sigma", ctypes.c_float),
        ("query_mode", ctypes.c_int32), ("zstar", ctypes.c_float),
        ("q_noise", ctypes.c_float), ("pad", ctypes.c_int32),
    ]


SEQ_DTYPE = np.dtype([("looping", np.int32), ("start", np.int32),
                      ("period", np.int32), ("fresh_from", np.int32)])


def mix64(x: int) -> int:
    """splitmix64 finaliser on Python ints (host-side draws of workload shape)."""
    x = (x + 0x9E3779B97F4A7C15) & M64
    x = ((x ^ (x >> 30)) * 0xBF58476D1CE4E5B9) & M64
    x = ((x ^ (x >> 27)) * 0x94D049BB133111EB) & M64
    return x ^ (x >> 31)


def _u24(seed: int, tag: int, idx: int) -> int:
    return mix64(mix64(mix64(seed) ^ (0xC0FFEE00 + tag)) ^ idx) >> 40


def _uniform(seed: int, tag: int, idx: int) -> float:
    return _u24(seed, tag, idx) / float(1 << 24)


def _randint(seed: int, tag: int, idx: int, lo: int, hi: int) -> int:
    """uniform integer in [lo, hi], exact integer arithmetic"""
    return lo + ((_u24(seed, tag, idx) * (hi - lo + 1)) >> 24)


def _choose(seed: int, tag: int, batch: int, frac: float) -> np.ndarray:
    """exactly round(frac * batch) sequences, chosen by hash rank"""
    k = int(round(frac * batch))
    keys = [(_u24(seed, tag, b), b) for b in range(batch)]
    chosen = np.zeros(batch, dtype=bool)
    for _, b in sorted(keys)[:k]:
        chosen[b] = True
    return chosen


@dataclass
class Workload:
    name: str
    L: int
    H_q: int
    H_kv: int
    d: int
    dtype: str
    batch: int
    n0: np.ndarray
    budget: np.ndarray
    steps: int
    seed: int
    seqs: np.ndarray
    head_scale: int = 1
    n_sink: int = 0
    sink_factor: float = 1.0
    sigma: float = 0.02
    query_mode: int = Q_ZSTAR
    zstar: float = 12.0
    q_noise: float = 0.05
    cap: np.ndarray = field(default=None)
    seq_off: np.ndarray = field(default=None)
    S_total: int = 0
    note: str = ""

    def __post_init__(self):
        self.n0 = np.asarray(self.n0, dtype=np.int32)
        self.budget = np.asarray(self.budget, dtype=np.int32)
        if self.cap is None:
            # Length never exceeds max(n0, budget) + 1 under either policy; the
            # extra rows keep ungated runs (no pruning) valid for `steps` steps.
            self.cap = np.maximum(self.n0, self.budget) + self.steps + 1
        self.cap = np.asarray(self.cap, dtype=np.int32)
        self.seq_off = np.zeros(self.batch, dtype=np.int64)
        self.seq_off[1:] = np.cumsum(self.cap.astype(np.int64))[:-1]
        self.S_total = int(self.cap.astype(np.int64).sum())

    @property
    def g(self) -> int:
        return self.H_q // self.H_kv

    @property
    def esize(self) -> int:
        return 2 if self.dtype == "bf16" else 4

    @property
    def np_dtype(self):
        return np.uint16 if self.dtype == "bf16" else np.float32

    def c_struct(self) -> SynWorkload:
        return SynWorkload(
            seed=self.seed, L=self.L, H_q=self.H_q, H_kv=self.H_kv, d=self.d,
            dtype=BF16 if self.dtype == "bf16" else F32, head_scale=self.head_scale,
            n_sink=self.n_sink, sink_factor=self.sink_factor, sigma=self.sigma,
            query_mode=self.query_mode, zstar=self.zstar, q_noise=self.q_noise, pad=0)

    def kv_bytes(self) -> int:
        return 2 * self.L * self.H_kv * self.S_total * self.d * self.esize

    def describe(self) -> dict:
        return {"workload": self.name, "layers": self.L, "H_q": self.H_q, "H_kv": self.H_kv,
                "head_dim": self.d, "dtype": self.dtype, "batch": self.batch,
                "cache_len": int(self.n0.max()) if len(set(self.n0.tolist())) == 1 else
                "ragged %d..%d" % (self.n0.min(), self.n0.max()),
                "budget": int(self.budget.max()) if len(set(self.budget.tolist())) == 1 else
                "ragged", "decode_steps": self.steps,
                "looping_seqs": int(self.seqs["looping"].sum())}


def _seqs(batch):
    s = np.zeros(batch, dtype=SEQ_DTYPE)
    s["fresh_from"] = NEVER
    return s


def make_workload(i: int, **ov) -> Workload:
    """Benchmark workload i (1..6); keyword overrides shrink it for tests."""
    if i == 1:
        n = ov.get("n", 512)
        loop_len = ov.get("loop_len", 192)
        P = ov.get("period", 24)
        seqs = _seqs(1)
        seqs[0] = (1, n - loop_len, P, NEVER)
        return Workload(
            name=ov.get("name", "tiny single-layer guard: 1 layer, 8/8 heads, d=64, fp32, "
                        "b=1, n=%d, B=%d" % (n, ov.get("budget", 256))),
            L=1, H_q=8, H_kv=8, d=64, dtype="f32", batch=1, n0=[n],
            budget=[ov.get("budget", 256)], steps=ov.get("steps", 1), seed=ov.get("seed", 0),
            seqs=seqs, head_scale=0, sigma=0.1, query_mode=Q_LITERAL, q_noise=0.05)
    if i == 2:
        L = ov.get("L", 32); b = ov.get("batch", 8); n = ov.get("n", 8192)
        B = ov.get("budget", 4096); seed = ov.get("seed", 1)
        tail_lo, tail_hi = ov.get("tail", (1024, 3072))
        p_lo, p_hi = ov.get("periods", (16, 128))
        seqs = _seqs(b)
        looping = _choose(seed, 1, b, 0.5)
        for s in range(b):
            if looping[s]:
                P = _randint(seed, 2, s, p_lo, p_hi)
                tail = _randint(seed, 3, s, tail_lo, tail_hi)
                seqs[s] = (1, n - tail, P, NEVER)
        return Workload(
            name=ov.get("name", "Llama-3-8B-shaped decode: %d layers, 32/8 heads, d=128, bf16, "
                        "b=%d, n=%d, B=%d" % (L, b, n, B)),
            L=L, H_q=ov.get("H_q", 32), H_kv=ov.get("H_kv", 8), d=128, dtype="bf16", batch=b,
            n0=[n] * b, budget=[B] * b, steps=ov.get("steps", 64), seed=seed, seqs=seqs)
    if i == 3:
        L = ov.get("L", 28); b = ov.get("batch", 32); n = ov.get("n", 32768)
        B = ov.get("budget", 8192); seed = ov.get("seed", 2)
        p_lo, p_hi = ov.get("periods", (8, 64))
        seqs = _seqs(b)
        looping = _choose(seed, 1, b, 0.6)
        for s in range(b):
            if looping[s]:
                P = _randint(seed, 2, s, p_lo, p_hi)
                lo = (3 * n) // 4
                start = _randint(seed, 3, s, lo, max(lo, n - 4 * P))
                seqs[s] = (1, start, P, NEVER)
        return Workload(
            name=ov.get("name", "small-model long context: %d layers, 12/2 heads, d=128, bf16, "
                        "b=%d, n=%d, B=%d, sinks" % (L, b, n, B)),
            L=L, H_q=12, H_kv=2, d=128, dtype="bf16", batch=b, n0=[n] * b, budget=[B] * b,
            steps=ov.get("steps", 128), seed=seed, seqs=seqs, n_sink=4, sink_factor=8.0)
    if i == 4:
        L = ov.get("L", 32); b = ov.get("batch", 64); seed = ov.get("seed", 3)
        n_lo, n_hi = ov.get("len_range", (1024, 65536))
        bmax = ov.get("budget_max", 16384)
        onset_max = ov.get("onset_max", 200)
        p_lo, p_hi = ov.get("periods", (16, 64))
        n0 = []
        for s in range(b):
            u = _uniform(seed, 4, s)
            n0.append(int(math.floor(n_lo * (n_hi / n_lo) ** u)))
        n0 = np.array(n0, dtype=np.int32)
        budget = np.minimum(n0 + 256, bmax)
        seqs = _seqs(b)
        looping = _choose(seed, 1, b, 0.3)
        for s in range(b):
            if looping[s]:
                P = _randint(seed, 2, s, p_lo, p_hi)
                onset = _randint(seed, 3, s, 0, onset_max)
                seqs[s] = (1, int(n0[s]) + onset, P, NEVER)
        return Workload(
            name=ov.get("name", "ragged serving batch: %d layers, 32/8 heads, d=128, bf16, b=%d, "
                        "n log-uniform [%d, %d], B=min(n+256, %d)" % (L, b, n_lo, n_hi, bmax)),
            L=L, H_q=32, H_kv=8, d=128, dtype="bf16", batch=b, n0=n0, budget=budget,
            steps=ov.get("steps", 256), seed=seed, seqs=seqs)
    if i == 5:
        L = ov.get("L", 32); b = ov.get("batch", 16); n = ov.get("n", 131072)
        B = ov.get("budget", 32768); seed = ov.get("seed", 4)
        tail = ov.get("tail", 16384); P = ov.get("period", 32)
        seqs = _seqs(b)
        looping = _choose(seed, 1, b, 0.5)
        for s in range(b):
            if looping[s]:
                seqs[s] = (1, n - tail, P, NEVER)
        return Workload(
            name=ov.get("name", "bandwidth sweep: %d layers, 64/8 heads, d=128, bf16, b=%d, "
                        "n=%d, B=%d" % (L, b, n, B)),
            L=L, H_q=64, H_kv=8, d=128, dtype="bf16", batch=b, n0=[n] * b, budget=[B] * b,
            steps=ov.get("steps", 2), seed=seed, seqs=seqs)
    if i == 6:
        # The paper's own setting (Sec. 6.1, App. C): a 1-2B model (Qwen3-1.7B shape: 28 layers,
        # 16 query / 8 kv heads, d=128), a LoopBench-DC-length prompt (3853 tokens on average),
        # budget 1024, generation capped at T_max = 2500; one loop whose onset falls where
        # most of the paper's interventions happen (800-1300 generated tokens, Sec. 6.4, Fig. 4).
        b = ov.get("batch", 1); seed = ov.get("seed", 5)
        n = ov.get("n", 3853); B = ov.get("budget", 1024)
        L = ov.get("L", 28)
        on_lo, on_hi = ov.get("onset", (800, 1300))
        p_lo, p_hi = ov.get("periods", (16, 64))
        seqs = _seqs(b)
        for s in range(b):
            P = _randint(seed, 2, s, p_lo, p_hi)
            onset = _randint(seed, 3, s, on_lo, on_hi)
            seqs[s] = (1, n + onset, P, NEVER)
        return Workload(
            name=ov.get("name", "paper-shaped guard: Qwen3-1.7B shape (%d layers, 16/8 heads, "
                        "d=128), bf16, b=%d, prompt %d, B=%d, T_max 2500" % (L, b, n, B)),
            L=L, H_q=16, H_kv=8, d=128, dtype="bf16", batch=b, n0=[n] * b, budget=[B] * b,
            steps=ov.get("steps", 2500), seed=seed, seqs=seqs)
    raise ValueError("workload index must be 1..6")


# ----------------------------------------------------------------------------- host generator

_host = None


def host_lib():
    global _host
    if _host is None:
        if not os.path.exists(HOST_LIB):
            raise RuntimeError("libsynth_host.so missing: run __graft_entry__.build()")
        lib = ctypes.CDLL(HOST_LIB)
        vp, i32, i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
        lib.syn_host_rows.argtypes = [ctypes.POINTER(SynWorkload), vp, i32, i32, i32, i32, i64,
                                      i64, vp]
        lib.syn_host_fill_cache.argtypes = [ctypes.POINTER(SynWorkload), vp, i32, vp, vp, i64,
                                            vp, vp]
        lib.syn_host_step.argtypes = [ctypes.POINTER(SynWorkload), vp, i32, vp, vp, vp, vp]
        lib.syn_host_normals.argtypes = [ctypes.c_uint64, i32, i32, i32, i32, ctypes.c_uint64,
                                         i64, vp]
        lib.syn_host_mix.argtypes = [ctypes.c_uint64]
        lib.syn_host_mix.restype = ctypes.c_uint64
        _host = lib
    return _host


def _ptr(a: np.ndarray):
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data_as(ctypes.c_void_p)


def host_rows(w: Workload, is_value: int, layer: int, kvh: int, seq: int, p0: int, count: int,
              seqs: np.ndarray | None = None) -> np.ndarray:
    """rows [p0, p0+count) of one (layer, kv-head, sequence) stream, [count][d] cache dtype"""
    seqs = w.seqs if seqs is None else seqs
    out = np.empty((count, w.d), dtype=w.np_dtype)
    s = np.ascontiguousarray(seqs[seq:seq + 1])
    cw = w.c_struct()
    host_lib().syn_host_rows(ctypes.byref(cw), _ptr(s), is_value, layer, kvh, seq, p0, count,
                             _ptr(out))
    return out


def host_cache(w: Workload, n_rows: np.ndarray | None = None):
    """full K, V caches [L][H_kv][S_total][d] with rows [0, n_rows[b]) filled (rest zero)"""
    n_rows = w.n0 if n_rows is None else np.asarray(n_rows, dtype=np.int32)
    K = np.zeros((w.L, w.H_kv, w.S_total, w.d), dtype=w.np_dtype)
    V = np.zeros_like(K)
    cw = w.c_struct()
    s = np.ascontiguousarray(w.seqs)
    host_lib().syn_host_fill_cache(ctypes.byref(cw), _ptr(s), w.batch, _ptr(w.seq_off),
                                   _ptr(np.ascontiguousarray(n_rows)), w.S_total, _ptr(K), _ptr(V))
    return K, V


def host_step(w: Workload, pos: np.ndarray, seqs: np.ndarray | None = None):
    """q [L][b][H_q][d], k_new / v_new [L][b][H_kv][d] for the tokens at positions pos[b]"""
    seqs = w.seqs if seqs is None else seqs
    pos = np.ascontiguousarray(pos, dtype=np.int64)
    q = np.empty((w.L, w.batch, w.H_q, w.d), dtype=w.np_dtype)
    kn = np.empty((w.L, w.batch, w.H_kv, w.d), dtype=w.np_dtype)
    vn = np.empty_like(kn)
    cw = w.c_struct()
    host_lib().syn_host_step(ctypes.byref(cw), _ptr(np.ascontiguousarray(seqs)), w.batch,
                             _ptr(pos), _ptr(q), _ptr(kn), _ptr(vn))
    return q, kn, vn


def host_normals(seed: int, role: int, layer: int, head: int, seq: int, idx0: int,
                 count: int) -> np.ndarray:
    out = np.empty(count, dtype=np.float32)
    host_lib().syn_host_normals(seed, role, layer, head, seq, idx0, count, _ptr(out))
    return out


def note_interventions(seqs: np.ndarray, pos: np.ndarray, flags: np.ndarray) -> None:
    """After a step: a sequence the guard intervened on turns loop-free from the next token
    on (the paper reports diversity restored after pruning, Sec. 6.2)."""
    for b in range(len(seqs)):
        if flags[b] and seqs["fresh_from"][b] == NEVER:
            seqs["fresh_from"][b] = int(pos[b]) + 1


# ----------------------------------------------------------------------------- device generator

_dev = None


def dev_lib():
    global _dev
    if _dev is None:
        if not os.path.exists(DEV_LIB):
            raise RuntimeError("libsynth_dev.so missing: run __graft_entry__.build()")
        lib = ctypes.CDLL(DEV_LIB)
        vp, i32, i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
        lib.syn_dev_fill_cache.argtypes = [ctypes.POINTER(SynWorkload), vp, i32, vp, vp, i64, i32,
                                           vp, vp, vp]
        lib.syn_dev_step.argtypes = [ctypes.POINTER(SynWorkload), vp, i32, vp, i32, vp, vp, vp,
                                     vp]
        lib.syn_dev_select3.argtypes = [vp, i32, i32, i32, i32, vp, vp, vp, vp, vp, vp, vp, vp,
                                        vp, vp, vp]
        lib.syn_dev_read_stream.argtypes = [vp, i64, vp, i32, vp]
        lib.syn_dev_read_bulk.argtypes = [vp, i64, i32, vp, vp, i32, vp]
        for f in (lib.syn_dev_fill_cache, lib.syn_dev_step, lib.syn_dev_select3,
                  lib.syn_dev_read_stream, lib.syn_dev_read_bulk):
            f.restype = ctypes.c_int
        _dev = lib
    return _dev


def _check(rc, what):
    if rc != 0:
        raise RuntimeError("%s failed (%d)" % (what, rc))


def seqs_tensor(seqs: np.ndarray, device):
    import torch
    raw = np.ascontiguousarray(seqs).view(np.int32).reshape(-1, 4)
    return torch.from_numpy(raw.copy()).to(device)


def dev_fill_cache(w: Workload, K, V, seqs_dev, seq_off_dev, n_rows_dev, max_rows: int, stream):
    cw = w.c_struct()
    _check(dev_lib().syn_dev_fill_cache(ctypes.byref(cw), seqs_dev.data_ptr(), w.batch,
                                        seq_off_dev.data_ptr(), n_rows_dev.data_ptr(),
                                        w.S_total, max_rows, K.data_ptr(), V.data_ptr(), stream),
           "syn_dev_fill_cache")


def dev_step(w: Workload, seqs_dev, pos_dev, q, kn, vn, stream, mode: int = 0):
    cw = w.c_struct()
    _check(dev_lib().syn_dev_step(ctypes.byref(cw), seqs_dev.data_ptr(), w.batch,
                                  pos_dev.data_ptr(), mode, q.data_ptr(), kn.data_ptr(),
                                  vn.data_ptr(), stream), "syn_dev_step")


def dev_read_stream(buf, sink, ctas: int, stream):
    """one read-only pass over the bytes of device tensor buf (harness: the read-only bandwidth
    denominator of bench.py); sink is a one-word int32 device tensor"""
    _check(dev_lib().syn_dev_read_stream(buf.data_ptr(), buf.numel() * buf.element_size(),
                                         sink.data_ptr(), ctas, stream), "syn_dev_read_stream")


def dev_read_bulk(buf, block: int, sink, err, ctas: int, stream):
    """the same read-only pass with 1-D bulk copies of `block` bytes into shared memory; err is
    a one-word int32 device tensor, set when a wait timed out"""
    _check(dev_lib().syn_dev_read_bulk(buf.data_ptr(), buf.numel() * buf.element_size(), block,
                                       sink.data_ptr(), err.data_ptr(), ctas, stream),
           "syn_dev_read_bulk")


TOKEN_VOCAB = 50_000


def _token_at(seed: int, seq: int, pos: int) -> int:
    return (mix64(mix64(seed ^ 0x70C3E5) ^ (seq << 32) ^ pos) >> 40) % TOKEN_VOCAB


def _pmax_at(seed: int, seq: int, pos: int) -> float:
    return 0.2 + 0.6 * ((mix64(mix64(seed ^ 0x9B1A) ^ (seq << 32) ^ pos) >> 40) / float(1 << 24))


def token_streams(w: Workload, steps: int):
    """Generated token ids and top-1 probabilities of every step, for a caller of the
    token-level monitor, in the two variants the decode inputs have: (tok_loop, tok_fresh,
    pm_loop, pm_fresh), each [steps][batch].  A healthy token is a hash of (sequence,
    position) over a 50 000-token vocabulary with p_max in [0.2, 0.8); a sequence inside its
    planted loop (position >= start) repeats the `period` tokens before the start, with
    p_max 0.95, in the loop-continuing variant."""
    tl = np.zeros((steps, w.batch), dtype=np.int32)
    tf = np.zeros_like(tl)
    pl = np.zeros((steps, w.batch), dtype=np.float32)
    pf = np.zeros_like(pl)
    for b in range(w.batch):
        sq = w.seqs[b]
        for t in range(steps):
            pos = int(w.n0[b]) + t
            tf[t, b] = _token_at(w.seed, b, pos)
            pf[t, b] = _pmax_at(w.seed, b, pos)
            if sq["looping"] and pos >= sq["start"]:
                P = int(sq["period"])
                src = int(sq["start"]) - P + (pos - int(sq["start"])) % P
                tl[t, b] = _token_at(w.seed, b, src)
                pl[t, b] = 0.95
            else:
                tl[t, b] = tf[t, b]
                pl[t, b] = pf[t, b]
    return tl, tf, pl, pf


class Select3:
    """one launch that picks each sequence's inputs of a step (q, k_new, v_new) from the
    loop-continuing or the loop-free variant: the loop-free one once the guard has intervened on
    the sequence (its state's intervention count, word n_int_word of each state_words-word
    record, is positive; the paper reports diversity restored after pruning, Sec. 6.2); with no
    state (the comparator policies) loops persist.  Argument arrays marshalled once."""

    def __init__(self, w, state, state_words, n_int_word, outs, rowlens):
        self.w = w
        self.state = None if state is None else state.data_ptr()
        self.state_words, self.n_int_word = state_words, n_int_word
        self.rowlens = (ctypes.c_int64 * 3)(*rowlens)
        self.outs = (ctypes.c_void_p * 3)(*[o.data_ptr() for o in outs])
        self.loop = (ctypes.c_void_p * 3)()
        self.fresh = (ctypes.c_void_p * 3)()

    def __call__(self, loop_bufs, fresh_bufs, stream, tokens=None):
        """tokens: None, or (tok_loop, tok_fresh, pm_loop, pm_fresh, tok, pm), [batch] each:
        the same launch also picks each sequence's token id and top-1 probability"""
        for k in range(3):
            self.loop[k] = loop_bufs[k].data_ptr()
            self.fresh[k] = fresh_bufs[k].data_ptr()
        tk = [None] * 6 if tokens is None else [x.data_ptr() for x in tokens]
        _check(dev_lib().syn_dev_select3(self.state, self.state_words, self.n_int_word,
                                         self.w.batch, self.w.L, self.rowlens, self.loop,
                                         self.fresh, self.outs, *tk, stream), "syn_dev_select3")


def build(out_dir: str = _HERE, jobs=None):
    """Compile the host generator (g++) and the device generator (nvcc, sm_103a).
    Returns the list of subprocess handles so a caller can run builds in parallel."""
    import subprocess
    src = os.path.join(_HERE, "csrc")
    procs = []
    procs.append(subprocess.Popen(
        ["g++", "-O2", "-std=c++17", "-ffp-contract=off", "-fopenmp", "-shared", "-fPIC",
         os.path.join(src, "synth_host.cpp"), "-o", HOST_LIB]))
    procs.append(subprocess.Popen(
        ["nvcc", "-gencode", "arch=compute_103a,code=sm_103a", "-O3", "--fmad=false",
         "-lineinfo", "-Xcompiler", "-fPIC", "-shared", os.path.join(src, "synth_dev.cu"),
         "-o", DEV_LIB]))
    return procs
