"""CPU oracle for the LoopGuard decode path -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
``--impl reference`` legs of ``bench.py`` may import this package.  The
product path (``paper_2604_10044_gb300``) never does, and the two share no
code: this package wraps ``liblgref.so`` (plain C, fp64, ``lgref.c``) and
orchestrates it step by step in the paper's order:

  append the step's row -> attention over the retained set (Sec. 3.1, Eq. 1)
  -> loop-onset test (Sec. 5.2, Eq. 8, Eq. 9) -> I_keep and index-gather
  (Sec. 5.3, Eq. 10, Eq. 11); or, on the comparator path, H2O eviction
  (Sec. 2.2, Sec. 6.1).

Parity pins (closed forms, brute force, invariants) are in
``tests/test_oracle_*.py``.  Every function here is pinned there; none is
"parity unpinned".
"""
from __future__ import annotations

import ctypes
import math
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "liblgref.so")


class Params(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in (
        "W", "K", "t_min", "cooldown", "n_anchor", "stall_len", "p_min", "p_max", "l_min",
        "m_rep", "suffix_w", "guard_layer", "level_max", "retrig_window", "headroom", "pad")] + \
        [(n, ctypes.c_double) for n in ("theta_ttr", "theta_nov", "theta_ent", "theta_lift",
                                         "tau_ham")]


class State(ctypes.Structure):
    _fields_ = [("t_gen", ctypes.c_int32), ("cd", ctypes.c_int32), ("level", ctypes.c_int32),
                ("last_trig", ctypes.c_int32), ("n_int", ctypes.c_int32),
                ("pad", ctypes.c_int32 * 3)]


# Paper constants (App. B.2, Sec. 6.1) and, where the paper is silent, the readings taken here.
DEFAULTS = dict(W=256, K=2, t_min=64, cooldown=32, n_anchor=32, stall_len=4, p_min=1, p_max=128,
                l_min=32, m_rep=3, suffix_w=64, guard_layer=0, level_max=3, retrig_window=64,
                headroom=64, theta_ttr=0.2, theta_nov=0.02, theta_ent=0.7, theta_lift=2.0,
                tau_ham=0.125)

NEVER_TRIGGERED = -(1 << 30)


class TokenParams(ctypes.Structure):
    _fields_ = [("cr_every", ctypes.c_int32), ("theta_streak", ctypes.c_int32),
                ("hist", ctypes.c_int32), ("pad", ctypes.c_int32),
                ("theta_cr", ctypes.c_double), ("theta_conf", ctypes.c_double)]


class TokenState(ctypes.Structure):
    _fields_ = [("streak", ctypes.c_int32), ("synced", ctypes.c_int32),
                ("appended", ctypes.c_int32), ("pad", ctypes.c_int32), ("cr", ctypes.c_double)]


# App. B.2 thresholds of the token-level monitor; the paper fixes neither cr_every nor hist.
TOKEN_DEFAULTS = dict(cr_every=16, theta_streak=6, hist=512, theta_cr=0.12, theta_conf=0.9)


def token_params(**over) -> TokenParams:
    d = dict(TOKEN_DEFAULTS)
    d.update(over)
    return TokenParams(**d)


def new_token_state() -> TokenState:
    return TokenState(streak=0, synced=-1, appended=0, pad=0, cr=1.0)


def params(**over) -> Params:
    d = dict(DEFAULTS)
    d.update(over)
    return Params(**d)


def new_state(t_gen: int = 64) -> State:
    return State(t_gen=t_gen, cd=0, level=0, last_trig=NEVER_TRIGGERED, n_int=0)


def build():
    """Compile liblgref.so with gcc (OpenMP when available).  Returns a Popen handle."""
    src = os.path.join(_HERE, "lgref.c")
    cmd = ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fopenmp", "-shared", "-fPIC", src,
           "-o", LIB_PATH, "-lm"]
    return subprocess.Popen(cmd)


_lib = None


def lib():
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError("liblgref.so missing: run __graft_entry__.build()")
        L = ctypes.CDLL(LIB_PATH)
        vp, i32, i64, dbl = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_double
        L.lgref_attend_group.argtypes = [i32, i32, i32, vp, vp, i32, vp, dbl, i32, vp, vp, vp]
        L.lgref_attend_all.argtypes = [i32, i32, i32, i32, i32, i32, i64, vp, vp, vp, vp, vp, dbl,
                                       i32, vp, vp, vp]
        L.lgref_sketch.argtypes = [i32, i32, vp, vp]
        L.lgref_sketch.restype = None
        L.lgref_match.argtypes = [vp, vp, i32, i32]
        L.lgref_detect.argtypes = [i32, i32, vp, i32, vp, i32, i32, ctypes.POINTER(Params),
                                   ctypes.POINTER(State), vp, vp, vp]
        L.lgref_keep_set.argtypes = [i32, i32, i32, i32, i32, i32, ctypes.POINTER(Params), vp]
        L.lgref_compact_rows.argtypes = [vp, ctypes.c_size_t, vp, i32]
        L.lgref_compact_rows.restype = None
        L.lgref_h2o_select.argtypes = [i32, vp, vp, i32, ctypes.c_int32, vp]
        L.lgref_h2o_argmin.argtypes = [i32, vp, vp, i32, ctypes.c_int32]
        L.lgref_streaming_select.argtypes = [i32, vp, i32, i32, ctypes.c_int32, vp]
        L.lgref_streaming_oldest.argtypes = [i32, vp, i32]
        L.lgref_lz77_phrases.argtypes = [vp, i32]
        L.lgref_token_detect.argtypes = [vp, i32, dbl, i32, vp, i32, ctypes.POINTER(Params),
                                         ctypes.POINTER(TokenParams), ctypes.POINTER(State),
                                         ctypes.POINTER(TokenState), vp, vp, vp]
        _lib = L
    return _lib


def _p(a: np.ndarray):
    assert a.flags["C_CONTIGUOUS"], "array must be C-contiguous"
    return a.ctypes.data_as(ctypes.c_void_p)


def _dt(a: np.ndarray) -> int:
    if a.dtype == np.uint16:
        return 0
    if a.dtype == np.float32:
        return 1
    raise TypeError("cache arrays are bf16 bits (uint16) or float32")


# ------------------------------------------------------------------ single functions

def attend_group(q, K, V, scale=None, suffix_w=64, want_alpha=False):
    """Eq. 1 for g query heads over one kv-head's n rows.
    q [g][d], K/V [n][d] (uint16 bf16 bits or float32).  Returns out [g][d], stats [g][4]
    (m, l, H, S) and alpha [g][n] (or None)."""
    q, K, V = (np.ascontiguousarray(x) for x in (q, K, V))
    g, d = q.shape
    n = K.shape[0]
    scale = 1.0 / math.sqrt(d) if scale is None else scale
    out = np.zeros((g, d))
    stats = np.zeros((g, 4))
    alpha = np.zeros((g, n)) if want_alpha else None
    rc = lib().lgref_attend_group(_dt(K), d, n, _p(K), _p(V), g, _p(q), scale, suffix_w,
                                  _p(out), _p(stats), None if alpha is None else _p(alpha))
    if rc:
        raise ValueError("lgref_attend_group rejected its arguments")
    return out, stats, alpha


def sketch(row) -> np.ndarray:
    row = np.ascontiguousarray(row).reshape(-1)
    words = np.zeros(row.size // 32, dtype=np.uint32)
    lib().lgref_sketch(_dt(row), row.size, _p(row), _p(words))
    return words


def match(a, b, thr) -> bool:
    a = np.ascontiguousarray(a, dtype=np.uint32)
    b = np.ascontiguousarray(b, dtype=np.uint32)
    return bool(lib().lgref_match(_p(a), _p(b), a.size, thr))


def detect(stats, sketches, budget, prm: Params, st: State):
    """Loop-onset test for one sequence.  stats [L][H_q][4] (float64), sketches [n][nwords].
    Returns (flag, (lo, hi), diag dict); st is updated in place."""
    stats = np.ascontiguousarray(stats, dtype=np.float64)
    sk = np.ascontiguousarray(sketches, dtype=np.uint32)
    L, H_q = stats.shape[0], stats.shape[1]
    n, nwords = sk.shape
    flag = np.zeros(1, dtype=np.int32)
    span = np.zeros(2, dtype=np.int32)
    diag = np.zeros(10)
    rc = lib().lgref_detect(L, H_q, _p(stats), n, _p(sk) if n else None, nwords, int(budget),
                            ctypes.byref(prm), ctypes.byref(st), _p(flag), _p(span), _p(diag))
    if rc:
        raise ValueError("lgref_detect rejected its arguments")
    keys = ("ebar", "lbar", "ttr", "sig1", "sig2", "sig3", "warn", "stall", "P", "trigger")
    return int(flag[0]), (int(span[0]), int(span[1])), dict(zip(keys, diag.tolist()))


def lz77_phrases(x) -> int:
    """phrases of the greedy LZ77 parse of a token sequence (Sec. 4.3's comp(), read as LZ77)"""
    x = np.ascontiguousarray(x, dtype=np.int32)
    return int(lib().lgref_lz77_phrases(_p(x), x.size))


TOKEN_DIAG_KEYS = ("ttr", "cr", "streak", "sig1", "sig2", "sig3", "warn", "stall", "P", "trigger")


def token_detect(tokens, pmax, n, prm: Params, tp: TokenParams, st: State, ts: TokenState,
                 kept=None):
    """Token-level monitor for one sequence and one step: tokens = every generated token so far
    (the last is this step's), pmax this step's top-1 probability, n the cache length after the
    step's append, kept the retained slots of the prune after the previous step (None if there
    was none).  Returns (flag, (lo, hi) in cache slots, diag dict); st, ts updated."""
    y = np.ascontiguousarray(tokens, dtype=np.int32)
    flag = np.zeros(1, dtype=np.int32)
    span = np.zeros(2, dtype=np.int32)
    diag = np.zeros(10)
    k = None if kept is None else np.ascontiguousarray(kept, dtype=np.int32)
    rc = lib().lgref_token_detect(_p(y), y.size, float(pmax), int(n),
                                  None if k is None or k.size == 0 else _p(k),
                                  -1 if k is None else int(k.size), ctypes.byref(prm), ctypes.byref(tp), ctypes.byref(st),
                                  ctypes.byref(ts), _p(flag), _p(span), _p(diag))
    if rc:
        raise ValueError("lgref_token_detect rejected its arguments")
    return int(flag[0]), (int(span[0]), int(span[1])), dict(zip(TOKEN_DIAG_KEYS, diag.tolist()))


def keep_set(n, budget, flag, span, level, prm: Params) -> np.ndarray:
    kept = np.zeros(max(n, 1), dtype=np.int32)
    c = lib().lgref_keep_set(int(n), int(budget), int(flag), int(span[0]), int(span[1]),
                             int(level), ctypes.byref(prm), _p(kept))
    if c < 0:
        raise ValueError("lgref_keep_set: budget too small")
    return kept[:c].copy()


def compact_rows(rows: np.ndarray, kept: np.ndarray) -> None:
    """in place: rows[j] <- rows[kept[j]]; rows is a C-contiguous view [n][...]"""
    kept = np.ascontiguousarray(kept, dtype=np.int32)
    row_bytes = rows[0].nbytes if rows.shape[0] else 0
    lib().lgref_compact_rows(_p(rows), row_bytes, _p(kept), kept.size)


def h2o_select(score, pos, budget, pos_now) -> np.ndarray:
    score = np.ascontiguousarray(score, dtype=np.float64)
    pos = np.ascontiguousarray(pos, dtype=np.int32)
    kept = np.zeros(max(score.size, 1), dtype=np.int32)
    c = lib().lgref_h2o_select(score.size, _p(score), _p(pos), int(budget), int(pos_now),
                               _p(kept))
    return kept[:c].copy()


def h2o_argmin(score, pos, budget, pos_now) -> int:
    score = np.ascontiguousarray(score, dtype=np.float64)
    pos = np.ascontiguousarray(pos, dtype=np.int32)
    return int(lib().lgref_h2o_argmin(score.size, _p(score), _p(pos), int(budget), int(pos_now)))


def streaming_select(pos, budget, n_sink, pos_now) -> np.ndarray:
    pos = np.ascontiguousarray(pos, dtype=np.int32)
    kept = np.zeros(max(pos.size, 1), dtype=np.int32)
    c = lib().lgref_streaming_select(pos.size, _p(pos), int(budget), int(n_sink), int(pos_now),
                                     _p(kept))
    return kept[:c].copy()


def streaming_oldest(pos, n_sink) -> int:
    pos = np.ascontiguousarray(pos, dtype=np.int32)
    return int(lib().lgref_streaming_oldest(pos.size, _p(pos), int(n_sink)))


N_SINK = 4   # StreamingLLM attention sinks (the paper does not state the count)


# ------------------------------------------------------------------ full decode step

class OracleGuard:
    """The whole per-step path on host arrays laid out like the device cache:
    K, V [L][H_kv][S_total][d]; sketches [S_total][H_kv*d/32] of the guard layer's V rows;
    per-sequence lengths, guard state; H2O scores and positions [L][H_kv][S_total].

    policy: 'loopguard' (detect + I_keep), 'h2o' (accumulated-score eviction), 'streaming'
    (attention sinks + sliding window) or 'full' (no eviction)."""

    def __init__(self, w, K, V, prm: Params | None = None, policy="loopguard", t_gen0=64,
                 threads=None):
        self.w = w
        self.prm = prm or params()
        self.policy = policy
        self.K = np.ascontiguousarray(K)
        self.V = np.ascontiguousarray(V)
        self.len = w.n0.astype(np.int32).copy()
        self.cap = w.cap.astype(np.int32)
        self.off = w.seq_off.astype(np.int64)
        self.nwords = w.H_kv * w.d // 32
        self.sk = np.zeros((w.S_total, self.nwords), dtype=np.uint32)
        for b in range(w.batch):
            for i in range(int(self.len[b])):
                self.sk[self.off[b] + i] = self._row_sketch(b, i)
        self.state = [new_state(t_gen0) for _ in range(w.batch)]
        self.h2o = None
        self.pos = None
        if policy in ("h2o", "streaming"):
            self.h2o = np.zeros((w.L, w.H_kv, w.S_total))
            self.pos = np.zeros((w.L, w.H_kv, w.S_total), dtype=np.int32)
            for b in range(w.batch):
                n = int(self.len[b])
                self.pos[:, :, self.off[b]:self.off[b] + n] = np.arange(n, dtype=np.int32)
        if threads is not None:
            os.environ["OMP_NUM_THREADS"] = str(threads)

    def _row_sketch(self, b, i):
        gl = self.prm.guard_layer
        row = self.V[gl, :, self.off[b] + i, :]
        return sketch(np.ascontiguousarray(row))

    def attend(self, q):
        """Eq. 1 over every layer for the current lengths; returns out, stats (float64)"""
        w = self.w
        q = np.ascontiguousarray(q)
        out = np.zeros((w.L, w.batch, w.H_q, w.d))
        stats = np.zeros((w.L, w.batch, w.H_q, 4))
        threads = lib().lgref_attend_all(
            _dt(self.K), w.L, w.H_kv, w.H_q, w.d, w.batch, w.S_total, _p(self.off), _p(self.len),
            _p(self.K), _p(self.V), _p(q), 1.0 / math.sqrt(w.d), self.prm.suffix_w, _p(out),
            _p(stats), None if self.h2o is None else _p(self.h2o))
        if threads < 0:
            raise ValueError("lgref_attend_all rejected its arguments")
        self.threads = threads
        return out, stats

    def append(self, kn, vn, pos_new=None):
        w = self.w
        for b in range(w.batch):
            if self.len[b] + 1 > self.cap[b]:
                raise RuntimeError("sequence %d over capacity" % b)
            slot = self.off[b] + self.len[b]
            self.K[:, :, slot, :] = kn[:, b]
            self.V[:, :, slot, :] = vn[:, b]
            self.len[b] += 1
            self.sk[slot] = self._row_sketch(b, int(self.len[b]) - 1)
            if self.h2o is not None:
                self.h2o[:, :, slot] = 0.0
                self.pos[:, :, slot] = pos_new[b]

    def detect_all(self, stats, budget=None, seqs=None):
        w = self.w
        budget = w.budget if budget is None else budget
        seqs = range(w.batch) if seqs is None else seqs
        flags = np.zeros(w.batch, dtype=np.int32)
        spans = np.zeros((w.batch, 2), dtype=np.int32)
        diags = [None] * w.batch
        for b in seqs:
            n = int(self.len[b])
            sk = self.sk[self.off[b]:self.off[b] + n]
            f, sp, dg = detect(stats[:, b], sk, budget[b], self.prm, self.state[b])
            flags[b], spans[b], diags[b] = f, sp, dg
        return flags, spans, diags

    def prune(self, flags, spans, budget=None):
        """I_keep per sequence and the index-gather of K, V and sketches (Sec. 5.3)"""
        w = self.w
        budget = w.budget if budget is None else budget
        kept_all = []
        for b in range(w.batch):
            n = int(self.len[b])
            kept = keep_set(n, budget[b], flags[b], spans[b], self.state[b].level, self.prm)
            kept_all.append(kept)
            if len(kept) == n:
                continue
            o = self.off[b]
            for layer in range(w.L):
                for kvh in range(w.H_kv):
                    compact_rows(self.K[layer, kvh, o:o + n], kept)
                    compact_rows(self.V[layer, kvh, o:o + n], kept)
            compact_rows(self.sk[o:o + n], kept)
            self.len[b] = len(kept)
        return kept_all

    def h2o_evict(self, pos_now, budget=None):
        """H2O comparator after a step: one swap-remove per (layer, kv-head) when one row over
        budget, else a cut to the budget keeping recent + heavy rows in slot order."""
        w = self.w
        budget = w.budget if budget is None else budget
        events = {}
        for b in range(w.batch):
            n = int(self.len[b])
            B = int(budget[b])
            if n <= B:
                continue
            o = self.off[b]
            for layer in range(w.L):
                for kvh in range(w.H_kv):
                    sc = self.h2o[layer, kvh, o:o + n]
                    ps = self.pos[layer, kvh, o:o + n]
                    if n == B + 1:
                        x = h2o_argmin(sc, ps, B, pos_now[b])
                        events[(b, layer, kvh)] = x
                        if x != n - 1:
                            for arr in (self.K, self.V):
                                arr[layer, kvh, o + x] = arr[layer, kvh, o + n - 1]
                            sc[x] = sc[n - 1]
                            ps[x] = ps[n - 1]
                    else:
                        kept = h2o_select(sc, ps, B, pos_now[b])
                        events[(b, layer, kvh)] = kept
                        compact_rows(self.K[layer, kvh, o:o + n], kept)
                        compact_rows(self.V[layer, kvh, o:o + n], kept)
                        sc[:len(kept)] = sc[kept].copy()
                        ps[:len(kept)] = ps[kept].copy()
            self.len[b] = B
        return events

    def streaming_evict(self, pos_now, budget=None, n_sink=N_SINK):
        """StreamingLLM comparator after a step: sinks + the most recent positions; one
        swap-remove per (layer, kv-head) when one row over budget, else an ordered cut"""
        w = self.w
        budget = w.budget if budget is None else budget
        for b in range(w.batch):
            n, B, o = int(self.len[b]), int(budget[b]), self.off[b]
            if n <= B:
                continue
            for layer in range(w.L):
                for kvh in range(w.H_kv):
                    ps = self.pos[layer, kvh, o:o + n]
                    if n == B + 1:
                        x = streaming_oldest(ps, n_sink)
                        if x != n - 1:
                            for arr in (self.K, self.V):
                                arr[layer, kvh, o + x] = arr[layer, kvh, o + n - 1]
                            ps[x] = ps[n - 1]
                    else:
                        kept = streaming_select(ps, B, n_sink, pos_now[b])
                        compact_rows(self.K[layer, kvh, o:o + n], kept)
                        compact_rows(self.V[layer, kvh, o:o + n], kept)
                        ps[:len(kept)] = ps[kept].copy()
            self.len[b] = B
        return None

    def step(self, q, kn, vn, pos_new, budget=None):
        """one decode step: append, attend (Eq. 1), then the policy's cache update"""
        self.append(kn, vn, pos_new)
        out, stats = self.attend(q)
        res = dict(out=out, stats=stats)
        if self.policy == "loopguard":
            flags, spans, diags = self.detect_all(stats, budget)
            res.update(flags=flags, spans=spans, diags=diags,
                       kept=self.prune(flags, spans, budget))
        elif self.policy == "h2o":
            res.update(events=self.h2o_evict(pos_new, budget))
        elif self.policy == "streaming":
            res.update(events=self.streaming_evict(pos_new, budget))
        res["len"] = self.len.copy()
        return res
