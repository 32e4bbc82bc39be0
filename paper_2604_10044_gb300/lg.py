"""Python binding of liblg.so (include/lg.h): argument marshalling only.

Every function named ``lg_*`` here calls the C function of the same name with raw device
pointers taken from torch tensors and the caller's CUDA stream; every step of the decode path
runs in the library's kernels.  ``Cache`` and ``Guard`` bundle the device buffers of one batch
and issue a whole guarded decode step in the order the ABI documents.  There is no CPU path:
loading fails loudly when the shared library is missing.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np
import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "liblg.so")

LG_OK, LG_BF16, LG_F32 = 0, 0, 1
STATUS = {0: "LG_OK", 1: "LG_ERR_INVALID_ARG", 2: "LG_ERR_UNSUPPORTED", 3: "LG_ERR_CUDA",
          4: "LG_ERR_CAPACITY", 5: "LG_ERR_TIMEOUT", 6: "LG_ERR_WORKSPACE", 7: "LG_ERR_BUDGET"}


class LgError(RuntimeError):
    def __init__(self, fn, code):
        super().__init__("%s -> %s" % (fn, STATUS.get(code, code)))
        self.code = code


class LgCache(ctypes.Structure):
    _fields_ = [("k", ctypes.c_void_p), ("v", ctypes.c_void_p), ("dtype", ctypes.c_int32),
                ("L", ctypes.c_int32), ("H_kv", ctypes.c_int32), ("d", ctypes.c_int32),
                ("batch", ctypes.c_int32), ("pad", ctypes.c_int32), ("S_total", ctypes.c_int64),
                ("seq_off", ctypes.c_void_p), ("cap", ctypes.c_void_p), ("len", ctypes.c_void_p),
                ("sketch", ctypes.c_void_p), ("h2o", ctypes.c_void_p), ("pos", ctypes.c_void_p),
                ("dev_status", ctypes.c_void_p)]


class LgGuardParams(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in (
        "W", "K", "t_min", "cooldown", "n_anchor", "stall_len", "p_min", "p_max", "l_min",
        "m_rep", "suffix_w", "guard_layer", "level_max", "retrig_window", "headroom", "pad")] + \
        [(n, ctypes.c_double) for n in ("theta_ttr", "theta_nov", "theta_ent", "theta_lift",
                                         "tau_ham")]


class LgTokenParams(ctypes.Structure):
    _fields_ = [("cr_every", ctypes.c_int32), ("theta_streak", ctypes.c_int32),
                ("hist", ctypes.c_int32), ("pad", ctypes.c_int32),
                ("theta_cr", ctypes.c_double), ("theta_conf", ctypes.c_double)]


STATE_BYTES = 32  # lg_guard_state: 8 x int32
STATE_WORD_N_INT = 4  # lg_guard_state.n_int: interventions so far

_lib = None


def lib():
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError("liblg.so is not built (run __graft_entry__.build()); "
                               "there is no fallback path")
        L = ctypes.CDLL(LIB_PATH)
        vp, i32, i64, P = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.POINTER
        sig = {
            "lg_default_params": [P(LgGuardParams)],
            "lg_workspace_size": [P(LgCache), i32, i32, i32, i32],
            "lg_state_init": [P(LgCache), vp, i32, vp],
            "lg_begin_step": [P(LgCache), vp],
            "lg_append": [P(LgCache), i32, i32, vp, vp, vp, P(LgGuardParams), vp],
            "lg_sketch_build": [P(LgCache), P(LgGuardParams), i32, vp],
            "lg_decode_attend": [P(LgCache), i32, i32, vp, i32, ctypes.c_float, vp, vp, i32, i32,
                                 i32, vp, ctypes.c_size_t, vp],
            "lg_detect": [P(LgCache), vp, i32, vp, vp, P(LgGuardParams), vp, vp, vp, vp, vp],
            "lg_detect_state_size": [P(LgCache), P(LgGuardParams)],
            "lg_detect_prune": [P(LgCache), vp, i32, vp, vp, P(LgGuardParams), vp, vp, vp, vp,
                                vp, vp, i32, i32, vp],
            "lg_default_token_params": [P(LgTokenParams)],
            "lg_token_state_size": [P(LgCache), P(LgGuardParams), P(LgTokenParams)],
            "lg_token_detect": [P(LgCache), vp, vp, vp, vp, i32, vp, P(LgGuardParams),
                                P(LgTokenParams), vp, vp, vp, vp, vp],
            "lg_token_detect_prune": [P(LgCache), vp, vp, vp, vp, P(LgGuardParams),
                                      P(LgTokenParams), vp, vp, vp, vp, vp, vp, i32, i32, vp],
            "lg_prune_compact": [P(LgCache), vp, vp, vp, vp, P(LgGuardParams), vp, vp, i32, i32,
                                 vp],
            "lg_h2o_reset": [P(LgCache), i32, vp],
            "lg_h2o_evict": [P(LgCache), vp, vp, i32, vp],
            "lg_streaming_evict": [P(LgCache), vp, vp, i32, i32, vp],
            "lg_read_device_status": [P(LgCache), vp, vp],
            "lg_decode_attend_noalloc": [P(LgCache), i32, i32, vp, i32, ctypes.c_float, vp, vp,
                                         i32, i32, i32, vp],
            "lg_status_string": [i32],
        }
        for name, args in sig.items():
            f = getattr(L, name)
            f.argtypes = args
            f.restype = ctypes.c_int
        L.lg_workspace_size.restype = ctypes.c_size_t
        L.lg_detect_state_size.restype = ctypes.c_size_t
        L.lg_token_state_size.restype = ctypes.c_size_t
        L.lg_status_string.restype = ctypes.c_char_p
        _lib = L
    return _lib


def exported_symbols():
    """names of the C ABI functions declared in include/lg.h"""
    return ["lg_default_params", "lg_status_string", "lg_workspace_size", "lg_state_init",
            "lg_begin_step", "lg_append", "lg_sketch_build", "lg_decode_attend", "lg_detect",
            "lg_prune_compact", "lg_h2o_reset", "lg_h2o_evict", "lg_read_device_status",
            "lg_decode_attend_noalloc", "lg_detect_state_size", "lg_streaming_evict",
            "lg_detect_prune", "lg_default_token_params", "lg_token_state_size",
            "lg_token_detect", "lg_token_detect_prune"]

NOALLOC_SCRATCH_BYTES = 32 << 20  # LG_NOALLOC_SCRATCH_BYTES in include/lg.h


def _ptr(t):
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(stream):
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _call(name, *args):
    rc = getattr(lib(), name)(*args)
    if rc != LG_OK:
        raise LgError(name, rc)


# ------------------------------------------------------------------ thin wrappers, same names

def lg_default_params(**over) -> LgGuardParams:
    p = LgGuardParams()
    _call("lg_default_params", ctypes.byref(p))
    for k, v in over.items():
        setattr(p, k, v)
    return p


def lg_status_string(code: int) -> str:
    return lib().lg_status_string(code).decode()


def lg_workspace_size(cache, H_q, n_layers, max_len, accumulate_h2o=0) -> int:
    return int(lib().lg_workspace_size(ctypes.byref(cache.c), H_q, n_layers, max_len,
                                       accumulate_h2o))


def lg_state_init(cache, state, t_gen0=64, stream=None):
    _call("lg_state_init", ctypes.byref(cache.c), _ptr(state), t_gen0, _stream(stream))


def lg_begin_step(cache, stream=None):
    _call("lg_begin_step", ctypes.byref(cache.c), _stream(stream))


def lg_append(cache, layer0, n_layers, k_new, v_new, pos_new, params, stream=None):
    _call("lg_append", ctypes.byref(cache.c), layer0, n_layers, _ptr(k_new), _ptr(v_new),
          _ptr(pos_new), ctypes.byref(params), _stream(stream))


def lg_sketch_build(cache, params, max_len, stream=None):
    _call("lg_sketch_build", ctypes.byref(cache.c), ctypes.byref(params), max_len,
          _stream(stream))


def lg_decode_attend(cache, layer0, n_layers, q, H_q, scale, out, stats, suffix_w,
                     accumulate_h2o, max_len, ws, stream=None):
    _call("lg_decode_attend", ctypes.byref(cache.c), layer0, n_layers, _ptr(q), H_q,
          float(scale), _ptr(out), _ptr(stats), suffix_w, accumulate_h2o, max_len, _ptr(ws),
          ws.numel() * ws.element_size(), _stream(stream))


def lg_decode_attend_noalloc(cache, layer0, n_layers, q, H_q, scale, out, stats, suffix_w,
                             accumulate_h2o, max_len, stream=None):
    """lg_decode_attend with the library's own static scratch (no workspace argument)"""
    _call("lg_decode_attend_noalloc", ctypes.byref(cache.c), layer0, n_layers, _ptr(q), H_q,
          float(scale), _ptr(out), _ptr(stats), suffix_w, accumulate_h2o, max_len,
          _stream(stream))


def lg_detect_state_size(cache, params) -> int:
    return int(lib().lg_detect_state_size(ctypes.byref(cache.c), ctypes.byref(params)))


def lg_default_token_params(**over) -> LgTokenParams:
    tp = LgTokenParams()
    _call("lg_default_token_params", ctypes.byref(tp))
    for k, v in over.items():
        setattr(tp, k, v)
    return tp


def lg_token_state_size(cache, params, tparams) -> int:
    return int(lib().lg_token_state_size(ctypes.byref(cache.c), ctypes.byref(params),
                                         ctypes.byref(tparams)))


def lg_token_detect(cache, tokens, pmax, state, params, tparams, flags, spans, diag, tstate,
                    kept_idx=None, kept_count=None, stream=None):
    """kept_idx / kept_count: the buffers lg_prune_compact wrote after the previous call (or
    None): the trailing kept rows that are still consecutive tokens keep mapping the span"""
    max_keep = int(kept_idx.shape[1]) if kept_idx is not None else 0
    _call("lg_token_detect", ctypes.byref(cache.c), _ptr(tokens), _ptr(pmax), _ptr(kept_idx),
          _ptr(kept_count), max_keep, _ptr(state), ctypes.byref(params), ctypes.byref(tparams),
          _ptr(flags), _ptr(spans), _ptr(diag), _ptr(tstate), _stream(stream))


def lg_token_detect_prune(cache, tokens, pmax, state, budget, params, tparams, flags, spans,
                          diag, tstate, kept_idx, kept_count, max_keep, max_len, stream=None):
    """lg_token_detect then lg_prune_compact in two launches; kept_idx / kept_count carry the
    previous prune's lists in and this step's out"""
    _call("lg_token_detect_prune", ctypes.byref(cache.c), _ptr(tokens), _ptr(pmax), _ptr(state),
          _ptr(budget), ctypes.byref(params), ctypes.byref(tparams), _ptr(flags), _ptr(spans),
          _ptr(diag), _ptr(tstate), _ptr(kept_idx), _ptr(kept_count), max_keep, max_len,
          _stream(stream))


def lg_detect(cache, stats, H_q, state, budget, params, flags, spans, diag, dstate, stream=None):
    _call("lg_detect", ctypes.byref(cache.c), _ptr(stats), H_q, _ptr(state), _ptr(budget),
          ctypes.byref(params), _ptr(flags), _ptr(spans), _ptr(diag), _ptr(dstate),
          _stream(stream))


def lg_detect_prune(cache, stats, H_q, state, budget, params, flags, spans, diag, dstate,
                    kept_idx, kept_count, max_keep, max_len, stream=None):
    _call("lg_detect_prune", ctypes.byref(cache.c), _ptr(stats), H_q, _ptr(state), _ptr(budget),
          ctypes.byref(params), _ptr(flags), _ptr(spans), _ptr(diag), _ptr(dstate),
          _ptr(kept_idx), _ptr(kept_count), max_keep, max_len, _stream(stream))


def lg_prune_compact(cache, flags, spans, state, budget, params, kept_idx, kept_count, max_keep,
                     max_len, stream=None):
    _call("lg_prune_compact", ctypes.byref(cache.c), _ptr(flags), _ptr(spans), _ptr(state),
          _ptr(budget), ctypes.byref(params), _ptr(kept_idx), _ptr(kept_count), max_keep,
          max_len, _stream(stream))


def lg_h2o_reset(cache, max_len, stream=None):
    _call("lg_h2o_reset", ctypes.byref(cache.c), max_len, _stream(stream))


def lg_h2o_evict(cache, budget, pos_now, max_len, stream=None):
    _call("lg_h2o_evict", ctypes.byref(cache.c), _ptr(budget), _ptr(pos_now), max_len,
          _stream(stream))


def lg_streaming_evict(cache, budget, pos_now, n_sink, max_len, stream=None):
    _call("lg_streaming_evict", ctypes.byref(cache.c), _ptr(budget), _ptr(pos_now), n_sink,
          max_len, _stream(stream))


N_SINK = 4  # StreamingLLM attention sinks (count not stated by the paper)


def lg_read_device_status(cache, stream=None) -> int:
    code = ctypes.c_int32(0)
    _call("lg_read_device_status", ctypes.byref(cache.c), ctypes.byref(code), _stream(stream))
    return code.value


# ------------------------------------------------------------------ device buffers of a batch

def _torch_dtype(dtype: str):
    return torch.bfloat16 if dtype == "bf16" else torch.float32


def host_to_device(a: np.ndarray, device, dtype: str):
    """numpy cache-dtype array (bf16 as uint16 bits, or float32) -> torch tensor on device"""
    if dtype == "bf16":
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(
            torch.bfloat16).to(device)
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(device)


def device_to_host(t: torch.Tensor) -> np.ndarray:
    t = t.detach().cpu()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view(np.uint16)
    return t.numpy()


class Cache:
    """Device KV cache of a batch laid out as lg_cache documents, plus its metadata.
    policy 'loopguard' allocates sketches; 'h2o' allocates scores and positions."""

    def __init__(self, L, H_kv, d, dtype, seq_off, cap, n0, device, policy="loopguard",
                 k=None, v=None):
        self.L, self.H_kv, self.d, self.dtype = L, H_kv, d, dtype
        self.device = torch.device(device)
        self.batch = len(cap)
        self.S_total = int(np.asarray(cap, dtype=np.int64).sum())
        tdt = _torch_dtype(dtype)
        shape = (L, H_kv, self.S_total, d)
        self.k = k if k is not None else torch.zeros(shape, dtype=tdt, device=self.device)
        self.v = v if v is not None else torch.zeros(shape, dtype=tdt, device=self.device)
        self.seq_off = torch.as_tensor(np.asarray(seq_off, dtype=np.int64), device=self.device)
        self.cap = torch.as_tensor(np.asarray(cap, dtype=np.int32), device=self.device)
        self.len = torch.as_tensor(np.asarray(n0, dtype=np.int32), device=self.device).clone()
        self.nwords = H_kv * d // 32
        self.sketch = None
        self.h2o = self.pos = None
        if policy == "loopguard":
            self.sketch = torch.zeros((self.S_total, self.nwords), dtype=torch.int32,
                                      device=self.device)
        if policy in ("h2o", "streaming", "full"):
            self.h2o = torch.zeros((L, H_kv, self.S_total), dtype=torch.float32,
                                   device=self.device)
            self.pos = torch.zeros((L, H_kv, self.S_total), dtype=torch.int32,
                                   device=self.device)
        self.status = torch.zeros(1, dtype=torch.int32, device=self.device)
        self.c = LgCache(k=_ptr(self.k), v=_ptr(self.v), dtype=LG_BF16 if dtype == "bf16" else
                         LG_F32, L=L, H_kv=H_kv, d=d, batch=self.batch, pad=0,
                         S_total=self.S_total, seq_off=_ptr(self.seq_off), cap=_ptr(self.cap),
                         len=_ptr(self.len), sketch=_ptr(self.sketch), h2o=_ptr(self.h2o),
                         pos=_ptr(self.pos), dev_status=_ptr(self.status))

    @classmethod
    def from_host(cls, w, K, V, device, policy="loopguard", params=None):
        """cache of workload w from host arrays K, V [L][H_kv][S_total][d] (rows [0, n0))"""
        k = host_to_device(K, device, w.dtype)
        v = host_to_device(V, device, w.dtype)
        c = cls(w.L, w.H_kv, w.d, w.dtype, w.seq_off, w.cap, w.n0, device, policy, k, v)
        c.prepare(int(w.n0.max()), params)
        return c

    def prepare(self, max_len, params=None):
        """after a prefill: sketches of the guard layer, or H2O positions and scores"""
        if self.sketch is not None:
            lg_sketch_build(self, params or lg_default_params(), max_len)
        if self.h2o is not None:
            lg_h2o_reset(self, max_len)

    def to_host(self):
        return device_to_host(self.k), device_to_host(self.v)

    def lengths(self) -> np.ndarray:
        return self.len.cpu().numpy()


class Guard:
    """Device buffers and call order of one guarded decode step (lg.h) for a Cache."""

    def __init__(self, cache: Cache, H_q: int, params: LgGuardParams | None = None,
                 policy="loopguard", max_len=None, t_gen0=64, n_layers_per_call=None,
                 fused_prune=True):
        self.cache = cache
        self.fused_prune = fused_prune  # lg_detect_prune, else lg_detect + lg_prune_compact
        self.H_q = H_q
        self.p = params or lg_default_params()
        self.policy = policy
        dev = cache.device
        cap = cache.cap.cpu().numpy()
        self.max_len = int(cap.max()) if max_len is None else int(max_len)
        self.max_keep = self.max_len
        self.n_layers_per_call = n_layers_per_call or cache.L
        L, b = cache.L, cache.batch
        self.state = torch.zeros((b, STATE_BYTES // 4), dtype=torch.int32, device=dev)
        # flags and spans side by side (one read-back of a step's decisions)
        self.flags_spans = torch.zeros(3 * b, dtype=torch.int32, device=dev)
        self.flags = self.flags_spans[:b]
        self.spans = self.flags_spans[b:].view(b, 2)
        self.kept_idx = torch.zeros((b, self.max_keep), dtype=torch.int32, device=dev)
        self.kept_count = torch.zeros(b, dtype=torch.int32, device=dev)
        self.diag = torch.zeros((b, 8), dtype=torch.float64, device=dev)
        ds_words = lg_detect_state_size(cache, self.p) // 4 if policy == "loopguard" else 1
        self.dstate = torch.zeros(ds_words, dtype=torch.int32, device=dev)
        tdt = _torch_dtype(cache.dtype)
        self.out = torch.zeros((L, b, H_q, cache.d), dtype=tdt, device=dev)
        self.stats = torch.zeros((L, b, H_q, 4), dtype=torch.float32, device=dev)
        h2o = 1 if policy == "h2o" else 0
        ws_bytes = lg_workspace_size(cache, H_q, self.n_layers_per_call, self.max_len, h2o)
        self.ws = torch.empty(ws_bytes // 4 + 64, dtype=torch.float32, device=dev)
        self.scale = 1.0 / float(np.sqrt(cache.d))
        lg_state_init(cache, self.state, t_gen0)

    def step(self, q, k_new, v_new, budget, pos_new=None, stream=None):
        """one guarded decode step on device tensors:
        q [L][b][H_q][d], k_new/v_new [L][b][H_kv][d], budget [b] int32, pos_new [b] int32"""
        c, p = self.cache, self.p
        lg_begin_step(c, stream)
        lg_append(c, 0, c.L, k_new, v_new, pos_new, p, stream)
        for l0 in range(0, c.L, self.n_layers_per_call):
            nl = min(self.n_layers_per_call, c.L - l0)   # the last call takes what is left
            lg_decode_attend(c, l0, nl, q[l0:l0 + nl], self.H_q, self.scale, self.out[l0:l0 + nl],
                             self.stats[l0:l0 + nl], p.suffix_w, 1 if self.policy == "h2o" else 0,
                             self.max_len, self.ws, stream)
        if self.policy == "loopguard" and self.fused_prune:
            lg_detect_prune(c, self.stats, self.H_q, self.state, budget, p, self.flags,
                            self.spans, self.diag, self.dstate, self.kept_idx, self.kept_count,
                            self.max_keep, self.max_len, stream)
        elif self.policy == "loopguard":
            lg_detect(c, self.stats, self.H_q, self.state, budget, p, self.flags, self.spans,
                      self.diag, self.dstate, stream)
            lg_prune_compact(c, self.flags, self.spans, self.state, budget, p, self.kept_idx,
                             self.kept_count, self.max_keep, self.max_len, stream)
        elif self.policy == "h2o":
            lg_h2o_evict(c, budget, pos_new, self.max_len, stream)
        elif self.policy == "streaming":
            lg_streaming_evict(c, budget, pos_new, N_SINK, self.max_len, stream)

    def step_host(self, q, k_new, v_new, budget, pos_new=None):
        """same step from host numpy arrays; returns host copies of every output"""
        dev, dt = self.cache.device, self.cache.dtype
        qd = host_to_device(q, dev, dt)
        kd = host_to_device(k_new, dev, dt)
        vd = host_to_device(v_new, dev, dt)
        bd = torch.as_tensor(np.asarray(budget, dtype=np.int32), device=dev)
        pd = None if pos_new is None else torch.as_tensor(np.asarray(pos_new, dtype=np.int32),
                                                          device=dev)
        self.step(qd, kd, vd, bd, pd)
        return self.results()

    def results(self):
        torch.cuda.current_stream().synchronize()
        st = lg_read_device_status(self.cache)
        if st != 0:
            raise LgError("device status", st)
        r = dict(out=device_to_host(self.out).astype(np.float32) if self.cache.dtype == "f32"
                 else (device_to_host(self.out).astype(np.uint32) << 16).view(np.float32),
                 stats=self.stats.cpu().numpy(), len=self.cache.lengths())
        if self.policy == "loopguard":
            r.update(flags=self.flags.cpu().numpy(), spans=self.spans.cpu().numpy(),
                     kept_count=self.kept_count.cpu().numpy(),
                     kept_idx=self.kept_idx.cpu().numpy(),
                     state=self.state.cpu().numpy(), diag=self.diag.cpu().numpy())
        return r
