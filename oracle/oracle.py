"""ctypes wrapper of the fp64 C oracle (``pipo_oracle.c``).

TEST INFRASTRUCTURE ONLY: imported by the tests, by the package smoke check
and by the CPU-baseline leg of the benchmark, never by the product path.
It builds ``liboracle.so`` next to this file with gcc (OpenMP) on first use.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading
from typing import Dict, Optional

import numpy as np
import torch

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "pipo_oracle.c")
LIB = os.path.join(HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

OK, EINVAL, ECAPACITY = 0, 1, 3


def build(force: bool = False) -> str:
    """Compile the oracle with gcc; returns the library path."""
    if force or not os.path.exists(LIB) or os.path.getmtime(LIB) < os.path.getmtime(SRC):
        tmp = LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-fopenmp", "-fPIC", "-shared", "-Wall",
                               "-o", tmp, SRC, "-lm"])
        os.replace(tmp, LIB)
    return LIB


class OrcConfig(C.Structure):
    _fields_ = [(n, C.c_int) for n in ("H", "L", "n_q", "n_kv", "d_h", "F", "V",
                                        "compressor", "mtp_block", "wdtype", "kv_bf16")] + \
               [("rope_theta", C.c_double), ("eps", C.c_double), ("max_ctx", C.c_int), ("comp_residual", C.c_int)]


_WNAMES = [
    ("E", "E"), ("x_pad", "x_pad"),
    ("comp_W", "comp.W"), ("comp_b", "comp.b"), ("comp_W1", "comp.W1"), ("comp_W2", "comp.W2"),
    ("attn_norm", "blk.attn_norm"), ("Wq", "blk.Wq"), ("Wk", "blk.Wk"), ("Wv", "blk.Wv"),
    ("Wo", "blk.Wo"), ("ffn_norm", "blk.ffn_norm"), ("Wgate", "blk.Wgate"), ("Wup", "blk.Wup"),
    ("Wdown", "blk.Wdown"), ("final_norm", "final_norm"),
    ("mtp_norm_h", "mtp.norm_h"), ("mtp_norm_e", "mtp.norm_e"), ("mtp_W_fc", "mtp.W_fc"),
    ("m_attn_norm", "mtp.attn_norm"), ("m_Wq", "mtp.Wq"), ("m_Wk", "mtp.Wk"), ("m_Wv", "mtp.Wv"),
    ("m_Wo", "mtp.Wo"), ("m_ffn_norm", "mtp.ffn_norm"), ("m_Wgate", "mtp.Wgate"),
    ("m_Wup", "mtp.Wup"), ("m_Wdown", "mtp.Wdown"), ("mtp_norm_post", "mtp.norm_post"),
    ("conf_norm", "conf.norm"), ("conf_W1", "conf.W1"), ("conf_W2", "conf.W2"),
]


class OrcWeights(C.Structure):
    _fields_ = [(f, C.c_void_p) for f, _ in _WNAMES]


_D = C.POINTER(C.c_double)
_I = C.POINTER(C.c_int32)


class OrcOut(C.Structure):
    _fields_ = [("tokens", _I), ("n_acc", _I), ("logits_b", _D), ("logits_d", _D),
                ("conf", _D), ("h_b", _D), ("h_d", _D), ("margin_b", _D), ("margin_d", _D),
                ("x_b", _I), ("x_d", _I)]


def lib():
    global _lib
    with _lock:
        if _lib is None:
            L = C.CDLL(build())
            L.orc_new.restype = C.c_void_p
            L.orc_new.argtypes = [C.POINTER(OrcConfig), C.POINTER(OrcWeights), C.c_int]
            L.orc_free.argtypes = [C.c_void_p]
            L.orc_step.argtypes = [C.c_void_p, C.c_double, C.c_int, C.POINTER(OrcOut)]
            L.orc_prefill.argtypes = [C.c_void_p, _I, _I, C.c_int, C.c_double, C.c_int, C.POINTER(OrcOut)]
            L.orc_regular_step.argtypes = [C.c_void_p, C.POINTER(OrcOut)]
            L.orc_regular_prefill.argtypes = [C.c_void_p, _I, _I, C.c_int, C.POINTER(OrcOut)]
            L.orc_set_pending.argtypes = [C.c_void_p, _I]
            L.orc_rollback.argtypes = [C.c_void_p, _I]
            L.orc_get_seq.argtypes = [C.c_void_p, C.c_int, _I, _I, _I, C.POINTER(C.c_int64)]
            L.orc_get_cache.argtypes = [C.c_void_p, C.c_int, C.c_int, C.c_int, _D, _D]
            L.orc_set_cache.argtypes = [C.c_void_p, C.c_int, C.c_int, C.POINTER(C.c_float), C.POINTER(C.c_float)]
            L.orc_bruteforce.argtypes = [C.POINTER(OrcConfig), C.POINTER(OrcWeights), C.c_int, _I, _I,
                                         C.c_double, C.c_int, C.POINTER(OrcOut)]
            L.orc_rmsnorm.argtypes = [_D, C.c_int, C.c_void_p, C.c_size_t, C.c_int, C.c_double, _D]
            L.orc_matvec.argtypes = [C.c_void_p, C.c_size_t, C.c_int, C.c_int, C.c_int, _D, _D]
            L.orc_rope.argtypes = [_D, C.c_int, C.c_int, C.c_int, C.c_double]
            L.orc_attend.argtypes = [_D, _D, _D, C.c_int, C.c_int, C.c_int, C.c_int, _D]
            L.orc_sample.argtypes = [_D, C.c_int, _I, C.c_int, C.c_double, C.c_int, C.c_double, C.c_double,
                                     C.c_double]
            L.orc_sample.restype = C.c_int
            L.orc_sample_ex.argtypes = [_D, C.c_int, _I, C.c_int, C.c_double, C.c_int, C.c_double, C.c_double,
                                        C.c_double, _D]
            L.orc_sample_ex.restype = C.c_int
            L.orc_set_sampler.argtypes = [C.c_void_p, C.c_double, C.c_int, C.c_double, C.c_double]
            L.orc_step_u.argtypes = [C.c_void_p, C.c_double, C.c_int, _D, C.POINTER(OrcOut)]
            L.orc_prefill_u.argtypes = [C.c_void_p, _I, _I, C.c_int, C.c_double, C.c_int, _D, C.POINTER(OrcOut)]
            L.orc_get_hist.argtypes = [C.c_void_p, C.c_int, _I, C.c_int]
            L.orc_get_hist.restype = C.c_int
            L.orc_argmax.argtypes = [_D, C.c_int, _D]
            L.orc_argmax.restype = C.c_int
            for f in ("orc_silu", "orc_sigmoid", "orc_round_bf16"):
                getattr(L, f).argtypes = [C.c_double]
                getattr(L, f).restype = C.c_double
            L.orc_confidence.argtypes = [C.POINTER(OrcConfig), C.POINTER(OrcWeights), _D, _D]
            L.orc_confidence.restype = C.c_double
            L.orc_compress.argtypes = [C.POINTER(OrcConfig), C.POINTER(OrcWeights), C.c_int, C.c_int, _D]
            _lib = L
    return _lib


def _dp(a: np.ndarray):
    assert a.dtype == np.float64 and a.flags.c_contiguous
    return a.ctypes.data_as(_D)


def _ip(a: np.ndarray):
    assert a.dtype == np.int32 and a.flags.c_contiguous
    return a.ctypes.data_as(_I)


def _host_array(t) -> np.ndarray:
    """torch tensor / ndarray -> contiguous numpy buffer in storage type."""
    if isinstance(t, torch.Tensor):
        t = t.detach().cpu().contiguous()
        if t.dtype == torch.bfloat16:
            return t.view(torch.int16).numpy().view(np.uint16)
        return t.numpy()
    return np.ascontiguousarray(t)


class Model:
    """Config + weights handed to the C oracle (keeps the buffers alive)."""

    def __init__(self, shape, weights: Dict[str, torch.Tensor], max_ctx: int = 256,
                 kv_bf16: Optional[bool] = None):
        self.shape = shape
        wd = 1 if shape.dtype == "bf16" else 0
        kvb = wd if kv_bf16 is None else int(kv_bf16)
        self.cfg = OrcConfig(shape.H, shape.L, shape.n_q, shape.n_kv, shape.d_h, shape.F, shape.V,
                             0 if shape.compressor == "linear" else 1, shape.mtp_block, wd, kvb,
                             shape.rope_theta, shape.eps, max_ctx, int(shape.comp_residual))
        self._keep = {}
        self.w = OrcWeights()
        for f, name in _WNAMES:
            if name in weights:
                a = _host_array(weights[name])
                self._keep[name] = a
                setattr(self.w, f, a.ctypes.data)


def _out(B: int, V: int, H: int, full: bool = True):
    o = dict(tokens=np.zeros((B, 2), np.int32), n_acc=np.zeros(B, np.int32),
             conf=np.zeros(B), margin_b=np.zeros(B), margin_d=np.zeros(B),
             x_b=np.zeros(B, np.int32), x_d=np.zeros(B, np.int32),
             h_b=np.zeros((B, H)), h_d=np.zeros((B, H)))
    if full:
        o["logits_b"] = np.zeros((B, V))
        o["logits_d"] = np.zeros((B, V))
    s = OrcOut()
    for k, v in o.items():
        setattr(s, k, _ip(v) if v.dtype == np.int32 else _dp(v))
    return o, s


class State:
    """A batch of B sequences with KV caches, as the oracle decodes them."""

    def __init__(self, model: Model, batch: int):
        self.m = model
        self.B = batch
        self.ptr = lib().orc_new(C.byref(model.cfg), C.byref(model.w), batch)
        if not self.ptr:
            raise MemoryError("oracle state allocation failed")

    def __del__(self):
        if getattr(self, "ptr", None):
            lib().orc_free(self.ptr)
            self.ptr = None

    def _draws(self, u):
        if u is None:
            return None, None
        a = np.ascontiguousarray(np.asarray(u, dtype=np.float64).reshape(self.B, 2))
        return a, _dp(a)

    def prefill(self, ids, lens=None, tau=0.5, force=0, logits=True, u=None):
        """u: draws [B, 2] of the two heads at the last position (sampler on)."""
        ids = np.ascontiguousarray(np.asarray(ids, dtype=np.int32))
        if lens is None:
            lens = np.full(self.B, ids.shape[1], np.int32)
        lens = np.ascontiguousarray(np.asarray(lens, dtype=np.int32))
        o, s = _out(self.B, self.m.shape.V, self.m.shape.H, logits)
        keep, up = self._draws(u)
        rc = lib().orc_prefill_u(self.ptr, _ip(ids), _ip(lens), ids.shape[1], tau, force, up, C.byref(s))
        if rc != OK:
            raise ValueError(f"oracle prefill failed: {rc}")
        return o

    def step(self, tau=0.5, force=0, logits=True, u=None):
        """u: draws [B, 2] of the two heads (sampler on)."""
        o, s = _out(self.B, self.m.shape.V, self.m.shape.H, logits)
        keep, up = self._draws(u)
        rc = lib().orc_step_u(self.ptr, tau, force, up, C.byref(s))
        if rc != OK:
            raise ValueError(f"oracle step failed: {rc}")
        return o

    def set_sampler(self, temperature=1.0, top_k=20, top_p=0.95, rep_penalty=1.5):
        """Sampling in both heads (temperature <= 0: greedy again)."""
        if lib().orc_set_sampler(self.ptr, temperature, top_k, top_p, rep_penalty) != OK:
            raise ValueError("oracle sampler: bad settings")

    def history(self, b):
        n = lib().orc_get_hist(self.ptr, b, None, 0)
        h = np.zeros(n, np.int32)
        lib().orc_get_hist(self.ptr, b, _ip(h), n)
        return h

    def regular_prefill(self, ids, lens=None, logits=True):
        """Regular decoding (one token per backbone pass, the paper's baseline):
        run the prompt, return the first output token (tokens[:, 0])."""
        ids = np.ascontiguousarray(np.asarray(ids, dtype=np.int32))
        if lens is None:
            lens = np.full(self.B, ids.shape[1], np.int32)
        lens = np.ascontiguousarray(np.asarray(lens, dtype=np.int32))
        o, s = _out(self.B, self.m.shape.V, self.m.shape.H, logits)
        rc = lib().orc_regular_prefill(self.ptr, _ip(ids), _ip(lens), ids.shape[1], C.byref(s))
        if rc != OK:
            raise ValueError(f"oracle regular prefill failed: {rc}")
        return o

    def regular_step(self, logits=True):
        """One regular decode step: the pending token through the backbone and
        the LM head; the argmax becomes the next pending token."""
        o, s = _out(self.B, self.m.shape.V, self.m.shape.H, logits)
        rc = lib().orc_regular_step(self.ptr, C.byref(s))
        if rc != OK:
            raise ValueError(f"oracle regular step failed: {rc}")
        return o

    def set_pending(self, pairs):
        p = np.ascontiguousarray(np.asarray(pairs, dtype=np.int32).reshape(self.B, 2))
        lib().orc_set_pending(self.ptr, _ip(p))

    def rollback(self, n):
        n = np.ascontiguousarray(np.asarray(n, dtype=np.int32).reshape(self.B))
        rc = lib().orc_rollback(self.ptr, _ip(n))
        if rc != OK:
            raise ValueError("oracle rollback: bad length")

    def seq(self, b):
        p0, p1, n = C.c_int32(), C.c_int32(), C.c_int32()
        e = C.c_int64()
        lib().orc_get_seq(self.ptr, b, C.byref(p0), C.byref(p1), C.byref(n), C.byref(e))
        return dict(p0=p0.value, p1=p1.value, n=n.value, emitted=e.value)

    def cache(self, b, layer, n):
        kd = self.m.shape.n_kv * self.m.shape.d_h
        K = np.zeros((n, kd))
        V = np.zeros((n, kd))
        lib().orc_get_cache(self.ptr, b, layer, n, _dp(K), _dp(V))
        return K, V

    def set_cache(self, b, K, V):
        K = np.ascontiguousarray(np.asarray(K, dtype=np.float32))
        V = np.ascontiguousarray(np.asarray(V, dtype=np.float32))
        n = K.shape[1]
        rc = lib().orc_set_cache(self.ptr, b, n, K.ctypes.data_as(C.POINTER(C.c_float)),
                                 V.ctypes.data_as(C.POINTER(C.c_float)))
        if rc != OK:
            raise ValueError("oracle set_cache: capacity")


def bruteforce(model: Model, pairs, mtp_tok, tau=0.5, force=0):
    pairs = np.ascontiguousarray(np.asarray(pairs, dtype=np.int32).reshape(-1, 2))
    n1 = pairs.shape[0]
    mt = np.zeros(n1, np.int32)
    mt[: len(mtp_tok)] = np.asarray(mtp_tok, dtype=np.int32)[:n1]
    o, s = _out(1, model.shape.V, model.shape.H, True)
    lib().orc_bruteforce(C.byref(model.cfg), C.byref(model.w), n1, _ip(pairs), _ip(mt), tau, force, C.byref(s))
    return o


# ---- primitives (for the pins) -----------------------------------------

def rmsnorm(x, gamma, eps=1e-6):
    x = np.ascontiguousarray(x, dtype=np.float64)
    g = np.ascontiguousarray(gamma, dtype=np.float32)
    y = np.zeros_like(x)
    lib().orc_rmsnorm(_dp(x), x.size, g.ctypes.data, 0, 0, eps, _dp(y))
    return y


def matvec(W, x):
    W = np.ascontiguousarray(W, dtype=np.float32)
    x = np.ascontiguousarray(x, dtype=np.float64)
    N, K = W.shape
    y = np.zeros(N)
    lib().orc_matvec(W.ctypes.data, 0, 0, N, K, _dp(x), _dp(y))
    return y


def rope(v, n_heads, d, pos, theta):
    v = np.array(v, dtype=np.float64).reshape(-1).copy()
    lib().orc_rope(_dp(v), n_heads, d, pos, theta)
    return v


def attend(q, K, V, n_q, n_kv, d):
    q = np.ascontiguousarray(q, dtype=np.float64).reshape(-1)
    K = np.ascontiguousarray(K, dtype=np.float64)
    V = np.ascontiguousarray(V, dtype=np.float64)
    out = np.zeros(n_q * d)
    lib().orc_attend(_dp(q), _dp(K), _dp(V), K.shape[0], n_q, n_kv, d, _dp(out))
    return out


def sample_ex(logits, u, hist=(), temperature=1.0, top_k=20, top_p=0.95, rep_penalty=1.5):
    """orc_sample_ex: (token, decision margin)."""
    x = np.ascontiguousarray(logits, dtype=np.float64)
    h = np.ascontiguousarray(np.asarray(hist, dtype=np.int32).reshape(-1))
    nh = h.size
    if nh == 0:
        h = np.zeros(1, np.int32)
    m = C.c_double()
    t = lib().orc_sample_ex(_dp(x), x.size, _ip(h), nh, float(temperature), int(top_k), float(top_p),
                            float(rep_penalty), float(u), C.byref(m))
    return t, m.value


def argmax(x):
    x = np.ascontiguousarray(x, dtype=np.float64)
    m = C.c_double()
    i = lib().orc_argmax(_dp(x), x.size, C.byref(m))
    return i, m.value


def sample(logits, u, hist=(), temperature=1.0, top_k=20, top_p=0.95, rep_penalty=1.5):
    """The evaluation sampler (see orc_sample); u in [0, 1) is the draw."""
    x = np.ascontiguousarray(logits, dtype=np.float64)
    h = np.ascontiguousarray(np.asarray(hist, dtype=np.int32).reshape(-1))
    if h.size == 0:
        h = np.zeros(1, np.int32)
        nh = 0
    else:
        nh = h.size
    return lib().orc_sample(_dp(x), x.size, _ip(h), nh, float(temperature), int(top_k), float(top_p),
                            float(rep_penalty), float(u))


def silu(x):
    return lib().orc_silu(float(x))


def sigmoid(x):
    return lib().orc_sigmoid(float(x))


def round_bf16(x):
    return lib().orc_round_bf16(float(x))


def compress(model: Model, t0, t1):
    z = np.zeros(model.shape.H)
    lib().orc_compress(C.byref(model.cfg), C.byref(model.w), t0, t1, _dp(z))
    return z


def confidence(model: Model, hb, hd):
    hb = np.ascontiguousarray(hb, dtype=np.float64)
    hd = np.ascontiguousarray(hd, dtype=np.float64)
    return lib().orc_confidence(C.byref(model.cfg), C.byref(model.w), _dp(hb), _dp(hd))
