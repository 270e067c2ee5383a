"""Thin ctypes binding of the C ABI in ``include/pipo.h``.

Argument marshalling only: every step of the decode path runs in the CUDA
library (``lib/libpipo.so``).  There is no Python or CPU fallback; loading
fails loudly when the library has not been built.  Function names mirror the
C entry points (``pipo_init``, ``pipo_prefill``, ``pipo_decode_step`` ...);
``Pipo`` wraps one context for convenience.
"""
from __future__ import annotations

import ctypes as C
import os
import threading
from typing import Dict, Optional

import numpy as np
import torch

from .synth import ModelShape

LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "lib", "libpipo.so")

PIPO_OK, PIPO_EINVAL, PIPO_ENOMEM, PIPO_ECAPACITY, PIPO_ECUDA, PIPO_ESTATE = range(6)
_NAMES = {0: "OK", 1: "EINVAL", 2: "ENOMEM", 3: "ECAPACITY", 4: "ECUDA", 5: "ESTATE"}


class PipoError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"PIPO_{_NAMES.get(status, status)}: {msg}")
        self.status = status


class pipo_config(C.Structure):
    _fields_ = [(n, C.c_int32) for n in ("hidden", "n_layers", "n_q_heads", "n_kv_heads", "head_dim", "ffn",
                                         "vocab", "compressor", "mtp_block", "dtype")] + \
               [("rope_theta", C.c_float), ("rms_eps", C.c_float)] + \
               [(n, C.c_int32) for n in ("max_batch", "max_ctx", "page_size")] + \
               [("tau", C.c_float), ("force_mode", C.c_int32), ("debug", C.c_int32),
                ("page_shuffle_seed", C.c_uint32), ("comp_residual", C.c_int32)]


# C field -> tensor name of synth.tensor_shapes
WEIGHT_FIELDS = [
    ("E", "E"), ("x_pad", "x_pad"), ("comp_W", "comp.W"), ("comp_b", "comp.b"),
    ("comp_W1", "comp.W1"), ("comp_W2", "comp.W2"),
    ("attn_norm", "blk.attn_norm"), ("Wq", "blk.Wq"), ("Wk", "blk.Wk"), ("Wv", "blk.Wv"),
    ("Wo", "blk.Wo"), ("ffn_norm", "blk.ffn_norm"), ("Wgate", "blk.Wgate"), ("Wup", "blk.Wup"),
    ("Wdown", "blk.Wdown"), ("final_norm", "final_norm"),
    ("mtp_norm_h", "mtp.norm_h"), ("mtp_norm_e", "mtp.norm_e"), ("mtp_W_fc", "mtp.W_fc"),
    ("m_attn_norm", "mtp.attn_norm"), ("m_Wq", "mtp.Wq"), ("m_Wk", "mtp.Wk"), ("m_Wv", "mtp.Wv"),
    ("m_Wo", "mtp.Wo"), ("m_ffn_norm", "mtp.ffn_norm"), ("m_Wgate", "mtp.Wgate"), ("m_Wup", "mtp.Wup"),
    ("m_Wdown", "mtp.Wdown"), ("mtp_norm_post", "mtp.norm_post"),
    ("conf_norm", "conf.norm"), ("conf_W1", "conf.W1"), ("conf_W2", "conf.W2"),
]


class pipo_weights(C.Structure):
    _fields_ = [("location", C.c_int32)] + [(f, C.c_void_p) for f, _ in WEIGHT_FIELDS]


_FP = C.POINTER(C.c_float)
_IP = C.POINTER(C.c_int32)


class pipo_debug(C.Structure):
    _fields_ = [("logits_b", _FP), ("logits_d", _FP), ("conf", _FP), ("h_b", _FP), ("h_d", _FP),
                ("x_b", _IP), ("x_d", _IP)]


# name -> (restype, argtypes): every entry point declared in include/pipo.h
SIGNATURES = {
    "pipo_init": (C.c_int, [C.POINTER(pipo_config), C.POINTER(pipo_weights), C.POINTER(C.c_void_p)]),
    "pipo_prefill": (C.c_int, [C.c_void_p, C.c_int32, _IP, C.c_int32, _IP, _IP, _IP]),
    "pipo_prefill_slot": (C.c_int, [C.c_void_p, C.c_int32, _IP, C.c_int32, _IP, _IP]),
    "pipo_decode_step": (C.c_int, [C.c_void_p, _IP, _IP]),
    "pipo_decode_step_async": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p]),
    "pipo_decode_steps": (C.c_int, [C.c_void_p, C.c_int32, _IP, _IP]),
    "pipo_regular_prefill": (C.c_int, [C.c_void_p, C.c_int32, _IP, C.c_int32, _IP, _IP, _IP]),
    "pipo_regular_step": (C.c_int, [C.c_void_p, _IP]),
    "pipo_regular_step_async": (C.c_int, [C.c_void_p, C.c_void_p]),
    "pipo_rollback": (C.c_int, [C.c_void_p, _IP]),
    "pipo_set_threshold": (C.c_int, [C.c_void_p, C.c_float, C.c_int32]),
    "pipo_set_sampler": (C.c_int, [C.c_void_p, C.c_float, C.c_int32, C.c_float, C.c_float, _FP, C.c_int32]),
    "pipo_set_pending": (C.c_int, [C.c_void_p, _IP]),
    "pipo_get_counters": (C.c_int, [C.c_void_p, _IP, C.POINTER(C.c_int64)]),
    "pipo_debug_dump": (C.c_int, [C.c_void_p, C.POINTER(pipo_debug)]),
    "pipo_read_cache": (C.c_int, [C.c_void_p, C.c_int32, C.c_int32, C.c_int32, _FP, _FP]),
    "pipo_load_cache": (C.c_int, [C.c_void_p, C.c_int32, C.c_int32, _FP, _FP]),
    "pipo_set_stream": (C.c_int, [C.c_void_p, C.c_void_p]),
    "pipo_op_gemv": (C.c_int, [C.c_int32, C.c_int32, C.c_void_p, C.c_int32, C.c_int32, C.c_void_p, C.c_int32,
                               C.c_void_p, C.c_void_p]),
    "pipo_op_gemv_chain": (C.c_int, [C.c_int32, C.c_int32, C.POINTER(C.c_void_p), C.c_int32, C.c_int32, C.c_int32,
                                     C.c_void_p, C.c_int32, C.c_void_p, C.c_int32, C.c_void_p]),
    "pipo_op_lm_head_argmax": (C.c_int, [C.c_int32, C.c_void_p, C.c_int32, C.c_int32, C.c_void_p, C.c_void_p,
                                         C.c_float, C.c_int32, C.c_void_p, C.c_void_p, C.c_void_p, C.c_size_t,
                                         C.c_void_p]),
    "pipo_op_lm_head_argmax_noalloc": (C.c_int, [C.c_int32, C.c_void_p, C.c_int32, C.c_int32, C.c_void_p,
                                                 C.c_void_p, C.c_float, C.c_int32, C.c_void_p, C.c_void_p,
                                                 C.c_void_p]),
    "pipo_op_gemm_tc": (C.c_int, [C.c_int32, C.c_void_p, C.c_int32, C.c_int32, C.c_void_p, C.c_int32, C.c_void_p,
                                  C.c_int32, C.c_void_p, C.c_size_t, C.c_void_p]),
    "pipo_op_gemm_tc_scratch": (C.c_size_t, [C.c_int32, C.c_int32, C.c_int32, C.c_int32, C.c_int32]),
    "pipo_op_gemm_tc_norm": (C.c_int, [C.c_int32, C.c_void_p, C.c_int32, C.c_void_p, C.c_int32, C.c_void_p,
                                       C.c_void_p, C.c_int32, C.c_void_p, C.c_int32, C.c_float, C.c_int32,
                                       C.c_void_p, C.c_int32, C.c_void_p, C.c_size_t, C.c_void_p]),
    "pipo_describe_step": (C.c_int, [C.c_void_p, C.c_char_p, C.c_size_t]),
    "pipo_replay_family": (C.c_int, [C.c_void_p, C.c_int32, C.c_int32, C.POINTER(C.c_double), _IP]),
    "pipo_selftest_wait": (C.c_int, [C.c_int32, C.c_uint64, C.POINTER(C.c_uint32)]),
    "pipo_profile_step": (C.c_int, [C.c_void_p, C.c_int32, _IP, C.POINTER(C.c_double), _FP, _IP]),
    "pipo_step_launches": (C.c_int32, [C.c_void_p]),
    "pipo_last_error": (C.c_char_p, [C.c_void_p]),
    "pipo_free": (None, [C.c_void_p]),
}

_lib = None
_lock = threading.Lock()


def load(path: str = LIB_PATH):
    """Load the CUDA library (raises if it is missing: no fallback)."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(path):
                raise RuntimeError(f"PIPO CUDA library not built: {path} (run __graft_entry__.build())")
            L = C.CDLL(path)
            for name, (res, args) in SIGNATURES.items():
                fn = getattr(L, name)
                fn.restype = res
                fn.argtypes = args
            _lib = L
    return _lib


def _check(rc: int, ctx) -> None:
    if rc != PIPO_OK:
        msg = load().pipo_last_error(ctx).decode()
        raise PipoError(rc, msg)


def _i32(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.int32))


def _ip(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data_as(_IP)


def _fp(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data_as(_FP)


# ---- entry points (same names as the C ABI) -----------------------------

def pipo_init(cfg: pipo_config, w: pipo_weights):
    ctx = C.c_void_p()
    _check(load().pipo_init(C.byref(cfg), C.byref(w), C.byref(ctx)), None)
    return ctx


def pipo_prefill(ctx, ids: np.ndarray, lens: Optional[np.ndarray] = None):
    ids = _i32(ids)
    B, stride = ids.shape
    lens = _i32(np.full(B, stride) if lens is None else lens)
    tok = np.zeros((B, 2), np.int32)
    nacc = np.zeros(B, np.int32)
    _check(load().pipo_prefill(ctx, B, _ip(ids), stride, _ip(lens), _ip(tok), _ip(nacc)), ctx)
    return tok, nacc


def pipo_prefill_slot(ctx, slot: int, ids: np.ndarray):
    ids = _i32(np.asarray(ids).reshape(-1))
    tok = np.zeros((1, 2), np.int32)
    nacc = np.zeros(1, np.int32)
    _check(load().pipo_prefill_slot(ctx, int(slot), _ip(ids), ids.size, _ip(tok), _ip(nacc)), ctx)
    return tok, nacc


def pipo_decode_step(ctx, B: int):
    tok = np.zeros((B, 2), np.int32)
    nacc = np.zeros(B, np.int32)
    _check(load().pipo_decode_step(ctx, _ip(tok), _ip(nacc)), ctx)
    return tok, nacc


def pipo_decode_steps(ctx, B: int, n: int):
    tok = np.zeros((n, B, 2), np.int32)
    nacc = np.zeros((n, B), np.int32)
    _check(load().pipo_decode_steps(ctx, int(n), _ip(tok), _ip(nacc)), ctx)
    return tok, nacc


def pipo_decode_step_async(ctx, d_tokens: int = 0, d_nacc: int = 0):
    _check(load().pipo_decode_step_async(ctx, C.c_void_p(d_tokens or None), C.c_void_p(d_nacc or None)), ctx)


def pipo_regular_prefill(ctx, ids: np.ndarray, lens: Optional[np.ndarray] = None):
    ids = _i32(ids)
    B, stride = ids.shape
    lens = _i32(np.full(B, stride) if lens is None else lens)
    tok = np.zeros((B, 2), np.int32)
    nacc = np.zeros(B, np.int32)
    _check(load().pipo_regular_prefill(ctx, B, _ip(ids), stride, _ip(lens), _ip(tok), _ip(nacc)), ctx)
    return tok, nacc


def pipo_regular_step(ctx, B: int):
    tok = np.zeros((B, 2), np.int32)
    _check(load().pipo_regular_step(ctx, _ip(tok)), ctx)
    return tok


def pipo_regular_step_async(ctx, d_tokens: int = 0):
    _check(load().pipo_regular_step_async(ctx, C.c_void_p(d_tokens or None)), ctx)


def pipo_rollback(ctx, n_pairs) -> None:
    _check(load().pipo_rollback(ctx, _ip(_i32(n_pairs))), ctx)


def pipo_set_threshold(ctx, tau: float, force_mode: int = 0) -> None:
    _check(load().pipo_set_threshold(ctx, float(tau), int(force_mode)), ctx)


def pipo_set_sampler(ctx, temperature: float, top_k: int, top_p: float, rep_penalty: float, u) -> None:
    """u: [n_u, max_batch, 2] uniform draws in [0, 1)."""
    u = np.ascontiguousarray(np.asarray(u, dtype=np.float32))
    n_u = u.shape[0] if u.ndim == 3 else 0
    _check(load().pipo_set_sampler(ctx, float(temperature), int(top_k), float(top_p), float(rep_penalty),
                                   _fp(u) if u.size else None, n_u), ctx)


def pipo_set_pending(ctx, pairs) -> None:
    _check(load().pipo_set_pending(ctx, _ip(_i32(pairs))), ctx)


def pipo_get_counters(ctx, B: int):
    n = np.zeros(B, np.int32)
    e = np.zeros(B, np.int64)
    _check(load().pipo_get_counters(ctx, _ip(n), e.ctypes.data_as(C.POINTER(C.c_int64))), ctx)
    return n, e


def pipo_debug_dump(ctx, B: int, V: int, H: int) -> Dict[str, np.ndarray]:
    o = dict(logits_b=np.zeros((B, V), np.float32), logits_d=np.zeros((B, V), np.float32),
             conf=np.zeros(B, np.float32), h_b=np.zeros((B, H), np.float32), h_d=np.zeros((B, H), np.float32),
             x_b=np.zeros(B, np.int32), x_d=np.zeros(B, np.int32))
    d = pipo_debug(*[(_ip(v) if v.dtype == np.int32 else _fp(v)) for v in o.values()])
    _check(load().pipo_debug_dump(ctx, C.byref(d)), ctx)
    return o


def pipo_read_cache(ctx, b: int, layer: int, n: int, kd: int):
    K = np.zeros((n, kd), np.float32)
    V = np.zeros((n, kd), np.float32)
    _check(load().pipo_read_cache(ctx, b, layer, n, _fp(K), _fp(V)), ctx)
    return K, V


def pipo_load_cache(ctx, b: int, K: np.ndarray, V: np.ndarray) -> None:
    K = np.ascontiguousarray(K, dtype=np.float32)
    V = np.ascontiguousarray(V, dtype=np.float32)
    _check(load().pipo_load_cache(ctx, b, K.shape[1], _fp(K), _fp(V)), ctx)


def pipo_set_stream(ctx, stream: int) -> None:
    _check(load().pipo_set_stream(ctx, C.c_void_p(stream or None)), ctx)


def pipo_op_gemv(dtype: int, mode: int, W: int, N: int, K: int, x: int, B: int, y: int, stream: int = 0) -> None:
    """Device pointers (ints); see include/pipo.h."""
    _check(load().pipo_op_gemv(dtype, mode, C.c_void_p(W), N, K, C.c_void_p(x), B, C.c_void_p(y),
                               C.c_void_p(stream or None)), None)


def pipo_op_gemv_chain(dtype: int, mode: int, Ws, N: int, K: int, x: int, B: int, y: int, pdl: bool = True,
                       stream: int = 0) -> None:
    """len(Ws) GEMVs back to back (device pointers as ints); see include/pipo.h."""
    arr = (C.c_void_p * len(Ws))(*[C.c_void_p(w) for w in Ws])
    _check(load().pipo_op_gemv_chain(dtype, mode, arr, len(Ws), N, K, C.c_void_p(x), B, C.c_void_p(y), int(pdl),
                                     C.c_void_p(stream or None)), None)


def pipo_op_lm_head_argmax(dtype: int, E: int, V: int, H: int, h: int, gamma: int, eps: float, B: int,
                           tokens: int, logits: int, scratch: int, scratch_bytes: int, stream: int = 0) -> None:
    """Device pointers (ints; 0 = NULL); see include/pipo.h."""
    _check(load().pipo_op_lm_head_argmax(dtype, C.c_void_p(E), V, H, C.c_void_p(h), C.c_void_p(gamma or None),
                                         float(eps), B, C.c_void_p(tokens), C.c_void_p(logits or None),
                                         C.c_void_p(scratch or None), scratch_bytes, C.c_void_p(stream or None)),
           None)


def pipo_op_gemm_tc_scratch(mode: int, N: int, K: int, B: int, splits: int = 0) -> int:
    """Scratch bytes pipo_op_gemm_tc needs (0: rejected arguments)."""
    return int(load().pipo_op_gemm_tc_scratch(mode, N, K, B, splits))


def pipo_op_gemm_tc(mode: int, W: int, N: int, K: int, x: int, B: int, y: int, splits: int, scratch: int,
                    scratch_bytes: int, stream: int = 0) -> None:
    """Tensor-core projection on device pointers (ints); see include/pipo.h."""
    _check(load().pipo_op_gemm_tc(mode, C.c_void_p(W), N, K, C.c_void_p(x), B, C.c_void_p(y), splits,
                                  C.c_void_p(scratch), scratch_bytes, C.c_void_p(stream or None)), None)


def pipo_op_gemm_tc_norm(mode: int, W: int, N: int, x0: int, K0: int, gamma0: int, x1: int, K1: int, gamma1: int,
                         joint: int, eps: float, B: int, y: int, splits: int, scratch: int, scratch_bytes: int,
                         stream: int = 0) -> None:
    """Tensor-core projection of RMS-normalised segments on device pointers
    (ints, 0 for NULL); see include/pipo.h."""
    _check(load().pipo_op_gemm_tc_norm(mode, C.c_void_p(W or None), N, C.c_void_p(x0 or None), K0,
                                       C.c_void_p(gamma0 or None), C.c_void_p(x1 or None), K1,
                                       C.c_void_p(gamma1 or None), joint, eps, B, C.c_void_p(y or None), splits,
                                       C.c_void_p(scratch or None), scratch_bytes, C.c_void_p(stream or None)), None)


def pipo_selftest_wait(signal: int, limit_ns: int):
    """Bounded-wait self-test (see include/pipo.h): returns (status, message,
    wait record [site, block, iteration, parity]) without raising."""
    info = (C.c_uint32 * 4)()
    st = load().pipo_selftest_wait(signal, limit_ns, info)
    return st, pipo_last_error(None), list(info)


def pipo_op_lm_head_argmax_noalloc(dtype: int, E: int, V: int, H: int, h: int, gamma: int, eps: float, B: int,
                                   tokens: int, logits: int, stream: int = 0) -> None:
    """The LM-head argmax for callers that cannot allocate device memory: no
    scratch argument, at most 64 sequences, calls on one device must not
    overlap (see include/pipo.h).  Device pointers are ints (0 = NULL)."""
    _check(load().pipo_op_lm_head_argmax_noalloc(dtype, C.c_void_p(E), V, H, C.c_void_p(h),
                                                 C.c_void_p(gamma or None), float(eps), B, C.c_void_p(tokens),
                                                 C.c_void_p(logits or None), C.c_void_p(stream or None)), None)


def pipo_profile_step(ctx, cap: int = 4096):
    """Per-launch (kind, algorithmic bytes, ms) of one eagerly run decode step."""
    kind = np.zeros(cap, np.int32)
    by = np.zeros(cap, np.float64)
    ms = np.zeros(cap, np.float32)
    n = np.zeros(1, np.int32)
    _check(load().pipo_profile_step(ctx, cap, _ip(kind), by.ctypes.data_as(C.POINTER(C.c_double)), _fp(ms), _ip(n)),
           ctx)
    k = int(min(n[0], cap))
    return kind[:k], by[:k], ms[:k]


def pipo_step_launches(ctx) -> int:
    return int(load().pipo_step_launches(ctx))


def pipo_last_error(ctx=None) -> str:
    return load().pipo_last_error(ctx).decode()


def pipo_free(ctx) -> None:
    if ctx:
        load().pipo_free(ctx)


# ---- convenience --------------------------------------------------------

def make_config(s: ModelShape, max_batch: int, max_ctx: int, *, tau: Optional[float] = None,
                force_mode: int = 0, debug: bool = False, page_size: int = 64,
                page_shuffle_seed: int = 0) -> pipo_config:
    return pipo_config(s.H, s.L, s.n_q, s.n_kv, s.d_h, s.F, s.V, 0 if s.compressor == "linear" else 1,
                       s.mtp_block, 1 if s.dtype == "bf16" else 0, s.rope_theta, s.eps, max_batch, max_ctx,
                       page_size, s.tau if tau is None else tau, force_mode, int(debug), page_shuffle_seed,
                       int(s.comp_residual))


def make_weights(weights: Dict[str, torch.Tensor], keep: list) -> pipo_weights:
    """pipo_weights over a dict of torch tensors (all on the CPU or all on
    the GPU); ``keep`` receives the contiguous buffers that must outlive
    pipo_init."""
    w = pipo_weights()
    loc = None
    for field, name in WEIGHT_FIELDS:
        t = weights.get(name)
        if t is None:
            continue
        t = t.contiguous()
        keep.append(t)
        here = 1 if t.is_cuda else 0
        if loc is not None and here != loc:
            raise ValueError("weights must all be on the host or all on the device")
        loc = here
        setattr(w, field, t.data_ptr())
    w.location = loc or 0
    return w


class Pipo:
    """One library context: ``Pipo(shape, weights, max_batch, max_ctx)``."""

    def __init__(self, shape: ModelShape, weights: Dict[str, torch.Tensor], max_batch: int, max_ctx: int, **kw):
        self.shape = shape
        self.cfg = make_config(shape, max_batch, max_ctx, **kw)
        keep: list = []
        self.ctx = pipo_init(self.cfg, make_weights(weights, keep))
        self.B = 0

    def close(self):
        if getattr(self, "ctx", None):
            pipo_free(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def prefill(self, ids, lens=None):
        ids = _i32(ids)
        self.B = ids.shape[0]
        return pipo_prefill(self.ctx, ids, lens)

    def prefill_slot(self, slot, ids):
        """Prefill one slot while the others keep their state (continuous
        batching); the steps then cover slots 0 .. max(slot, B - 1)."""
        out = pipo_prefill_slot(self.ctx, slot, ids)
        self.B = max(self.B, int(slot) + 1)
        return out

    def step(self):
        return pipo_decode_step(self.ctx, self.B)

    def steps(self, n):
        """n decode steps in one call: (tokens [n, B, 2], n_accepted [n, B])."""
        return pipo_decode_steps(self.ctx, self.B, n)

    def step_async(self, d_tokens: int = 0, d_nacc: int = 0):
        pipo_decode_step_async(self.ctx, d_tokens, d_nacc)

    def regular_prefill(self, ids, lens=None):
        """Regular decoding (one token per backbone pass): run the prompt,
        return (tokens [B,2] = (first token, -1), n_accepted = 0)."""
        ids = _i32(ids)
        self.B = ids.shape[0]
        return pipo_regular_prefill(self.ctx, ids, lens)

    def regular_step(self):
        return pipo_regular_step(self.ctx, self.B)

    def regular_step_async(self, d_tokens: int = 0):
        pipo_regular_step_async(self.ctx, d_tokens)

    def set_threshold(self, tau, force_mode=0):
        pipo_set_threshold(self.ctx, tau, force_mode)

    def set_sampler(self, u, temperature=1.0, top_k=20, top_p=0.95, rep_penalty=1.5):
        """Sampling in both heads with the draws u [n_u, max_batch, 2]
        (temperature <= 0: greedy again)."""
        pipo_set_sampler(self.ctx, temperature, top_k, top_p, rep_penalty, u)

    def set_pending(self, pairs):
        pipo_set_pending(self.ctx, pairs)

    def rollback(self, n):
        pipo_rollback(self.ctx, n)

    def counters(self):
        return pipo_get_counters(self.ctx, self.B)

    def debug(self):
        return pipo_debug_dump(self.ctx, self.B, self.shape.V, self.shape.H)

    def read_cache(self, b, layer, n):
        return pipo_read_cache(self.ctx, b, layer, n, self.shape.n_kv * self.shape.d_h)

    def load_cache(self, b, K, V):
        pipo_load_cache(self.ctx, b, K, V)

    def set_stream(self, stream: int):
        pipo_set_stream(self.ctx, stream)

    def launches(self) -> int:
        return pipo_step_launches(self.ctx)

    def describe(self) -> str:
        """The kernels the next decode step launches (pipo_describe_step)."""
        buf = C.create_string_buffer(512)
        _check(load().pipo_describe_step(self.ctx, buf, 512), self.ctx)
        return buf.value.decode()

    def profile_step(self):
        return pipo_profile_step(self.ctx)

    def replay_family(self, family: int, n: int):
        """Enqueue n replays of one kernel family of the step (pipo_replay_family);
        returns (algorithmic bytes per replay, launches per replay)."""
        by, nl = C.c_double(), C.c_int32()
        _check(load().pipo_replay_family(self.ctx, family, n, C.byref(by), C.byref(nl)), self.ctx)
        return by.value, nl.value
