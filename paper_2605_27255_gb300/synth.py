"""Seeded synthetic inputs: model shapes, weights and prompts.

This module is the one piece shared by the CUDA path and the CPU oracle.  It
holds no arithmetic of the PIPO method itself: it only names the tensors of a
PIPO model (compressor, backbone blocks, MTP head, confidence head; paper
Sec. 3.2 and App. A) with their shapes, and fills them with seeded numbers.

Generator.  Every value is a pure function of (seed, tensor name, element
index), computed with 32-bit integer hashing in int64 torch ops, so the same
call gives bit-identical tensors on the CPU and on a GPU:

* ``_mix32`` is the integer finaliser ``x ^= x>>16; x *= 0x45d9f3b`` (twice)
  ``; x ^= x>>16`` on 32-bit words (products stay below 2**59, no overflow).
* A weight element takes two hashed words, splits them into four 16-bit
  uniforms and sums them (Irwin-Hall, n=4): an integer in [-131070, 131070],
  exact in fp32.  One fp32 multiply scales it to the requested standard
  deviation (mean 0, std exactly ``std`` in distribution).  This stands in for
  the N(0, 0.02) initialisation of the benchmark configurations; it is bounded
  at +-3.46 std.
* Norm gains are ``1 + g`` with ``g`` drawn like a weight at std
  ``gain_std`` (0.1 by default, so within [0.65, 1.35]; a gain drawn around
  0 would zero the signal).  Each norm has its own name and so its own
  values: every layer's attention and FFN norms, the final norm, the MTP
  input norms of h_b and of E[x_b], the MTP block's norms, the MTP post-norm
  and both halves of the confidence head's joint norm all differ, so a gain
  applied to the wrong norm changes the results.  ``gain_std = 0`` gives the
  unit gains of an untrained RMSNorm.
* Token ids are a hashed word modulo V, per sequence from ``seed + b``.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Dict, Tuple

import torch

M32 = 0xFFFFFFFF
_C = 0x45D9F3B
# std of the sum of four independent uniforms on {0..65535}
_IH4_STD = math.sqrt((65536.0 * 65536.0 - 1.0) / 3.0)
_IH4_MEAN = 4 * 65535 // 2  # 131070

PAD = -1  # id of the padding slot in a pair (never a vocabulary row)


@dataclasses.dataclass(frozen=True)
class ModelShape:
    """Dimensions and switches of one PIPO model instance."""
    name: str
    H: int            # hidden size
    L: int            # backbone layers
    n_q: int          # query heads
    n_kv: int         # key/value heads
    d_h: int          # head dim
    F: int            # SwiGLU inner size
    V: int            # vocabulary
    compressor: str = "mlp"   # "linear": W[a;b]+b  |  "mlp": W2 SiLU(W1[a;b])
    mtp_block: int = 1        # 1: W_fc then one decoder block; 0: W_fc only
    dtype: str = "bf16"       # storage type of weights, embeddings and KV
    rope_theta: float = 1.0e6
    eps: float = 1.0e-6
    tau: float = 0.5
    std: float = 0.02
    comp_residual: int = 0    # 1: the MLP compressor adds a + b (the residual form)

    @property
    def qkv_rows(self) -> int:
        return (self.n_q + 2 * self.n_kv) * self.d_h

    def with_(self, **kw) -> "ModelShape":
        return dataclasses.replace(self, **kw)


TINY = ModelShape("tiny", H=256, L=2, n_q=4, n_kv=2, d_h=64, F=1024, V=4096,
                  compressor="linear", mtp_block=1, dtype="f32",
                  rope_theta=1.0e4, tau=0.5)
B4 = ModelShape("4b", H=2560, L=36, n_q=32, n_kv=8, d_h=128, F=9728, V=151936,
                compressor="mlp", mtp_block=1, dtype="bf16", rope_theta=1.0e6,
                tau=0.5)
B9 = ModelShape("9b", H=4096, L=36, n_q=32, n_kv=8, d_h=128, F=12288, V=151936,
                compressor="mlp", mtp_block=1, dtype="bf16", rope_theta=1.0e6,
                tau=0.5)
PRESETS = {s.name: s for s in (TINY, B4, B9)}


def _block_shapes(s: ModelShape, n: int, prefix: str) -> Dict[str, Tuple[int, ...]]:
    H, qd, kd = s.H, s.n_q * s.d_h, s.n_kv * s.d_h
    return {
        f"{prefix}.attn_norm": (n, H),
        f"{prefix}.Wq": (n, qd, H),
        f"{prefix}.Wk": (n, kd, H),
        f"{prefix}.Wv": (n, kd, H),
        f"{prefix}.Wo": (n, H, qd),
        f"{prefix}.ffn_norm": (n, H),
        f"{prefix}.Wgate": (n, s.F, H),
        f"{prefix}.Wup": (n, s.F, H),
        f"{prefix}.Wdown": (n, H, s.F),
    }


def tensor_shapes(s: ModelShape) -> Dict[str, Tuple[int, ...]]:
    """Name -> shape of every tensor of the model (row-major, out x in)."""
    H = s.H
    d: Dict[str, Tuple[int, ...]] = {"E": (s.V, H), "x_pad": (H,)}
    if s.compressor == "linear":
        d["comp.W"] = (H, 2 * H)
        d["comp.b"] = (H,)
    elif s.compressor == "mlp":
        d["comp.W1"] = (H, 2 * H)
        d["comp.W2"] = (H, H)
    else:
        raise ValueError(s.compressor)
    d.update(_block_shapes(s, s.L, "blk"))
    d["final_norm"] = (H,)
    d["mtp.norm_h"] = (H,)
    d["mtp.norm_e"] = (H,)
    d["mtp.W_fc"] = (H, 2 * H)
    if s.mtp_block:
        d.update(_block_shapes(s, 1, "mtp"))
    d["mtp.norm_post"] = (H,)
    d["conf.norm"] = (2 * H,)
    d["conf.W1"] = (H, 2 * H)
    d["conf.W2"] = (1, H)
    return d


def is_gain(name: str) -> bool:
    return name.endswith("norm") or name.endswith("norm_h") or \
        name.endswith("norm_e") or name.endswith("norm_post")


def _name_id(name: str) -> int:
    """FNV-1a of the tensor name, 32 bits."""
    h = 0x811C9DC5
    for ch in name.encode():
        h = ((h ^ ch) * 0x01000193) & M32
    return h


def _mix32_int(x: int) -> int:
    """Python-int twin of ``_mix32`` (used for keys and in the tests)."""
    x &= M32
    x = (((x >> 16) ^ x) * _C) & M32
    x = (((x >> 16) ^ x) * _C) & M32
    return (x >> 16) ^ x


def _mix32(x: torch.Tensor) -> torch.Tensor:
    """``_mix32_int`` over an int64 tensor of values in [0, 2**32)."""
    x = ((x >> 16) ^ x) * _C & M32
    x = ((x >> 16) ^ x) * _C & M32
    return (x >> 16) ^ x


def _keys(seed: int, name: str) -> Tuple[int, int]:
    k1 = _mix32_int(_mix32_int(seed * 0x9E3779B1 + 0x7F4A7C15) ^ _name_id(name))
    k2 = _mix32_int(k1 ^ 0x5BD1E995)
    return k1, k2


def hashed_words(seed: int, name: str, idx: torch.Tensor) -> Tuple[torch.Tensor, torch.Tensor]:
    """Two 32-bit words per element index (int64 tensor, 0 <= idx < 2**31)."""
    k1, k2 = _keys(seed, name)
    c = 2 * idx
    h1 = _mix32((_mix32(c ^ k1) + k2) & M32)
    h2 = _mix32((_mix32((c + 1) ^ k1) + k2) & M32)
    return h1, h2


def hashed_words_int(seed: int, name: str, i: int) -> Tuple[int, int]:
    k1, k2 = _keys(seed, name)
    h1 = _mix32_int((_mix32_int((2 * i) ^ k1) + k2) & M32)
    h2 = _mix32_int((_mix32_int((2 * i + 1) ^ k1) + k2) & M32)
    return h1, h2


def _ih4(h1: torch.Tensor, h2: torch.Tensor) -> torch.Tensor:
    s = (h1 & 0xFFFF) + (h1 >> 16) + (h2 & 0xFFFF) + (h2 >> 16) - _IH4_MEAN
    return s.to(torch.float32)


def gen_tensor(seed: int, name: str, shape, std: float, dtype: torch.dtype,
               device="cpu", chunk: int = 1 << 26) -> torch.Tensor:
    """Seeded zero-mean tensor of the given std (see module docstring)."""
    n = 1
    for d in shape:
        n *= d
    assert n < (1 << 31)
    out = torch.empty(n, dtype=dtype, device=device)
    scale = torch.tensor(std / _IH4_STD, dtype=torch.float32, device=device)
    for s0 in range(0, n, chunk):
        s1 = min(n, s0 + chunk)
        idx = torch.arange(s0, s1, dtype=torch.int64, device=device)
        h1, h2 = hashed_words(seed, name, idx)
        out[s0:s1] = (_ih4(h1, h2) * scale).to(dtype)
        del idx, h1, h2
    return out.view(*shape)


def torch_dtype(s: ModelShape) -> torch.dtype:
    return {"f32": torch.float32, "bf16": torch.bfloat16}[s.dtype]


GAIN_STD = 0.1


def gen_weights(s: ModelShape, seed: int = 0, device="cpu",
                gain_std: float = GAIN_STD) -> Dict[str, torch.Tensor]:
    """All tensors of ``s``: gains ``1 + N(0, gain_std)`` per norm (rounded
    to the storage type), everything else seeded with std ``s.std``."""
    dt = torch_dtype(s)
    w = {}
    for name, shape in tensor_shapes(s).items():
        if is_gain(name):
            if gain_std == 0.0:
                w[name] = torch.ones(shape, dtype=dt, device=device)
            else:
                g = gen_tensor(seed, name, shape, gain_std, torch.float32, device)
                w[name] = (1.0 + g).to(dt)
        else:
            w[name] = gen_tensor(seed, name, shape, s.std, dt, device)
    return w


def gen_prompts(batch: int, length: int, V: int, seed: int = 1, device="cpu") -> torch.Tensor:
    """Uniform token ids in [0, V): row b is seeded by ``seed + b``."""
    rows = []
    idx = torch.arange(length, dtype=torch.int64, device=device)
    for b in range(batch):
        h1, _ = hashed_words(seed + b, "prompt", idx)
        rows.append((h1 % V).to(torch.int32))
    if not rows:
        return torch.empty(0, length, dtype=torch.int32, device=device)
    return torch.stack(rows)


def gen_kv_fill(s: ModelShape, n_entries: int, seed: int = 7, device="cpu") -> Tuple[torch.Tensor, torch.Tensor]:
    """Seeded K and V contents for ``L+1`` caches, [L+1, n, n_kv*d_h] fp32.

    Used only where a timing run needs a filled cache at a given context
    length and the values do not matter (std 1, the scale of rotated keys)."""
    shape = (s.L + 1, n_entries, s.n_kv * s.d_h)
    k = gen_tensor(seed, "kv.K", shape, 1.0, torch.float32, device)
    v = gen_tensor(seed, "kv.V", shape, 1.0, torch.float32, device)
    if s.dtype == "bf16":
        k, v = k.to(torch.bfloat16).float(), v.to(torch.bfloat16).float()
    return k, v
