"""Algorithmic bytes and flops of one PIPO pair-decode step.

What the method must move per step, whatever the implementation:
  * every weight of the compressor, the L backbone blocks, the MTP input
    projection and block, and the confidence head, once;
  * the tied embedding E twice: the draft head needs the backbone token x_b
    from the first LM-head pass before its own pass can start (Eq. 3-5);
  * the KV cache of every block: entries 0..n of each sequence, read once
    (keys and values, backbone blocks + the MTP block), plus the new entry
    written.
Activations are a few KB per sequence and are left out.
"""
from __future__ import annotations

from .synth import ModelShape


def esize(s: ModelShape) -> int:
    return 2 if s.dtype == "bf16" else 4


def block_params(s: ModelShape) -> int:
    qd, kd = s.n_q * s.d_h, s.n_kv * s.d_h
    return 2 * s.H + (qd + 2 * kd) * s.H + s.H * qd + 3 * s.F * s.H


def weight_params(s: ModelShape) -> int:
    """Parameters streamed once per step (E excluded)."""
    H = s.H
    comp = H * 2 * H + (H * H if s.compressor == "mlp" else H)
    mtp = 2 * H + H * 2 * H + (block_params(s) if s.mtp_block else 0) + H
    conf = 2 * H + H * 2 * H + H
    return comp + s.L * block_params(s) + H + mtp + conf


def kv_entry_bytes(s: ModelShape) -> int:
    """Bytes of one KV entry across every cached block (K and V)."""
    layers = s.L + (1 if s.mtp_block else 0)
    return layers * 2 * s.n_kv * s.d_h * esize(s)


def step_bytes(s: ModelShape, batch: int, ctx_avg: float) -> float:
    """Algorithmic HBM bytes of one step; ctx_avg = mean entries per sequence
    before the step (the step reads ctx_avg + 1 entries and writes one)."""
    e = esize(s)
    w = (weight_params(s) + 2 * s.V * s.H) * e
    kv = batch * (ctx_avg + 1) * kv_entry_bytes(s) + batch * kv_entry_bytes(s)
    return float(w + kv)


def step_flops(s: ModelShape, batch: int, ctx_avg: float) -> float:
    """Multiply-add flops of one step (2 per MAC): weights x batch + attention."""
    macs = (weight_params(s) + 2 * s.V * s.H) * batch
    layers = s.L + (1 if s.mtp_block else 0)
    macs += batch * layers * (ctx_avg + 1) * s.n_q * s.d_h * 2
    return 2.0 * macs


def prefill_flops(s: ModelShape, batch: int, n_pairs: int) -> float:
    """Multiply-add flops (2 per MAC) of a pair prefill of n_pairs positions
    per sequence: at every position the compressor, the L backbone blocks,
    the teacher-forced MTP input projection and the MTP block; causal
    attention of each position over itself and the positions before it
    (q.k and p.v, every cached block); the heads once, at the last position
    (two LM-head passes and the confidence head).  Norms and activations are
    left out."""
    H, qd, kd = s.H, s.n_q * s.d_h, s.n_kv * s.d_h
    block = (qd + 2 * kd) * H + H * qd + 3 * s.F * H
    comp = H * 2 * H + (H * H if s.compressor == "mlp" else 0)
    mtp = H * 2 * H + (block if s.mtp_block else 0)
    per_pos = comp + s.L * block + mtp
    layers = s.L + (1 if s.mtp_block else 0)
    attn = layers * s.n_q * s.d_h * 2 * (n_pairs * (n_pairs + 1) / 2.0)
    heads = 2 * s.V * H + H * 2 * H + H
    return 2.0 * batch * (n_pairs * per_pos + attn + heads)


def regular_step_bytes(s: ModelShape, batch: int, ctx_avg: float) -> float:
    """Algorithmic HBM bytes of one step of regular decoding (the baseline of
    Sec. 4): the L backbone blocks and the final norm once, E once (one LM-head
    pass), the backbone caches' entries 0..n read and the new one written.  The
    input embedding is a gather of one row per sequence (left out, like the
    activations)."""
    e = esize(s)
    w = (s.L * block_params(s) + s.H + s.V * s.H) * e
    entry = s.L * 2 * s.n_kv * s.d_h * e
    return float(w + batch * (ctx_avg + 1) * entry + batch * entry)


# ------------------------------------------------------------ recorded DRAM traffic

def sources_digest(csrc_dir: str) -> str:
    """SHA-256 (hex, first 16 digits) over the kernel sources (every .cu, .cuh
    and .h file of csrc, by name order): a traffic figure recorded with ncu
    describes these kernels only while the digest is unchanged."""
    import hashlib
    import os
    h = hashlib.sha256()
    for name in sorted(os.listdir(csrc_dir)):
        if name.endswith((".cu", ".cuh", ".h")):
            h.update(name.encode())
            with open(os.path.join(csrc_dir, name), "rb") as f:
                h.update(f.read())
    return h.hexdigest()[:16]


def recorded_traffic(profiles_dir: str, workload: str, csrc_dir: str = None):
    """DRAM bytes per projection launch that an ncu capture recorded for this
    workload, from a line of a profiles/*.md summary of the form

        traffic: workload=<name> bytes_per_launch=<float> sources=<digest>

    Returns {"bytes_per_launch", "source"} when the recorded digest equals the
    current kernel sources' digest, else None (no capture, or the kernels
    changed since it was taken)."""
    import os
    import re
    if csrc_dir is None:
        csrc_dir = os.path.join(os.path.dirname(os.path.abspath(__file__)), "csrc")
    if not os.path.isdir(profiles_dir):
        return None
    digest = sources_digest(csrc_dir)
    pat = re.compile(r"^traffic:\s+workload=(\S+)\s+bytes_per_launch=([0-9.eE+-]+)\s+sources=([0-9a-f]+)\s*$")
    for name in sorted(os.listdir(profiles_dir)):
        if not name.endswith(".md"):
            continue
        with open(os.path.join(profiles_dir, name)) as f:
            for line in f:
                m = pat.match(line.strip())
                if m and m.group(1) == workload and m.group(3) == digest:
                    return {"bytes_per_launch": float(m.group(2)), "source": f"profiles/{name} (ncu dram__bytes)"}
    return None
