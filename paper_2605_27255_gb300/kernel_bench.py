"""Time one decode-path kernel in isolation through the C ABI (pipo_op_gemv,
or with --tc the tensor-core projection pipo_op_gemm_tc: its activation-split
kernel and its GEMM, both in the timed region).

  python -m paper_2605_27255_gb300.kernel_bench --shape lm_head [--batch 1] [--iters 50] [--tc] [--splits S]

Shapes are the weight-streaming projections of the 4B-class model.  Weights
are random bf16; several copies are cycled so that every launch streams from
HBM (more than twice the 129 MB L2 in total).  Prints one JSON line per shape
with the CUDA-event time per launch and the achieved GB/s of algorithmic bytes.
"""
from __future__ import annotations

import argparse
import json

import torch

from . import capi

# name -> (output rows N, input length K, mode: 0 plain, 1 SwiGLU pairs)
SHAPES = {
    "qkv": (6144, 2560, 0),
    "o_proj": (2560, 4096, 0),
    "gate_up": (9728, 2560, 1),
    "down": (2560, 9728, 0),
    "w_fc": (2560, 5120, 0),
    "lm_head": (151936, 2560, 0),
}


def run(name: str, batch: int, iters: int, min_bytes: float = 300e6, tc: bool = False, splits: int = 0) -> dict:
    N, K, mode = SHAPES[name]
    rows = 2 * N if mode else N
    nbytes = rows * K * 2
    copies = max(1, int(-(-min_bytes // nbytes)))
    Ws = [(torch.randn(rows, K, device="cuda") * 0.02).to(torch.bfloat16) for _ in range(copies)]
    x = torch.randn(batch, K, device="cuda")
    y = torch.empty(batch, N, device="cuda")
    st = torch.cuda.current_stream()
    if tc:
        sb = capi.pipo_op_gemm_tc_scratch(mode, N, K, batch, splits)
        scratch = torch.empty(sb + 1024, dtype=torch.uint8, device="cuda")
        base = (scratch.data_ptr() + 1023) // 1024 * 1024

        def launch(i):
            capi.pipo_op_gemm_tc(mode, Ws[i % copies].data_ptr(), N, K, x.data_ptr(), batch, y.data_ptr(), splits,
                                 base, sb, st.cuda_stream)
    else:
        def launch(i):
            capi.pipo_op_gemv(1, mode, Ws[i % copies].data_ptr(), N, K, x.data_ptr(), batch, y.data_ptr(),
                              st.cuda_stream)
    for i in range(3):
        launch(i)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    e0.record(st)
    for i in range(iters):
        launch(i)
    e1.record(st)
    torch.cuda.synchronize()
    us = e0.elapsed_time(e1) * 1e3 / iters
    return dict(kernel="gemm_tc" if tc else "gemv", shape=name, batch=batch, N=N, K=K, us_per_launch=us,
                gbs=nbytes / us / 1e3, bytes_per_launch=nbytes, copies=copies)


def main() -> None:
    ap = argparse.ArgumentParser()
    ap.add_argument("--shape", default="all", choices=["all"] + sorted(SHAPES))
    ap.add_argument("--batch", type=int, default=1)
    ap.add_argument("--iters", type=int, default=50)
    ap.add_argument("--tc", action="store_true", help="tensor-core projection (bf16 hi/lo activations)")
    ap.add_argument("--splits", type=int, default=0, help="K splits of the tensor-core GEMM (0: automatic)")
    a = ap.parse_args()
    capi.load()
    for name in (sorted(SHAPES) if a.shape == "all" else [a.shape]):
        print(json.dumps(run(name, a.batch, a.iters, tc=a.tc, splits=a.splits)), flush=True)


if __name__ == "__main__":
    main()
