"""Time one decode-path kernel in isolation through the C ABI (pipo_op_gemv,
or with --tc the tensor-core projection pipo_op_gemm_tc: its activation-split
kernel and its GEMM, both in the timed region).

  python -m paper_2605_27255_gb300.kernel_bench --shape lm_head [--batch 1] [--iters 50] [--tc] [--splits S]

With --step, one eagerly launched decode step (pipo_profile_step, inside an
NVTX range "profile_step") of a small bf16 model -- 512 wide, 3 layers, 8/2
heads of 128, the attention shape of the 4B model -- with every cache filled
to --ctx seeded entries: a small case for profiler captures of the attention
and projection kernels.

  python -m paper_2605_27255_gb300.kernel_bench --step --batch 64 --ctx 512

With --prefill T, one pair prefill of T tokens per sequence on the same small
model, position by position or in chunks (--rows R, --tile for the causal
tile attention), inside an NVTX range "prefill".

  python -m paper_2605_27255_gb300.kernel_bench --prefill 8192 --rows 128 --tile

With --chain C, the fixed cost of a GEMV launch: a CUDA graph of C launches
of one shape (with programmatic dependent launch unless --no-pdl) against
one launch over the same rows.

  python -m paper_2605_27255_gb300.kernel_bench --chain 32 --shape o_proj

Shapes are the weight-streaming projections of the 4B-class model (and, with
the _9b suffix, of the 9B-class model).  Weights
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
    # the 9B-class model
    "qkv_9b": (6144, 4096, 0),
    "o_proj_9b": (4096, 4096, 0),
    "gate_up_9b": (12288, 4096, 1),
    "down_9b": (4096, 12288, 0),
}


def run(name: str, batch: int, iters: int, min_bytes: float = 300e6, tc: bool = False, splits: int = 0,
        fused: bool = False) -> dict:
    N, K, mode = SHAPES[name]
    rows = 2 * N if mode else N
    nbytes = rows * K * 2
    copies = max(1, int(-(-min_bytes // nbytes)))
    Ws = [(torch.randn(rows, K, device="cuda") * 0.02).to(torch.bfloat16) for _ in range(copies)]
    x = torch.randn(batch, K, device="cuda")
    y = torch.empty(batch, N, device="cuda")
    st = torch.cuda.current_stream()
    if tc or fused:
        sb = capi.pipo_op_gemm_tc_scratch(mode, N, K, batch, splits)
        scratch = torch.empty(sb + 1024, dtype=torch.uint8, device="cuda")
        base = (scratch.data_ptr() + 1023) // 1024 * 1024
        gamma = torch.ones(K, dtype=torch.bfloat16, device="cuda")

        def launch(i):
            if fused:  # normalised input: the converter warps inside the GEMM (batch 16 or 32)
                capi.pipo_op_gemm_tc_norm(mode, Ws[i % copies].data_ptr(), N, x.data_ptr(), K, gamma.data_ptr(),
                                          0, 0, 0, 0, 1e-6, batch, y.data_ptr(), splits, base, sb, st.cuda_stream)
            else:
                capi.pipo_op_gemm_tc(mode, Ws[i % copies].data_ptr(), N, K, x.data_ptr(), batch, y.data_ptr(),
                                     splits, base, sb, st.cuda_stream)
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
    return dict(kernel="gemm_tcf" if fused else "gemm_tc" if tc else "gemv", shape=name, batch=batch, N=N, K=K, us_per_launch=us,
                gbs=nbytes / us / 1e3, bytes_per_launch=nbytes, copies=copies)


STEP_SHAPE = dict(name="step", H=512, L=3, n_q=8, n_kv=2, d_h=128, F=1408, V=5056, compressor="mlp",
                  mtp_block=1, dtype="bf16", rope_theta=1.0e6, tau=0.5)


def run_step(batch: int, ctx: int) -> dict:
    from . import synth
    shape = synth.ModelShape(**STEP_SHAPE)
    w = synth.gen_weights(shape, seed=0, device="cuda")
    g = capi.Pipo(shape, w, max_batch=batch, max_ctx=ctx + 16)
    try:
        g.prefill(synth.gen_prompts(batch, 2, shape.V, seed=1).numpy())
        K, V = synth.gen_kv_fill(shape, ctx, seed=7, device="cuda")
        K, V = K.cpu().numpy(), V.cpu().numpy()
        for b in range(batch):
            g.load_cache(b, K, V)
        for _ in range(3):
            g.step_async()
        torch.cuda.synchronize()
        torch.cuda.nvtx.range_push("profile_step")
        kind, by, ms = g.profile_step()
        torch.cuda.nvtx.range_pop()
        torch.cuda.synchronize()
        out = dict(kernel="decode_step", shape=STEP_SHAPE["name"], batch=batch, ctx=ctx, path=g.describe(),
                   launches=len(kind))
        for k, name in ((0, "projections"), (1, "attention"), (2, "other")):
            sel = [i for i, kk in enumerate(kind) if int(kk) == k]
            t = float(sum(ms[i] for i in sel))
            b = float(sum(by[i] for i in sel))
            out[name] = dict(launches=len(sel), ms=t, gbs=(b / (t / 1e3) / 1e9) if t > 0 and b > 0 else None)
        return out
    finally:
        g.close()


def run_chain(name: str, count: int, batch: int, pdl: bool) -> dict:
    """The fixed cost of a GEMV launch: a CUDA graph of `count` launches of one
    projection shape (distinct weight copies, so every launch streams from
    HBM) against a graph of one launch over the same total rows."""
    N, K, mode = SHAPES[name]
    rows = 2 * N if mode else N
    Ws = [(torch.randn(rows, K, device="cuda") * 0.02).to(torch.bfloat16) for _ in range(count)]
    big = torch.cat(Ws, 0)  # one GEMV of count x N rows
    x = torch.randn(batch, K, device="cuda")
    y = torch.empty(batch, N * count, device="cuda")
    st = torch.cuda.Stream()
    ptrs = [w.data_ptr() for w in Ws]

    def timed(fn) -> float:
        with torch.cuda.stream(st):
            fn()  # load, set attributes
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=st):
            fn()
        for _ in range(3):
            g.replay()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(10):
            g.replay()
        e1.record()
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) * 1e3 / 10

    chain_us = timed(lambda: capi.pipo_op_gemv_chain(1, mode, ptrs, N, K, x.data_ptr(), batch, y.data_ptr(), pdl,
                                                     torch.cuda.current_stream().cuda_stream))
    one_us = timed(lambda: capi.pipo_op_gemv(1, mode, big.data_ptr(), N * count, K, x.data_ptr(), batch,
                                             y.data_ptr(), torch.cuda.current_stream().cuda_stream))
    nbytes = rows * K * 2 * count
    return dict(kernel="gemv_chain", shape=name, count=count, batch=batch, pdl=pdl, chain_us=chain_us,
                single_us=one_us, per_launch_overhead_us=(chain_us - one_us) / count,
                chain_gbs=nbytes / chain_us / 1e3, single_gbs=nbytes / one_us / 1e3)


def run_prefill(batch: int, tokens: int, rows: int, tile: bool) -> dict:
    """One pair prefill of `tokens` tokens per sequence on the small bf16 model
    (the shape of --step), with chunks of `rows` rows (0: position by position)
    and the tile or per-row chunk attention; wall time of the synchronous call
    after one warm-up prefill."""
    import os
    import time

    from . import synth
    os.environ["PIPO_PREFILL_ROWS"] = str(rows)
    os.environ["PIPO_PREFILL_ATTN"] = "tile" if tile else "rows"
    shape = synth.ModelShape(**STEP_SHAPE)
    w = synth.gen_weights(shape, seed=0, device="cuda")
    g = capi.Pipo(shape, w, max_batch=batch, max_ctx=(tokens + 1) // 2 + 4)
    try:
        prompts = synth.gen_prompts(batch, tokens, shape.V, seed=1).numpy()
        g.prefill(prompts)
        torch.cuda.synchronize()
        torch.cuda.nvtx.range_push("prefill")
        t0 = time.perf_counter()
        g.prefill(prompts)
        dt = time.perf_counter() - t0
        torch.cuda.nvtx.range_pop()
        return dict(kernel="prefill", shape=STEP_SHAPE["name"], batch=batch, tokens=tokens, rows=rows, tile=tile,
                    seconds=dt, pairs_per_s=batch * ((tokens + 1) // 2) / dt)
    finally:
        g.close()


def main() -> None:
    ap = argparse.ArgumentParser()
    ap.add_argument("--shape", default="all", choices=["all"] + sorted(SHAPES))
    ap.add_argument("--batch", type=int, default=1)
    ap.add_argument("--iters", type=int, default=50)
    ap.add_argument("--tc", action="store_true", help="tensor-core projection (bf16 hi/lo activations)")
    ap.add_argument("--splits", type=int, default=0, help="K splits of the tensor-core GEMM (0: automatic)")
    ap.add_argument("--fused", action="store_true",
                    help="the tensor-core projection with the activation split inside the GEMM (the decode step's "
                         "form at batch widths 16 and 32; --batch 16 or 32)")
    ap.add_argument("--step", action="store_true", help="one eager decode step of a small bf16 model")
    ap.add_argument("--ctx", type=int, default=512, help="--step: cached entries per sequence")
    ap.add_argument("--prefill", type=int, default=0, help="time a pair prefill of this many tokens per sequence")
    ap.add_argument("--chain", type=int, default=0,
                    help="graph of this many launches of --shape against one launch of the summed rows")
    ap.add_argument("--no-pdl", action="store_true", help="--chain: without programmatic dependent launch")
    ap.add_argument("--rows", type=int, default=0, help="--prefill: chunk rows (0: position by position)")
    ap.add_argument("--tile", action="store_true", help="--prefill: the causal tile chunk attention")
    a = ap.parse_args()
    capi.load()
    if a.prefill:
        print(json.dumps(run_prefill(a.batch, a.prefill, a.rows, a.tile)), flush=True)
        return
    if a.chain:
        shape = "o_proj" if a.shape == "all" else a.shape
        print(json.dumps(run_chain(shape, a.chain, a.batch, not a.no_pdl)), flush=True)
        return
    if a.step:
        print(json.dumps(run_step(a.batch, a.ctx)), flush=True)
        return
    for name in (sorted(SHAPES) if a.shape == "all" else [a.shape]):
        print(json.dumps(run(name, a.batch, a.iters, tc=a.tc, splits=a.splits, fused=a.fused)), flush=True)


if __name__ == "__main__":
    main()
