#!/usr/bin/env python
"""Throughput of the PIPO pair-decode step on one GB300 (one JSON line).

A step is one pass of the whole hot path for every sequence of the batch:
pair embed + compressor, L backbone blocks over the paged pair-KV cache, LM
head + argmax, MTP head + argmax, confidence head, acceptance and the device
bookkeeping.  Metric: accepted tokens/s over all sequences (1 + acceptance
per sequence and step), with the pair-step latency and the HBM roofline.

  python bench.py [--workload 9b-b8] [--steps K] [--warmup W] [--gpus N]
  python bench.py --impl reference ...   # the fp64 CPU oracle on host cores

The default workload is the largest single-GPU configuration: 9B-class
shapes at batch 8 with 4096-token prompts (20 GB moved per step).  Inputs are
synthetic and seeded (weights and prompts from synth.py); weights are
streamed from HBM every step (9-20 GB per step, far above the 129 MB L2), so
no L2 flush is needed between steps.

Roofline of the dominant kernel family (the weight-streaming projections):
after the timed steps, a CUDA graph holding only the step's projection
launches (same launch plan, step order and programmatic dependent launch) is
replayed and timed with CUDA events on the context stream
(pipo_replay_family); its algorithmic bytes per replay divided by its time
give the achieved bandwidth.  DRAM traffic per launch comes from the ncu
summary in profiles/ when its recorded source hash matches the kernels built
here, else it is null.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

# name -> model preset, batch, prompt tokens, pair-decode steps of the workload
WORKLOADS = {
    "tiny": dict(shape="tiny", batch=1, prompt=64, steps=32),
    "4b-b1": dict(shape="4b", batch=1, prompt=2048, steps=512),
    "4b-b4": dict(shape="4b", batch=4, prompt=1024, steps=256),
    "4b-b16": dict(shape="4b", batch=16, prompt=1024, steps=256),
    "4b-b64": dict(shape="4b", batch=64, prompt=1024, steps=256),
    "4b-lc": dict(shape="4b", batch=4, prompt=30720, steps=1024, kv_fill=True),
    "9b-b1": dict(shape="9b", batch=1, prompt=4096, steps=1024),
    "9b-b8": dict(shape="9b", batch=8, prompt=4096, steps=1024),
    # time to first token on a 16384-token prompt (8192 pairs): config.prefill_s
    "4b-ttft": dict(shape="4b", batch=1, prompt=16384, steps=32),
}
METRIC = "accepted tokens/s/GPU (PIPO pair-decode step)"
NOMINAL_HBM_GBS = 8000.0  # GB300 HBM3e nominal (~8 TB/s), context beside the measured peak
REF_BUDGET_S = 150.0      # reference arm: about this many seconds of timed oracle steps


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=None)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--workload", default="9b-b8", choices=sorted(WORKLOADS))
    ap.add_argument("--impl", default="pipo", choices=["pipo", "reference"])
    ap.add_argument("--tau", type=float, default=None)
    ap.add_argument("--force", type=int, default=0, help="0 rule, 1 accept all, 2 reject all")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--family-replays", type=int, default=None,
                    help="timed replays of the projection-only graph for the roofline (default: the step count, "
                         "at most 256)")
    ap.add_argument("--prefill-rows", type=int, default=128,
                    help="prefill in chunks of this many rows (positions x sequences, at most 128); "
                         "0: one position at a time")
    ap.add_argument("--sampler", action="store_true",
                    help="decode with the paper's evaluation sampler in both heads (T 1, top-k 20, top-p 0.95, "
                         "repetition penalty 1.5; seeded draws) instead of the greedy argmax")
    ap.add_argument("--regular", action="store_true",
                    help="also time regular decoding (one token per backbone pass, Sec. 4) on the same prompts "
                         "and report its time per output token beside the pair step's")
    return ap.parse_args()


# ---------------------------------------------------------------- clocks

class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.rows = []
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            threading.Thread(target=self._read, daemon=True).start()
            time.sleep(0.3)
        except OSError:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) == 8:
                self.rows.append(parts)

    def __exit__(self, *a):
        if self.proc:
            time.sleep(0.15)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        if not self.rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        sm = [float(r[0]) for r in self.rows if r[0].replace(".", "").isdigit()]
        mx = [float(r[1]) for r in self.rows if r[1].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in self.rows for i in range(4) if r[4 + i].lower().startswith("active")})
        pw = [float(r[2]) for r in self.rows if r[2].replace(".", "").isdigit()]
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(self.rows), "power_w_max": max(pw) if pw else None}


# ---------------------------------------------------------------- helpers

def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return d["hbm_gbs"], d.get("bf16_tflops"), "measured"
    return 6800.0, 1900.0, "fallback"


def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    return int(os.environ.get("RANK", "0")), ws, int(os.environ.get("LOCAL_RANK", "0"))


def aggregate_ranks(ms, tokens, e2e_s, e2e_tokens, device):
    """Whole-job figures over the ranks of a torch.distributed job: the
    slowest rank's times (max) and the tokens of all ranks (sum).  A single
    process returns its own figures."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return ms, tokens, e2e_s, e2e_tokens
    t = torch.tensor([ms, tokens, e2e_s, e2e_tokens], dtype=torch.float64, device=device)
    mx = t.clone()
    dist.all_reduce(mx, op=dist.ReduceOp.MAX)
    sm = t.clone()
    dist.all_reduce(sm, op=dist.ReduceOp.SUM)
    return float(mx[0]), float(sm[1]), float(mx[2]), float(sm[3])


def build_weights(shape, device):
    from paper_2605_27255_gb300 import synth
    return synth.gen_weights(shape, seed=0, device=device)


def oracle_sample(shape, weights_host, batch, n_ctx, tau, force, budget_s, max_steps=None):
    """Time the fp64 oracle on a bounded sample of the workload: decode
    steps of `batch` sequences at context n_ctx, caches filled with seeded
    values (the oracle's time does not depend on them)."""
    import numpy as np
    import torch

    from oracle import oracle as O
    from paper_2605_27255_gb300 import synth
    cap = max_steps or 256
    model = O.Model(shape, weights_host, max_ctx=n_ctx + cap + 1)
    st = O.State(model, batch)
    dev = "cuda" if torch.cuda.is_available() else "cpu"
    K, V = synth.gen_kv_fill(shape, n_ctx, seed=7, device=dev)
    K, V = K.cpu().numpy(), V.cpu().numpy()
    prompts = synth.gen_prompts(batch, 2, shape.V, seed=1).numpy()
    for b in range(batch):
        st.set_cache(b, K, V)
    st.set_pending(np.stack([prompts[:, 0], prompts[:, 1]], 1))
    del K, V
    steps, toks, t0 = 0, 0, time.perf_counter()
    while True:
        o = st.step(tau=tau, force=force, logits=False)
        steps += 1
        toks += int(batch + o["n_acc"].sum())
        el = time.perf_counter() - t0
        if el >= budget_s or steps >= cap:
            break
    return dict(seconds=el, steps=steps, tokens=toks)


# ---------------------------------------------------------------- reference arm

def run_reference(args):
    rank, ws, _ = dist_env()
    if rank != 0:
        return
    import torch

    from paper_2605_27255_gb300 import synth
    wl = WORKLOADS[args.workload]
    shape = synth.PRESETS[wl["shape"]]
    tau = shape.tau if args.tau is None else args.tau
    dev = "cuda" if torch.cuda.is_available() else "cpu"
    w = {k: v.cpu() for k, v in build_weights(shape, dev).items()}
    n_ctx = (wl["prompt"] + 1) // 2
    K = args.steps if args.steps is not None else 8
    W = args.warmup
    cores = os.cpu_count()
    # one untimed step, then K timed steps whose sample is bounded: the
    # oracle decodes sequences one after another, so fewer sequences per step
    # keep the tokens/s and bound the run to about REF_BUDGET_S
    B = wl["batch"]
    t1 = oracle_sample(shape, w, B, n_ctx, tau, args.force, 0.0, max_steps=1)
    per_seq_step = t1["seconds"] / B
    nb = B
    while nb > 1 and K * per_seq_step * nb > REF_BUDGET_S:
        nb //= 2
    r = oracle_sample(shape, w, nb, n_ctx, tau, args.force, 1e9, max_steps=K)
    tps = r["tokens"] / r["seconds"]
    line = {
        "impl": "reference", "metric": METRIC, "value": tps, "unit": "tokens/s", "n_gpus": ws, "steps": K,
        "warmup": W, "ms_per_step": 1e3 * r["seconds"] / r["steps"], "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic (seeded)",
        "config": {"workload": args.workload, "shape": wl["shape"], "batch": wl["batch"],
                   "context_entries": n_ctx, "tau": tau, "force_mode": args.force},
        "cpu_baseline": {"value": tps, "unit": "tokens/s", "cores": cores, "kind": "oracle",
                         "sample": f"{r['steps']} fp64 oracle decode steps of {nb} of the workload's {B} "
                                   f"sequence(s) at context {n_ctx}, caches filled with seeded values "
                                   f"({r['seconds']:.1f} s)"},
        "e2e": {"value": tps, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# ---------------------------------------------------------------- GPU arm

def run_regular(g, shape, wl, B, T, W, K, stream, seed):
    """Regular decoding on the same context and prompts: T prompt tokens take
    T cache entries, then W untimed and K timed steps of one token per
    sequence (CUDA events on the context stream)."""
    import torch

    from paper_2605_27255_gb300 import roofline, synth

    prompts = synth.gen_prompts(B, T if not wl.get("kv_fill") else 2, shape.V, seed=seed).numpy()
    t_pf = time.perf_counter()
    g.regular_prefill(prompts)  # synchronous
    t_pf = time.perf_counter() - t_pf
    if wl.get("kv_fill"):
        Kf, Vf = synth.gen_kv_fill(shape, T, seed=7, device="cuda")
        Kf, Vf = Kf.cpu().numpy(), Vf.cpu().numpy()
        for b in range(B):
            g.load_cache(b, Kf, Vf)
        del Kf, Vf
    for _ in range(W):
        g.regular_step_async()
    torch.cuda.synchronize()
    n0, e0 = g.counters()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for _ in range(K):
        g.regular_step_async()
    ev1.record(stream)
    torch.cuda.synchronize()
    ms = ev0.elapsed_time(ev1)
    n1, e1 = g.counters()
    tokens = int((e1 - e0).sum())
    ctx_avg = float(n0.mean()) + (K - 1) / 2.0
    step_bytes = roofline.regular_step_bytes(shape, B, ctx_avg)
    # the pair prefill of the same prompts once more, warm like the regular one
    pipo_pf = None
    if not wl.get("kv_fill"):
        pipo_pf = time.perf_counter()
        g.prefill(prompts)
        pipo_pf = time.perf_counter() - pipo_pf
    return {"ms_per_step": ms / K, "ms_per_token": ms / K, "tokens_per_s": tokens / (ms / 1e3),
            "context_entries_avg": ctx_avg, "steps": K, "gpu_launches": g.launches() * K,
            "step_bytes": step_bytes, "achieved_gbs": step_bytes / (ms / K / 1e3) / 1e9,
            "prefill_s": None if wl.get("kv_fill") else t_pf, "pipo_prefill_warm_s": pipo_pf,
            "note": "one token per backbone pass from the token embedding, final-norm tied LM head; tpot_ratio = "
                    "regular time per output token / pair-step time per output token (1 + acceptance tokens)"}


def make_line(m: dict) -> dict:
    """The benchmark's JSON line from the measured quantities of run_pipo
    (device time over the timed steps, graph replays of the projection and
    attention families, end-to-end loop, oracle baseline, clocks)."""
    K, B, hbm = m["steps"], m["batch"], m["hbm"]
    step_ms = m["ms"] / K
    step_gbs = m["step_bytes"] / (step_ms / 1e3) / 1e9
    fp, fa = m["fam"][0], m["fam"][1]
    proj_gbs = fp["bytes"] / (fp["ms"] / 1e3) / 1e9 if fp["ms"] > 0 else None
    attn_gbs = fa["bytes"] / (fa["ms"] / 1e3) / 1e9 if fa["ms"] > 0 else None
    acceptance = m["tokens"] / (K * B) - 1.0
    tr = m.get("traffic") or {}
    line = {
        "metric": METRIC, "value": m["tokens_all"] / (m["ms_all"] / 1e3), "unit": "tokens/s",
        "n_gpus": m["n_gpus"], "steps": K, "warmup": m["warmup"], "ms_per_step": m["ms_all"] / K,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": m["dtype"], "data": "synthetic (seeded weights and prompts)",
        "config": {"workload": m["workload"], "shape": m["shape_name"], "batch": B, "prompt_tokens": m["prompt_tokens"],
                   "context_entries_avg": m["ctx_avg"], "tau": m["tau"], "force_mode": m["force"],
                   "acceptance": acceptance, "pair_step_us": 1e3 * step_ms,
                   "prefill_s": m["prefill_s"], "prefill_rows": m["prefill_rows"],
                   "heads": "sampled (T 1, top-k 20, top-p 0.95, penalty 1.5)" if m["sampler"] else "greedy",
                   "l2": "weights streamed per step (GBs) > 129 MB L2; no flush needed",
                   "parallelism": f"replicas x{m['n_gpus']}"},
        "roofline": {"bound": "hbm", "kernel": f"weight-streaming projections (every projection and both LM-head "
                                                  f"launches of a step): {m['desc']}",
                     "achieved": proj_gbs, "peak": hbm, "unit": "GB/s",
                     "frac": (proj_gbs / hbm) if proj_gbs else None,
                     "traffic": tr.get("bytes_per_launch"),
                     "traffic_source": tr.get("source"),
                     "algorithmic_bytes_per_launch": fp["bytes"] / max(1, fp["launches"]),
                     "avg_launch_us": 1e3 * fp["ms"] / max(1, fp["launches"]),
                     "launches_per_step": fp["launches"],
                     "family_ms_per_step": fp["ms"],
                     "family_share_of_step": fp["ms"] / step_ms,
                     "timing": f"CUDA events on the context stream around {fp['replays']} replays of a graph of "
                               f"the step's projection launches alone (the step's launch plan, order and "
                               f"programmatic dependent launch), right after the timed steps",
                     "peak_source": f"{m['peak_source']} (MEASURED_PEAKS.json hbm_gbs)",
                     "step": {"algorithmic_bytes": m["step_bytes"], "achieved": step_gbs, "frac": step_gbs / hbm,
                              "frac_of_nominal": step_gbs / NOMINAL_HBM_GBS},
                     "attention": {"achieved": attn_gbs, "frac": (attn_gbs / hbm) if attn_gbs else None,
                                   "algorithmic_bytes_per_step": fa["bytes"], "launches_per_step": fa["launches"],
                                   "family_ms_per_step": fa["ms"], "family_share_of_step": fa["ms"] / step_ms}},
        "cpu_baseline": m["cpu"],
        "e2e": {"value": m["e2e_tokens"] / m["e2e_s"], "unit": "tokens/s",
                "h2d_bytes_per_step": B * 8, "d2h_bytes_per_step": B * 12,
                "loop": "host-driven: pipo_set_pending (pending pair from pinned host memory) + pipo_decode_step "
                        "(tokens and acceptances back), synchronous"},
        "gpu_launches": m["launches"] * K,
        "clocks": m["clocks"],
    }
    if m.get("prefill_s") and m.get("prefill_flops") and m.get("bf16_tflops"):
        # the prefill is tensor-bound (positions x sequences through the projections)
        tflops = m["prefill_flops"] / m["prefill_s"] / 1e12
        line["prefill"] = {"seconds": m["prefill_s"], "pair_positions": (m["prompt_tokens"] + 1) // 2,
                           "flops": m["prefill_flops"], "achieved_tflops": tflops,
                           "peak_tflops": m["bf16_tflops"], "frac": tflops / m["bf16_tflops"],
                           "bound": "tensor",
                           "timing": "host clock around the first pipo_prefill call of the context (its one-time "
                                     "set-up included), the time to first token"}
    regular = m.get("regular")
    if regular is not None:
        pipo_tpot = step_ms / (1.0 + acceptance)
        regular["tpot_ratio"] = regular["ms_per_token"] / pipo_tpot
        regular["frac"] = regular["achieved_gbs"] / hbm
        # time to first token on the same prompt: T tokens as T positions against T / 2 pairs (both warm)
        regular["ttft_ratio"] = (regular["prefill_s"] / regular["pipo_prefill_warm_s"]) \
            if regular["prefill_s"] and regular["pipo_prefill_warm_s"] else None
        line["regular"] = regular
    return line


def time_family(g, family, n, stream):
    """CUDA-event time of one replay of a kernel family's graph (ms), with its
    algorithmic bytes and launches per replay."""
    import torch
    by, nl = g.replay_family(family, 3)  # capture + warm-up
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    ev0.record(stream)
    g.replay_family(family, n)
    ev1.record(stream)
    torch.cuda.synchronize()
    return {"ms": ev0.elapsed_time(ev1) / n, "bytes": by, "launches": nl, "replays": n}


def run_pipo(args):
    import numpy as np
    import torch

    from paper_2605_27255_gb300 import capi, roofline, synth

    rank, ws, local = dist_env()
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    torch.cuda.set_device(local)
    wl = WORKLOADS[args.workload]
    shape = synth.PRESETS[wl["shape"]]
    tau = shape.tau if args.tau is None else args.tau
    B, T = wl["batch"], wl["prompt"]
    K = args.steps if args.steps is not None else wl["steps"]
    W = max(3, args.warmup)
    n_pairs = (T + 1) // 2
    max_ctx = n_pairs + W + 2 * K + 9
    if args.regular:
        max_ctx = max(max_ctx, T + W + K + 8)  # regular decoding: one cache entry per token

    w = build_weights(shape, "cuda")
    if args.prefill_rows:
        os.environ["PIPO_PREFILL_ROWS"] = str(args.prefill_rows)  # read when the context is created
    g = capi.Pipo(shape, w, max_batch=B, max_ctx=max_ctx, tau=tau, force_mode=args.force)
    w_host = None
    if rank == 0 and not args.no_cpu_baseline:
        w_host = {k: v.cpu() for k, v in w.items()}
    del w
    torch.cuda.empty_cache()
    stream = torch.cuda.Stream()
    g.set_stream(stream.cuda_stream)
    if args.sampler:
        # draws for every position that runs the heads (prefill, warm-up, timed, e2e, profile steps)
        n_u = 1 + W + 2 * K + 9
        u = np.random.default_rng(11 + rank).random((n_u, B, 2)).astype(np.float32)
        g.set_sampler(u, temperature=1.0, top_k=20, top_p=0.95, rep_penalty=1.5)

    prompts = synth.gen_prompts(B, T if not wl.get("kv_fill") else 2, shape.V, seed=1 + rank * 1000).numpy()
    t_pf = time.perf_counter()
    torch.cuda.nvtx.range_push("prefill")  # ncu --nvtx --nvtx-include "prefill/": the prefill's launches
    g.prefill(prompts)
    torch.cuda.nvtx.range_pop()
    t_pf = time.perf_counter() - t_pf
    if wl.get("kv_fill"):
        Kf, Vf = synth.gen_kv_fill(shape, n_pairs, seed=7, device="cuda")
        Kf, Vf = Kf.cpu().numpy(), Vf.cpu().numpy()
        for b in range(B):
            g.load_cache(b, Kf, Vf)
        del Kf, Vf

    for _ in range(W):
        g.step_async()
    torch.cuda.synchronize()
    n0, e0 = g.counters()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if ws > 1:
        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(torch.cuda.current_device()) as clk:
        ev0.record(stream)
        for _ in range(K):
            g.step_async()
        ev1.record(stream)
        torch.cuda.synchronize()
    if ws > 1:
        dist.barrier()
    ms = ev0.elapsed_time(ev1)
    n1, e1 = g.counters()
    tokens = int((e1 - e0).sum())
    ctx_avg = float(n0.mean()) + (K - 1) / 2.0
    # end to end through the public host API, a host-driven decode loop: every
    # step copies its input, the pending pair (the previous step's output pair,
    # 8 bytes per sequence), from pinned host memory to the device
    # (pipo_set_pending) and reads its outputs back (12 bytes per sequence)
    tok_h = torch.empty((B, 2), dtype=torch.int32, pin_memory=True)
    nacc_h = torch.empty((B,), dtype=torch.int32, pin_memory=True)
    import ctypes as C
    lib = capi.load()
    tok_p, nacc_p = C.cast(tok_h.data_ptr(), capi._IP), C.cast(nacc_h.data_ptr(), capi._IP)

    def e2e_check(rc):
        if rc != 0:
            raise capi.PipoError(rc, capi.pipo_last_error(g.ctx))

    e2e_check(lib.pipo_decode_step(g.ctx, tok_p, nacc_p))  # untimed: the first pair on the host
    _, e2a = g.counters()
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(K):
        # a refused pair means the previous step returned an id outside [0, V): a failed run
        e2e_check(lib.pipo_set_pending(g.ctx, tok_p))
        e2e_check(lib.pipo_decode_step(g.ctx, tok_p, nacc_p))
    e2e_s = time.perf_counter() - t0
    _, e2b = g.counters()
    e2e_tokens = int((e2b - e2a).sum())
    launches = g.launches()
    desc = g.describe()
    # the projection family and the attention family of the same step, each a
    # graph of its own launches replayed back to back (decode state unchanged)
    n_rep = args.family_replays or max(8, min(K, 256))
    fam = {0: time_family(g, 0, n_rep, stream), 1: time_family(g, 1, n_rep, stream)}
    # one more graph-replayed step inside an NVTX range: ncu --nvtx --nvtx-include "ncu_step/"
    # takes the launch list of exactly this step (untimed here)
    torch.cuda.nvtx.range_push("ncu_step")
    g.step_async()
    torch.cuda.synchronize()
    torch.cuda.nvtx.range_pop()
    regular = run_regular(g, shape, wl, B, T, W, K, stream, 1 + rank * 1000) if args.regular else None

    ms_all, tokens_all, e2e_all, e2e_tok_all = aggregate_ranks(ms, tokens, e2e_s, e2e_tokens, "cuda")
    hbm, tf, src = peaks()

    cpu = None
    if rank == 0 and not args.no_cpu_baseline and w_host is not None:
        nb = B if B <= 4 else 1
        try:
            r = oracle_sample(shape, w_host, nb, n_pairs, tau, args.force, args.cpu_seconds)
            cpu = {"value": r["tokens"] / r["seconds"], "unit": "tokens/s", "cores": os.cpu_count(),
                   "kind": "oracle",
                   "sample": f"{r['steps']} fp64 oracle decode step(s) of {nb} sequence(s) at context {n_pairs}, "
                             f"caches filled with seeded values ({r['seconds']:.1f} s)"}
        except Exception as e:  # the GPU line stands without its CPU baseline
            cpu = {"value": None, "unit": "tokens/s", "cores": os.cpu_count(), "kind": "oracle",
                   "error": f"{type(e).__name__}: {e}"}
    if rank != 0:
        if ws > 1:
            dist.destroy_process_group()
        return
    line = make_line(dict(
        workload=args.workload, shape_name=wl["shape"], dtype=shape.dtype, n_gpus=ws, steps=K, warmup=W, batch=B,
        prompt_tokens=T, ms=ms, ms_all=ms_all, tokens=tokens, tokens_all=tokens_all, ctx_avg=ctx_avg, tau=tau,
        force=args.force, prefill_s=t_pf, prefill_rows=args.prefill_rows, sampler=args.sampler, desc=desc, fam=fam,
        hbm=hbm, peak_source=src, step_bytes=roofline.step_bytes(shape, B, ctx_avg), bf16_tflops=tf,
        prefill_flops=None if wl.get("kv_fill") else roofline.prefill_flops(shape, B, (T + 1) // 2),
        traffic=roofline.recorded_traffic(os.path.join(ROOT, "profiles"), args.workload),
        cpu=cpu, e2e_s=e2e_all, e2e_tokens=e2e_tok_all, launches=launches,
        clocks=clk.summary(), regular=regular))
    print(json.dumps(line), flush=True)
    g.close()
    if ws > 1:
        dist.destroy_process_group()


def main():
    args = parse()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_pipo(args)


if __name__ == "__main__":
    main()
