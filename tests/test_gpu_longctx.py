"""Long-context parity: caches filled with seeded entries (many 64-entry
pages per attention split) on both sides, then forced-replay decode steps
against the oracle: at 1500 entries the split-KV attention with 8-CTA
clusters (default) and 16-CTA clusters (opt-in), and one sequence on the
deep stage ring; at 2500 entries the unclustered tensor-core attention."""
import os

import numpy as np
import pytest

from oracle import oracle as O
from paper_2605_27255_gb300 import capi, synth
from parity_util import Stats, compare, tol_for

pytestmark = pytest.mark.gpu

MID = synth.ModelShape("mid", H=512, L=3, n_q=8, n_kv=2, d_h=128, F=1376, V=5003,
                       compressor="mlp", mtp_block=1, dtype="bf16", rope_theta=1e6, tau=0.5)


@pytest.mark.parametrize("cs16", ["1", "0"])
def test_long_context_forced_replay(cs16, monkeypatch):
    monkeypatch.setenv("PIPO_ATTN_CS16", cs16)
    s = MID
    n_ctx, B, steps = 1500, 2, 3
    w = synth.gen_weights(s, seed=8)
    K, V = synth.gen_kv_fill(s, n_ctx, seed=9)
    K, V = K.numpy(), V.numpy()
    prompts = synth.gen_prompts(B, 4, s.V, seed=4).numpy()
    gpu = capi.Pipo(s, w, max_batch=B, max_ctx=n_ctx + steps + 2, debug=True, page_shuffle_seed=3)
    orc = O.State(O.Model(s, w, max_ctx=n_ctx + steps + 2), B)
    try:
        tok, _ = gpu.prefill(prompts)
        orc.prefill(prompts, tau=s.tau)
        for b in range(B):
            gpu.load_cache(b, K, V)
            orc.set_cache(b, K, V)
        st = Stats()
        for i in range(steps):
            pend = [[orc.seq(b)["p0"], orc.seq(b)["p1"]] for b in range(B)]
            gpu.set_pending(pend)
            tok, nacc = gpu.step()
            o = orc.step(tau=s.tau)
            compare(s, s.tau, o, gpu.debug(), tok, nacc, 0, st, tol_for(s), f"step {i}")
        n, _ = gpu.counters()
        assert list(n) == [n_ctx + steps] * B
    finally:
        gpu.close()


@pytest.mark.parametrize("B", [1, 2])
def test_long_context_unclustered_tensor_core_attention(B):
    """From 2048 cached pairs, when 8-CTA clusters would leave SMs idle, the
    tensor-core attention splits each (sequence, kv head) over unclustered
    CTAs whose partials the last arrival merges through global memory."""
    s = MID
    n_ctx, steps = 2500, 3
    w = synth.gen_weights(s, seed=18)
    K, V = synth.gen_kv_fill(s, n_ctx, seed=19)
    K, V = K.numpy(), V.numpy()
    prompts = synth.gen_prompts(B, 4, s.V, seed=14).numpy()
    gpu = capi.Pipo(s, w, max_batch=B, max_ctx=n_ctx + steps + 2, debug=True, page_shuffle_seed=5)
    orc = O.State(O.Model(s, w, max_ctx=n_ctx + steps + 2), B)
    try:
        gpu.prefill(prompts)
        orc.prefill(prompts, tau=s.tau)
        for b in range(B):
            gpu.load_cache(b, K, V)
            orc.set_cache(b, K, V)
        st = Stats()
        for i in range(steps):
            pend = [[orc.seq(b)["p0"], orc.seq(b)["p1"]] for b in range(B)]
            gpu.set_pending(pend)
            tok, nacc = gpu.step()
            if i == 0:
                d = gpu.describe()
                assert "attention=attn_mma_kernel unclustered splits=" in d, d
            o = orc.step(tau=s.tau)
            compare(s, s.tau, o, gpu.debug(), tok, nacc, 0, st, tol_for(s), f"step {i}")
        n, _ = gpu.counters()
        assert list(n) == [n_ctx + steps] * B
    finally:
        gpu.close()


@pytest.mark.parametrize("cs", ["2", "8"])
def test_long_context_deep_ring(cs, monkeypatch):
    """One sequence with each cluster CTA on an SM of its own takes the deep
    stage ring: with 2-CTA clusters a CTA's slice of 1500 entries spans about
    47 groups of 16, so every stage is refilled while the warps compute; with
    8 the whole slice is in flight from the CTA's entry."""
    monkeypatch.setenv("PIPO_ATTN_CS", cs)
    s = MID
    n_ctx, B, steps = 1500, 1, 3
    w = synth.gen_weights(s, seed=28)
    K, V = synth.gen_kv_fill(s, n_ctx, seed=29)
    K, V = K.numpy(), V.numpy()
    prompts = synth.gen_prompts(B, 4, s.V, seed=24).numpy()
    gpu = capi.Pipo(s, w, max_batch=B, max_ctx=n_ctx + steps + 2, debug=True, page_shuffle_seed=7)
    orc = O.State(O.Model(s, w, max_ctx=n_ctx + steps + 2), B)
    try:
        gpu.prefill(prompts)
        orc.prefill(prompts, tau=s.tau)
        gpu.load_cache(0, K, V)
        orc.set_cache(0, K, V)
        st = Stats()
        for i in range(steps):
            gpu.set_pending([[orc.seq(0)["p0"], orc.seq(0)["p1"]]])
            tok, nacc = gpu.step()
            if i == 0:
                d = gpu.describe()
                assert f"attention=attn_mma_kernel cluster={cs} stages=20" in d, d
            o = orc.step(tau=s.tau)
            compare(s, s.tau, o, gpu.debug(), tok, nacc, 0, st, tol_for(s), f"step {i}")
        n, _ = gpu.counters()
        assert list(n) == [n_ctx + steps]
    finally:
        gpu.close()
