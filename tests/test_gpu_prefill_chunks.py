"""Prefill in chunks (PIPO_PREFILL_ROWS=<rows>): the prompt positions before
the last go through the projections C positions x B sequences at a time,
each block appending the chunk's keys and values before its attention.

Checked against the fp64 oracle (prefill outputs, then forced-replay decode
steps that read the chunk-written caches), against the position-by-position
prefill of the same context shape (cache contents and outputs), for pair and
regular decoding, with ragged last chunks and several sequences.
"""
import os

import numpy as np
import pytest

from oracle import oracle as O
from paper_2605_27255_gb300 import capi, synth
from parity_util import MARGIN, run_forced_replay, tol_for

pytestmark = pytest.mark.gpu

MID = synth.ModelShape("mid", H=512, L=3, n_q=8, n_kv=2, d_h=128, F=1376, V=5003,
                       compressor="mlp", mtp_block=1, dtype="bf16", rope_theta=1e6, tau=0.5)


@pytest.mark.parametrize("attn", ["rows", "tile"])
@pytest.mark.parametrize("rows,B,T", [(16, 1, 150), (16, 2, 149), (128, 1, 300), (128, 4, 97), (128, 16, 40)])
def test_chunked_pair_prefill_matches_oracle(monkeypatch, attn, rows, B, T):
    """rows / B positions per chunk; T tokens give (T + 1) / 2 pairs, of which
    all but the last run in chunks (the last chunk ragged).  attn: one
    decode-style CTA per row, or causal tiles of positions
    (PIPO_PREFILL_ATTN=tile, attn_prefill_kernel)."""
    monkeypatch.setenv("PIPO_PREFILL_ROWS", str(rows))
    if attn == "tile":
        monkeypatch.setenv("PIPO_PREFILL_ATTN", "tile")
    w = synth.gen_weights(MID, seed=3)
    prompts = synth.gen_prompts(B, T, MID.V, seed=7).numpy()
    st = run_forced_replay(MID, w, prompts, 6)
    assert st.tok_checked >= 0.5 * st.tok_total


@pytest.mark.parametrize("variant", ["paper", "literal"])
def test_chunked_pair_prefill_tiny_fp32(monkeypatch, variant):
    monkeypatch.setenv("PIPO_PREFILL_ROWS", "24")
    s = synth.TINY.with_(mtp_block=1 if variant == "paper" else 0)
    w = synth.gen_weights(s, seed=0)
    prompts = synth.gen_prompts(3, 63, s.V, seed=1).numpy()  # 32 pairs: chunks of 8, 8, 8, 7, then the last
    st = run_forced_replay(s, w, prompts, 8)
    assert st.tok_checked >= 0.5 * st.tok_total


def _prefill_state(shape, w, prompts, rows, regular=False):
    if rows:
        os.environ["PIPO_PREFILL_ROWS"] = str(rows)
    else:
        os.environ.pop("PIPO_PREFILL_ROWS", None)
    B, T = prompts.shape
    n = T if regular else (T + 1) // 2
    g = capi.Pipo(shape, w, max_batch=B, max_ctx=n + 4, debug=True)
    try:
        out = g.regular_prefill(prompts) if regular else g.prefill(prompts)
        d = g.debug()
        layers = shape.L + (0 if regular or not shape.mtp_block else 1)
        caches = [[g.read_cache(b, l, n) for l in range(layers)] for b in range(B)]
        nxt = g.regular_step() if regular else g.step()
        return out, d, caches, nxt, g.counters()
    finally:
        g.close()
        os.environ.pop("PIPO_PREFILL_ROWS", None)


def test_tile_attention_equals_row_attention(monkeypatch):
    """The two chunk attentions read the same cache entries: caches and
    outputs agree within the rounding of the summation order."""
    s = MID
    w = synth.gen_weights(s, seed=8)
    prompts = synth.gen_prompts(3, 121, s.V, seed=2).numpy()  # 61 pairs: chunks of 42 rows (14 positions)
    a = _prefill_state(s, w, prompts, 42)
    monkeypatch.setenv("PIPO_PREFILL_ATTN", "tile")
    b = _prefill_state(s, w, prompts, 42)
    tol = tol_for(s)
    for cb_a, cb_b in zip(a[2], b[2]):
        for (Ka, Va), (Kb, Vb) in zip(cb_a, cb_b):
            scale = max(1.0, float(np.abs(Ka).max()), float(np.abs(Va).max()))
            assert np.abs(Ka - Kb).max() <= 2 * tol * scale
            assert np.abs(Va - Vb).max() <= 2 * tol * scale
    assert np.abs(a[1]["logits_b"] - b[1]["logits_b"]).max() <= 2 * tol


@pytest.mark.parametrize("regular", [False, True])
def test_chunked_equals_position_by_position(regular):
    """Same context shape, same prompts: the chunk-written caches hold the
    same entries as the position-by-position ones up to the rounding of the
    cache type (the projections sum in another order), and the outputs agree."""
    s = MID
    w = synth.gen_weights(s, seed=5)
    prompts = synth.gen_prompts(2, 70, s.V, seed=9).numpy()
    a = _prefill_state(s, w, prompts, 0, regular)
    b = _prefill_state(s, w, prompts, 32, regular)
    tol = tol_for(s)
    for cb_a, cb_b in zip(a[2], b[2]):
        for (Ka, Va), (Kb, Vb) in zip(cb_a, cb_b):
            scale = max(1.0, float(np.abs(Ka).max()), float(np.abs(Va).max()))
            assert np.abs(Ka - Kb).max() <= 2 * tol * scale
            assert np.abs(Va - Vb).max() <= 2 * tol * scale
    assert np.abs(a[1]["logits_b"] - b[1]["logits_b"]).max() <= 2 * tol
    assert list(a[4][0]) == list(b[4][0])  # cache lengths


@pytest.mark.parametrize("attn", ["rows", "tile"])
def test_chunked_regular_prefill_matches_oracle(monkeypatch, attn):
    monkeypatch.setenv("PIPO_PREFILL_ROWS", "64")
    if attn == "tile":
        monkeypatch.setenv("PIPO_PREFILL_ATTN", "tile")
    s = MID
    w = synth.gen_weights(s, seed=6)
    B, T = 2, 90  # 89 positions in chunks of 32, 32, 25, then the last
    prompts = synth.gen_prompts(B, T, s.V, seed=4).numpy()
    g = capi.Pipo(s, w, max_batch=B, max_ctx=T + 6, debug=True)
    try:
        orc = O.State(O.Model(s, w, max_ctx=T + 6), B)
        tok, _ = g.regular_prefill(prompts)
        o = orc.regular_prefill(prompts)
        tol = tol_for(s)
        for step in range(5):
            d = g.debug()
            for b in range(B):
                assert np.abs(d["logits_b"][b] - o["logits_b"][b]).max() <= tol, f"step {step} b={b}"
                if o["margin_b"][b] > MARGIN:
                    assert tok[b, 0] == o["tokens"][b, 0]
            g.set_pending([[orc.seq(b)["p0"], -1] for b in range(B)])
            tok = g.regular_step()
            o = orc.regular_step()
        n, _ = g.counters()
        assert list(n) == [T + 5] * B
    finally:
        g.close()


@pytest.mark.parametrize("attn", ["rows", "tile"])
def test_chunked_prefill_4b(monkeypatch, attn):
    """The 4B shapes of the benchmark: a 300-token prompt (150 pairs) in
    chunks of 128 rows at B = 1, then forced-replay steps, against the oracle."""
    monkeypatch.setenv("PIPO_PREFILL_ROWS", "128")
    if attn == "tile":
        monkeypatch.setenv("PIPO_PREFILL_ATTN", "tile")
    s = synth.B4
    w = synth.gen_weights(s, seed=0, device="cuda")
    host = {k: v.cpu() for k, v in w.items()}
    prompts = synth.gen_prompts(1, 300, s.V, seed=3).numpy()
    st = run_forced_replay(s, w, prompts, 3, oracle_weights=host)
    assert st.tok_checked >= 0.8 * st.tok_total
    del w
