"""The evaluation sampler in both heads on the GPU (pipo_set_sampler) against
the oracle's (State.set_sampler), the same uniform draws on both sides.

Both sides decode freely (no forced replay: the sampler's history is the
sequence's own tokens).  Per position: logits within the model's tolerance;
x_b and x_d equal wherever the oracle's decision margin (orc_sample_ex)
exceeds DELTA; the accept decision equal wherever |c - tau| > DELTA.  A
decision inside the margin that comes out differently ends the comparison
(the histories part there); the tests require enough positions compared.
"""

import numpy as np
import pytest

from oracle import oracle as O
from paper_2605_27255_gb300 import capi, synth
from parity_util import tol_for

pytestmark = pytest.mark.gpu

PAPER = dict(temperature=1.0, top_k=20, top_p=0.95, rep_penalty=1.5)
SMALL_BF16 = synth.ModelShape("samp-bf16", H=512, L=2, n_q=8, n_kv=2, d_h=128, F=1408, V=4096,
                              compressor="mlp", mtp_block=1, dtype="bf16", rope_theta=1.0e6, tau=0.5)


def _delta(shape):
    return 5e-2 if shape.dtype == "bf16" else 1e-3


def _free_run(shape, w, prompts, steps, cfg, n_u=None, seed=0, tau=0.5):
    """Returns the number of positions whose decisions were all compared."""
    B, T = prompts.shape
    n_u = n_u or steps + 1
    u = np.random.default_rng(seed).random((n_u, B, 2)).astype(np.float32)
    max_ctx = (T + 1) // 2 + steps + 2
    gpu = capi.Pipo(shape, w, max_batch=B, max_ctx=max_ctx, tau=tau, debug=True)
    try:
        gpu.set_sampler(u, **cfg)
        orc = O.State(O.Model(shape, w, max_ctx=max_ctx), B)
        orc.set_sampler(**cfg)
        tol, delta = tol_for(shape), _delta(shape)
        tok, nacc = gpu.prefill(prompts)
        o = orc.prefill(prompts, u=u[0].astype(np.float64), tau=tau)
        compared = 0
        for i in range(steps + 1):
            d = gpu.debug()
            assert np.abs(d["logits_b"] - o["logits_b"]).max() <= tol, f"position {i}"
            same = True
            for b in range(B):
                for key, mkey in (("x_b", "margin_b"), ("x_d", "margin_d")):
                    if o[mkey][b] > delta:
                        assert d[key][b] == o[key][b], f"position {i} b={b} {key}"
                    elif d[key][b] != o[key][b]:
                        same = False
                if abs(float(o["conf"][b]) - tau) > delta:
                    assert nacc[b] == o["n_acc"][b], f"position {i} b={b} accept"
                elif nacc[b] != o["n_acc"][b]:
                    same = False
            if not same:
                return compared
            assert np.array_equal(tok, o["tokens"]), f"position {i}"
            # the draft head ran on the same x_b on both sides
            assert np.abs(d["logits_d"] - o["logits_d"]).max() <= tol, f"position {i}"
            compared += 1
            if i == steps:
                break
            tok, nacc = gpu.step()
            o = orc.step(u=u[(i + 1) % n_u].astype(np.float64), tau=tau)
        return compared
    finally:
        gpu.close()


def test_paper_sampler_tiny_fp32():
    s = synth.TINY
    w = synth.gen_weights(s, seed=0)
    prompts = synth.gen_prompts(2, 40, s.V, seed=1).numpy()
    assert _free_run(s, w, prompts, 12, PAPER, seed=3) >= 4


def test_sampler_draw_ring_wraps():
    s = synth.TINY.with_(compressor="mlp")
    w = synth.gen_weights(s, seed=2)
    prompts = synth.gen_prompts(3, 25, s.V, seed=4).numpy()
    cfg = dict(temperature=0.7, top_k=8, top_p=0.8, rep_penalty=1.3)
    assert _free_run(s, w, prompts, 9, cfg, n_u=3, seed=5) >= 3


@pytest.mark.parametrize("B", [1, 4])
def test_paper_sampler_bf16(B):
    w = synth.gen_weights(SMALL_BF16, seed=3)
    prompts = synth.gen_prompts(B, 30, SMALL_BF16.V, seed=2).numpy()
    assert _free_run(SMALL_BF16, w, prompts, 6, PAPER, seed=7) >= 2


@pytest.mark.parametrize("shape", [synth.TINY, SMALL_BF16])
def test_top1_sampling_equals_greedy_on_the_gpu(shape):
    """top_k = 1 without a penalty picks the argmax: the same tokens and,
    since the same kernels run, bit-identical logits as the greedy context."""
    w = synth.gen_weights(shape, seed=1)
    B = 2
    prompts = synth.gen_prompts(B, 24, shape.V, seed=3).numpy()
    u = np.random.default_rng(0).random((4, B, 2)).astype(np.float32)
    a = capi.Pipo(shape, w, max_batch=B, max_ctx=24, debug=True)
    g = capi.Pipo(shape, w, max_batch=B, max_ctx=24, debug=True)
    try:
        a.set_sampler(u, temperature=1.0, top_k=1, top_p=0.95, rep_penalty=1.0)
        ra, rg = [a.prefill(prompts)], [g.prefill(prompts)]
        for _ in range(5):
            ra.append(a.step())
            rg.append(g.step())
            assert np.array_equal(a.debug()["logits_b"], g.debug()["logits_b"])
        for x, y in zip(ra, rg):
            assert all(np.array_equal(p, q) for p, q in zip(x, y))
    finally:
        a.close()
        g.close()


def test_sampler_argument_errors():
    s = synth.TINY
    w = synth.gen_weights(s, seed=0)
    g = capi.Pipo(s, w, max_batch=1, max_ctx=16)
    try:
        u = np.full((2, 1, 2), 0.5, np.float32)
        for bad in (dict(top_k=0), dict(top_k=33), dict(top_p=0.0), dict(top_p=1.5), dict(rep_penalty=0.0)):
            with pytest.raises(capi.PipoError):
                g.set_sampler(u, **bad)
        with pytest.raises(capi.PipoError):
            g.set_sampler(np.full((2, 1, 2), 1.0, np.float32))  # a draw of 1 is outside [0, 1)
        with pytest.raises(capi.PipoError):
            g.set_sampler(np.zeros((0, 1, 2), np.float32))  # no draws
        g.set_sampler(u, temperature=0.0)  # off again: greedy
        g.prefill(synth.gen_prompts(1, 8, s.V, seed=1).numpy())
        g.step()
    finally:
        g.close()


def test_paper_sampler_4b():
    """The 4B shapes (V = 151936): the full-vocabulary selection of the
    sampler kernel against the oracle's sort."""
    s = synth.B4
    w = synth.gen_weights(s, seed=0, device="cuda")
    host = {k: v.cpu() for k, v in w.items()}
    prompts = synth.gen_prompts(1, 40, s.V, seed=2).numpy()
    u = np.random.default_rng(9).random((5, 1, 2)).astype(np.float32)
    max_ctx = 40
    gpu = capi.Pipo(s, w, max_batch=1, max_ctx=max_ctx, debug=True)
    try:
        gpu.set_sampler(u, **PAPER)
        orc = O.State(O.Model(s, host, max_ctx=max_ctx), 1)
        orc.set_sampler(**PAPER)
        tok, nacc = gpu.prefill(prompts)
        o = orc.prefill(prompts, u=u[0].astype(np.float64), tau=s.tau)
        for i in range(4):
            d = gpu.debug()
            assert np.abs(d["logits_b"] - o["logits_b"]).max() <= tol_for(s)
            if (o["margin_b"][0] <= _delta(s) or o["margin_d"][0] <= _delta(s)
                    or abs(float(o["conf"][0]) - s.tau) <= _delta(s)):
                break  # a decision inside its margin: the histories may part here
            assert d["x_b"][0] == o["x_b"][0] and d["x_d"][0] == o["x_d"][0]
            assert nacc[0] == o["n_acc"][0]
            tok, nacc = gpu.step()
            o = orc.step(u=u[i + 1].astype(np.float64), tau=s.tau)
    finally:
        gpu.close()
        del w
