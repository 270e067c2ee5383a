"""Continuous batching on the GPU (pipo_prefill_slot): sequences of
different prompt lengths in one batch, and a sequence joining a batch that is
already decoding.  Each slot is checked against its own oracle sequence (a
batch is B independent sequences), with forced replay of the pending pairs.
"""

import numpy as np
import pytest

from oracle import oracle as O
from paper_2605_27255_gb300 import capi, synth
from parity_util import Stats, compare, tol_for

pytestmark = pytest.mark.gpu

MID = synth.ModelShape("mid", H=512, L=3, n_q=8, n_kv=2, d_h=128, F=1376, V=5003,
                       compressor="mlp", mtp_block=1, dtype="bf16", rope_theta=1e6, tau=0.5)


def _row(d, b):
    """Row b of a debug dump as a batch of one."""
    return {k: v[b:b + 1] for k, v in d.items()}


def _check_rows(shape, gpu, orcs, outs, tok, nacc, st, where):
    d = gpu.debug()
    for b, o in enumerate(outs):
        if o is None:
            continue
        compare(shape, shape.tau, o, _row(d, b), tok[b:b + 1], nacc[b:b + 1], 0, st, tol_for(shape), f"{where} slot {b}")


@pytest.mark.parametrize("shape", [synth.TINY, MID])
def test_ragged_prompts_by_slot(shape):
    w = synth.gen_weights(shape, seed=4)
    lens = [37, 20, 52]
    prompts = [synth.gen_prompts(1, n, shape.V, seed=10 + i).numpy()[0] for i, n in enumerate(lens)]
    max_ctx = max(lens) // 2 + 12
    gpu = capi.Pipo(shape, w, max_batch=3, max_ctx=max_ctx, debug=True, page_shuffle_seed=5)
    try:
        orcs = [O.State(O.Model(shape, w, max_ctx=max_ctx), 1) for _ in lens]
        st = Stats()
        tok = np.zeros((3, 2), np.int32)
        nacc = np.zeros(3, np.int32)
        for b in (2, 0, 1):  # any order; each slot prefill writes only its own rows
            t, a = gpu.prefill_slot(b, prompts[b])
            tok[b], nacc[b] = t[0], a[0]
        outs = [orcs[b].prefill(prompts[b][None, :], tau=shape.tau) for b in range(3)]
        _check_rows(shape, gpu, orcs, outs, tok, nacc, st, "prefill")
        for i in range(6):
            gpu.set_pending([[orcs[b].seq(0)["p0"], orcs[b].seq(0)["p1"]] for b in range(3)])
            tok, nacc = gpu.step()
            outs = [orcs[b].step(tau=shape.tau) for b in range(3)]
            _check_rows(shape, gpu, orcs, outs, tok, nacc, st, f"step {i}")
        n, _ = gpu.counters()
        assert list(n) == [orcs[b].seq(0)["n"] for b in range(3)]
        assert st.tok_checked >= 0.5 * st.tok_total
    finally:
        gpu.close()


def test_a_sequence_joins_a_decoding_batch():
    shape = MID
    w = synth.gen_weights(shape, seed=6)
    p0 = synth.gen_prompts(1, 40, shape.V, seed=1).numpy()[0]
    p1 = synth.gen_prompts(1, 25, shape.V, seed=2).numpy()[0]
    max_ctx = 40
    gpu = capi.Pipo(shape, w, max_batch=2, max_ctx=max_ctx, debug=True)
    try:
        o0 = O.State(O.Model(shape, w, max_ctx=max_ctx), 1)
        o1 = O.State(O.Model(shape, w, max_ctx=max_ctx), 1)
        st = Stats()
        tok, nacc = gpu.prefill_slot(0, p0)
        out0 = o0.prefill(p0[None, :], tau=shape.tau)
        _check_rows(shape, gpu, [o0], [out0], tok, nacc, st, "slot 0 prefill")
        for i in range(3):  # slot 0 decodes alone
            gpu.set_pending([[o0.seq(0)["p0"], o0.seq(0)["p1"]]])
            tok, nacc = gpu.step()
            _check_rows(shape, gpu, [o0], [o0.step(tau=shape.tau)], tok, nacc, st, f"alone {i}")
        tok1, nacc1 = gpu.prefill_slot(1, p1)  # joins; slot 0 keeps its state
        out1 = o1.prefill(p1[None, :], tau=shape.tau)
        d = gpu.debug()
        compare(shape, shape.tau, out1, _row(d, 1), tok1, nacc1, 0, st, tol_for(shape), "slot 1 prefill")
        for i in range(4):  # both decode
            gpu.set_pending([[o.seq(0)["p0"], o.seq(0)["p1"]] for o in (o0, o1)])
            tok, nacc = gpu.step()
            outs = [o0.step(tau=shape.tau), o1.step(tau=shape.tau)]
            _check_rows(shape, gpu, [o0, o1], outs, tok, nacc, st, f"together {i}")
        n, e = gpu.counters()
        assert list(n) == [o0.seq(0)["n"], o1.seq(0)["n"]]
        assert list(e) == [o0.seq(0)["emitted"], o1.seq(0)["emitted"]]
    finally:
        gpu.close()


def test_slot_errors():
    s = synth.TINY
    w = synth.gen_weights(s, seed=0)
    g = capi.Pipo(s, w, max_batch=2, max_ctx=8)
    try:
        ids = synth.gen_prompts(1, 10, s.V, seed=1).numpy()[0]
        with pytest.raises(capi.PipoError):
            g.prefill_slot(2, ids)  # slot out of range
        with pytest.raises(capi.PipoError):
            g.prefill_slot(0, np.concatenate([ids, ids]))  # 10 pairs > 8 entries
        bad = ids.copy()
        bad[3] = s.V
        with pytest.raises(capi.PipoError):
            g.prefill_slot(1, bad)
        g.regular_prefill(ids[None, :8])
        with pytest.raises(capi.PipoError):
            g.prefill_slot(0, ids)  # regular mode
    finally:
        g.close()


@pytest.mark.parametrize("shape", [synth.TINY, MID])
def test_ragged_batch_prefill(shape):
    """pipo_prefill with prompts of different pair counts (each prefilled as a
    slot) against the oracle's ragged prefill, then forced-replay steps."""
    from parity_util import run_forced_replay
    w = synth.gen_weights(shape, seed=9)
    lens = np.array([37, 20, 52], np.int32)
    prompts = synth.gen_prompts(3, 52, shape.V, seed=3).numpy()
    st = run_forced_replay(shape, w, prompts, 5, lens=lens)
    assert st.tok_checked >= 0.5 * st.tok_total
