"""More GPU invariants of the pair-decode path:

* re-prefill: prefill(prompt) then k accept-all steps leaves the same caches
  and the same next outputs as prefill(prompt + the emitted tokens) (every
  emitted pair is a full pair under accept-all, so the history is a plain
  token sequence whose pairs, positions and teacher-forced MTP tokens are
  those the steps used);
* the widest batch of the tensor-core path (B = 128, batch width 128)
  against the fp64 oracle;
* pipo_decode_steps (n steps per call) equals n single steps.
"""

import numpy as np
import pytest

from paper_2605_27255_gb300 import capi, synth
from parity_util import run_forced_replay, tol_for

pytestmark = pytest.mark.gpu

MID = synth.ModelShape("mid", H=512, L=3, n_q=8, n_kv=2, d_h=128, F=1376, V=5003,
                       compressor="mlp", mtp_block=1, dtype="bf16", rope_theta=1e6, tau=0.5)


@pytest.mark.parametrize("shape", [synth.TINY, MID])
def test_reprefill_of_the_emitted_history(shape):
    w = synth.gen_weights(shape, seed=12)
    B, T, k = 2, 30, 5
    prompts = synth.gen_prompts(B, T, shape.V, seed=13).numpy()
    max_ctx = T // 2 + k + 4
    a = capi.Pipo(shape, w, max_batch=B, max_ctx=max_ctx, force_mode=1, debug=True)
    b = capi.Pipo(shape, w, max_batch=B, max_ctx=max_ctx, force_mode=1, debug=True)
    try:
        tok, _ = a.prefill(prompts)
        hist = [tok.copy()]
        for _ in range(k):
            tok, _ = a.step()
            hist.append(tok.copy())
        # the pairs consumed after the prompt: the outputs of the prefill and
        # of the first k - 1 steps; the last output is the pending pair
        consumed = np.concatenate([h for h in hist[:-1]], axis=1)  # [B, 2k]
        assert (consumed >= 0).all()  # accept-all: no PAD
        b_tok, _ = b.prefill(np.concatenate([prompts, consumed], axis=1).astype(np.int32))
        assert np.array_equal(b_tok, hist[-1])
        n_a, _ = a.counters()
        n_b, _ = b.counters()
        assert list(n_a) == list(n_b) == [T // 2 + k] * B
        tol = tol_for(shape)
        for s in range(B):
            for layer in range(shape.L + 1):
                Ka, Va = a.read_cache(s, layer, int(n_a[s]))
                Kb, Vb = b.read_cache(s, layer, int(n_b[s]))
                scale = max(1.0, float(np.abs(Ka).max()), float(np.abs(Va).max()))
                assert np.abs(Ka - Kb).max() <= tol * scale and np.abs(Va - Vb).max() <= tol * scale
        ta, _ = a.step()
        tb, _ = b.step()
        assert np.abs(a.debug()["logits_b"] - b.debug()["logits_b"]).max() <= 2 * tol
    finally:
        a.close()
        b.close()


def test_widest_tensor_core_batch():
    w = synth.gen_weights(MID, seed=14)
    prompts = synth.gen_prompts(128, 12, MID.V, seed=15).numpy()
    st = run_forced_replay(MID, w, prompts, 2)
    assert st.tok_checked >= 0.5 * st.tok_total


@pytest.mark.parametrize("shape", [synth.TINY, MID])
def test_multi_step_call_equals_single_steps(shape):
    w = synth.gen_weights(shape, seed=16)
    prompts = synth.gen_prompts(3, 21, shape.V, seed=17).numpy()
    a = capi.Pipo(shape, w, max_batch=3, max_ctx=24)
    b = capi.Pipo(shape, w, max_batch=3, max_ctx=24)
    try:
        a.prefill(prompts)
        b.prefill(prompts)
        tok, nacc = a.steps(6)
        for i in range(6):
            t, n = b.step()
            assert np.array_equal(tok[i], t) and np.array_equal(nacc[i], n)
        assert list(a.counters()[0]) == list(b.counters()[0])
        with pytest.raises(capi.PipoError):
            a.steps(100)  # beyond max_ctx: refused before any step runs
        assert list(a.counters()[0]) == list(b.counters()[0])
    finally:
        a.close()
        b.close()
