"""GPU path vs the fp64 oracle through the C ABI (forced replay).

Sizes: the Tiny configuration (fp32, 64-token prompt, 32 steps), a bf16
model with ragged dimensions spanning several GEMV tiles, KV pages and
split-KV slices, and batches.  Full-size shapes are in test_gpu_fullsize.py.
"""
import numpy as np
import pytest
import torch

from paper_2605_27255_gb300 import capi, synth
from parity_util import run_forced_replay

pytestmark = pytest.mark.gpu

# bf16, ragged: F and V are not multiples of the 256-element GEMV stride, V of
# the row tiles; head_dim 128 with 4 query heads per KV head (as the 4B shape).
MID = synth.ModelShape("mid", H=512, L=3, n_q=8, n_kv=2, d_h=128, F=1376, V=5003,
                       compressor="mlp", mtp_block=1, dtype="bf16", rope_theta=1e6, tau=0.5)


@pytest.mark.parametrize("variant", ["paper", "literal"])
def test_tiny_fp32_forced_replay(variant):
    # "paper": MTP head = W_fc + one decoder block; "literal": W_fc only
    s = synth.TINY.with_(mtp_block=1 if variant == "paper" else 0)
    w = synth.gen_weights(s, seed=0)
    prompts = synth.gen_prompts(1, 64, s.V, seed=1).numpy()
    st = run_forced_replay(s, w, prompts, 32)
    assert st.tok_checked >= 0.5 * st.tok_total


def test_tiny_mlp_compressor_batch3_odd_prompts():
    s = synth.TINY.with_(compressor="mlp")
    w = synth.gen_weights(s, seed=2)
    prompts = synth.gen_prompts(3, 63, s.V, seed=5).numpy()
    st = run_forced_replay(s, w, prompts, 10)
    assert st.tok_checked >= 0.5 * st.tok_total


@pytest.mark.parametrize("force", [0, 1, 2])
def test_mid_bf16_forced_modes(force):
    w = synth.gen_weights(MID, seed=3)
    prompts = synth.gen_prompts(2, 150, MID.V, seed=7).numpy()  # 75 pairs: two KV pages
    st = run_forced_replay(MID, w, prompts, 12, force=force, page_shuffle_seed=11)
    assert st.tok_checked >= 0.5 * st.tok_total


def test_mid_bf16_tau_sweep():
    w = synth.gen_weights(MID, seed=4)
    prompts = synth.gen_prompts(1, 40, MID.V, seed=8).numpy()
    for tau in (0.3, 0.5, 0.7):
        run_forced_replay(MID, w, prompts, 4, tau=tau)


def test_page_layout_does_not_change_results():
    """Any permutation of the physical KV blocks gives bit-identical outputs."""
    s = MID
    w = synth.gen_weights(s, seed=5)
    prompts = synth.gen_prompts(2, 200, s.V, seed=9).numpy()
    outs = []
    for seed in (0, 12345):
        g = capi.Pipo(s, w, max_batch=2, max_ctx=120, debug=True, page_shuffle_seed=seed)
        r = [g.prefill(prompts)]
        for _ in range(6):
            r.append(g.step())
        r.append(g.debug()["logits_b"].copy())
        g.close()
        outs.append(r)
    for a, b in zip(*outs):
        if isinstance(a, tuple):
            assert all(np.array_equal(x, y) for x, y in zip(a, b))
        else:
            assert np.array_equal(a, b)


def test_batch_equals_independent_sequences_gpu():
    s = MID
    w = synth.gen_weights(s, seed=6)
    prompts = synth.gen_prompts(3, 30, s.V, seed=10).numpy()
    g = capi.Pipo(s, w, max_batch=3, max_ctx=40, debug=True)
    g.prefill(prompts)
    for _ in range(3):
        g.step()
    lb = g.debug()["logits_b"].copy()
    g.close()
    for b in range(3):
        g1 = capi.Pipo(s, w, max_batch=1, max_ctx=40, debug=True)
        g1.prefill(prompts[b:b + 1])
        for _ in range(3):
            g1.step()
        # not bit-exact: a different batch size picks another GEMV batch tile
        assert np.abs(g1.debug()["logits_b"][0] - lb[b]).max() < 2e-3
        g1.close()


def test_rollback_restores_state_gpu():
    """Append 5 entries, roll back 5: the caches, lengths and the next step
    equal those of a context that never appended (bit-exact)."""
    s = MID
    w = synth.gen_weights(s, seed=7)
    prompts = synth.gen_prompts(2, 60, s.V, seed=11).numpy()
    g = capi.Pipo(s, w, max_batch=2, max_ctx=50, debug=True)
    tok0, _ = g.prefill(prompts)
    n0, _ = g.counters()
    ref = capi.Pipo(s, w, max_batch=2, max_ctx=50, debug=True)
    ref.prefill(prompts)
    before = [g.read_cache(b, l, int(n0[b])) for b in range(2) for l in range(s.L + 1)]
    for _ in range(5):
        g.step()
    g.rollback(n0)
    g.set_pending(tok0)
    after = [g.read_cache(b, l, int(n0[b])) for b in range(2) for l in range(s.L + 1)]
    for (k0, v0), (k1, v1) in zip(before, after):
        assert np.array_equal(k0, k1) and np.array_equal(v0, v1)
    n1, _ = g.counters()
    assert list(n1) == list(n0)
    for _ in range(2):
        a, b = g.step(), ref.step()
        assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1])
        assert np.array_equal(g.debug()["logits_b"], ref.debug()["logits_b"])
    g.close()
    ref.close()


def test_errors_are_status_codes():
    s = synth.TINY
    w = synth.gen_weights(s, seed=0)
    g = capi.Pipo(s, w, max_batch=2, max_ctx=8)
    with pytest.raises(capi.PipoError) as e:
        g.step()
    assert e.value.status == capi.PIPO_ESTATE
    with pytest.raises(capi.PipoError) as e:
        g.prefill(np.array([[1, s.V]], np.int32))
    assert e.value.status == capi.PIPO_EINVAL
    with pytest.raises(capi.PipoError) as e:
        g.prefill(np.zeros((1, 40), np.int32))  # 20 pairs > 8
    assert e.value.status == capi.PIPO_ECAPACITY
    with pytest.raises(capi.PipoError) as e:
        g.prefill(np.zeros((3, 4), np.int32))  # batch > max_batch
    assert e.value.status == capi.PIPO_EINVAL
    g.prefill(np.zeros((1, 12), np.int32))  # 6 pairs
    g.step()
    g.step()
    with pytest.raises(capi.PipoError) as e:
        g.step()  # 9th entry > max_ctx 8
    assert e.value.status == capi.PIPO_ECAPACITY
    with pytest.raises(capi.PipoError) as e:
        g.rollback([9])
    assert e.value.status == capi.PIPO_EINVAL
    g.close()
