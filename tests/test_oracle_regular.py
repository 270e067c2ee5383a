"""Pins of the oracle's regular decoding, the baseline the paper compares PIPO
with (Sec. 4, "Regular"): one token per backbone pass, input E[t], position =
token index, final-norm tied LM head, greedy argmax.  CPU only."""
import numpy as np
import pytest
import torch

from oracle import oracle as O
from paper_2605_27255_gb300 import synth

SMALL = synth.ModelShape("reg", H=64, L=2, n_q=4, n_kv=2, d_h=16, F=96, V=257, compressor="linear",
                         mtp_block=1, dtype="f32", rope_theta=1.0e4, tau=0.5)


def _weights(shape, seed=0):
    return synth.gen_weights(shape, seed=seed, device="cpu")


def _rms(x, g, eps):
    return x / np.sqrt(np.mean(x * x) + eps) * g


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_identity_blocks_give_the_embedding_closed_form(dtype):
    """With every block's O and down projection zero, each block is the
    identity on the residual, so the next token is argmax_v E_v . RMSNorm(E[t])
    (no compressor on the input, the final norm before the tied head)."""
    s = synth.ModelShape("reg", H=64, L=2, n_q=4, n_kv=2, d_h=16, F=96, V=257, compressor="mlp", mtp_block=1,
                         dtype=dtype, rope_theta=1.0e4, tau=0.5)
    w = _weights(s, 3)
    w["blk.Wo"] = torch.zeros_like(w["blk.Wo"])
    w["blk.Wdown"] = torch.zeros_like(w["blk.Wdown"])
    w["final_norm"] = (1.0 + 0.25 * torch.linspace(-1, 1, s.H)).to(w["final_norm"].dtype)
    E = w["E"].double().numpy()
    g = w["final_norm"].double().numpy()
    ids = np.array([[5, 77, 200, 13]], np.int32)
    st = O.State(O.Model(s, w, max_ctx=16), 1)
    o = st.regular_prefill(ids)
    ref = E @ _rms(E[13], g, s.eps)
    assert np.allclose(o["logits_b"][0], ref, rtol=0, atol=1e-12)
    t = int(np.argmax(ref))
    assert o["tokens"][0, 0] == t and o["tokens"][0, 1] == -1 and o["n_acc"][0] == 0
    for _ in range(3):  # each step feeds back the previous argmax
        o = st.regular_step()
        ref = E @ _rms(E[t], g, s.eps)
        assert np.allclose(o["logits_b"][0], ref, rtol=0, atol=1e-12)
        t = int(np.argmax(ref))
        assert o["tokens"][0, 0] == t
    assert st.seq(0)["n"] == 4 + 3 and st.seq(0)["emitted"] == 3


def test_regular_equals_pipo_with_first_slot_compressor():
    """A Linear compressor W = [I 0], b = 0 maps the pair (t, PAD) to E[t]; PIPO
    fed the pairs (t_j, PAD) then runs the backbone exactly as regular decoding
    of t_0, t_1, ... does (position j, one cache entry each): equal logits."""
    s = SMALL
    w = _weights(s, 5)
    H = s.H
    w["comp.W"] = torch.cat([torch.eye(H), torch.zeros(H, H)], 1).to(w["comp.W"].dtype)
    w["comp.b"] = torch.zeros_like(w["comp.b"])
    toks = [11, 200, 3, 3, 150, 42]
    reg = O.State(O.Model(s, w, max_ctx=16), 1)
    o = reg.regular_prefill(np.array([toks[:1]], np.int32))
    reg_logits = [o["logits_b"][0].copy()]
    for t in toks[1:]:
        reg.set_pending([[t, -1]])
        reg_logits.append(reg.regular_step()["logits_b"][0].copy())
    pipo = O.State(O.Model(s, w, max_ctx=16), 1)
    o = pipo.prefill(np.array([toks[:1]], np.int32))  # one pair (t_0, PAD) at position 0
    pipo_logits = [o["logits_b"][0].copy()]
    for t in toks[1:]:
        pipo.set_pending([[t, -1]])
        pipo_logits.append(pipo.step()["logits_b"][0].copy())
    for j, (a, b) in enumerate(zip(reg_logits, pipo_logits)):
        assert np.array_equal(a, b), f"position {j}"
    # and the causal history matters: a different earlier token changes later logits
    other = O.State(O.Model(s, w, max_ctx=16), 1)
    other.regular_prefill(np.array([[12]], np.int32))
    other.set_pending([[toks[1], -1]])
    assert not np.allclose(other.regular_step()["logits_b"][0], reg_logits[1])


def test_prefill_of_a_prefix_then_steps_equals_prefill_of_the_whole():
    s = synth.ModelShape("reg", H=64, L=2, n_q=4, n_kv=2, d_h=16, F=96, V=257, compressor="mlp", mtp_block=1,
                         dtype="bf16", rope_theta=1.0e4, tau=0.5)
    w = _weights(s, 7)
    toks = np.array([[9, 30, 31, 250, 7, 7, 100]], np.int32)
    whole = O.State(O.Model(s, w, max_ctx=16), 1).regular_prefill(toks)
    part = O.State(O.Model(s, w, max_ctx=16), 1)
    part.regular_prefill(toks[:, :4])
    for t in toks[0, 4:]:
        part.set_pending([[int(t), -1]])
        o = part.regular_step()
    assert np.array_equal(o["logits_b"], whole["logits_b"])
    assert part.seq(0)["n"] == 7


def test_regular_errors():
    s = SMALL
    w = _weights(s, 1)
    st = O.State(O.Model(s, w, max_ctx=4), 1)
    with pytest.raises(ValueError):
        st.regular_prefill(np.array([[1, 2, 3, 4, 5]], np.int32))  # 5 tokens > 4 entries
    with pytest.raises(ValueError):
        st.regular_prefill(np.array([[1, s.V]], np.int32))  # id out of range
    st.regular_prefill(np.array([[1, 2, 3]], np.int32))
    st.regular_step()  # entry 3: the last one
    with pytest.raises(ValueError):
        st.regular_step()  # the cache is full
