"""Pins of the fp64 oracle against closed forms, special cases and
brute force (paper Sec. 3.1-3.2, Eq. 1-6, App. A).  CPU only.

Each test fixes a value that the mathematics or the paper determines, so that
a plausible slip in the oracle (a dropped term, a sign, an index, a transposed
operand, a wrong norm axis) fails at least one of them.
"""
import cmath
import math

import numpy as np
import pytest
import torch

from oracle import oracle as O
from paper_2605_27255_gb300 import synth

LN3 = math.log(3.0)


# ---------------------------------------------------------------- primitives

def test_round_bf16_matches_torch_and_ties_to_even():
    # ties: 1 + 2^-8 lies halfway between 1 and 1 + 2^-7 -> even (1.0)
    assert O.round_bf16(1.0 + 2.0 ** -8) == 1.0
    # 1 + 3*2^-8 lies halfway between 1+2^-7 (odd) and 1+2^-6 (even)
    assert O.round_bf16(1.0 + 3 * 2.0 ** -8) == 1.0 + 2.0 ** -6
    rng = np.random.default_rng(0)
    xs = rng.standard_normal(2000).astype(np.float32) * 10.0 ** rng.integers(-3, 3, 2000)
    ref = torch.from_numpy(xs).to(torch.bfloat16).double().numpy()
    got = np.array([O.round_bf16(float(x)) for x in xs])
    assert np.array_equal(got, ref)


def test_rmsnorm_closed_forms():
    # [3,4]: mean square 12.5 -> [3,4]/sqrt(12.5) = [3 sqrt2/5, 4 sqrt2/5]
    y = O.rmsnorm([3.0, 4.0], [1.0, 1.0], eps=0.0)
    assert np.allclose(y, [3 * math.sqrt(2) / 5, 4 * math.sqrt(2) / 5], rtol=0, atol=1e-15)
    # gains multiply per element (sign included)
    y = O.rmsnorm([3.0, 4.0], [2.0, -1.0], eps=0.0)
    assert np.allclose(y, [6 * math.sqrt(2) / 5, -4 * math.sqrt(2) / 5], atol=1e-15)
    # eps sits inside the root, added to the mean square: x = 1e-3 everywhere,
    # eps = 1e-6 -> 1e-3 / sqrt(2e-6) = 1/sqrt(2)
    y = O.rmsnorm(np.full(7, 1e-3), np.ones(7), eps=1e-6)
    assert np.allclose(y, 1 / math.sqrt(2), atol=1e-12)
    # zero vector stays zero (no division by zero)
    assert np.all(O.rmsnorm(np.zeros(5), np.ones(5)) == 0)


def test_matvec_is_row_major_out_by_in():
    rng = np.random.default_rng(1)
    W = rng.standard_normal((5, 9)).astype(np.float32)
    x = rng.standard_normal(9)
    assert np.allclose(O.matvec(W, x), W.astype(np.float64) @ x, atol=1e-12)


def test_silu_sigmoid_closed_forms():
    assert O.sigmoid(0.0) == 0.5
    assert abs(O.sigmoid(LN3) - 0.75) < 1e-15          # 1/(1+1/3)
    assert abs(O.sigmoid(-LN3) - 0.25) < 1e-15
    assert abs(O.silu(LN3) - 0.75 * LN3) < 1e-15       # x * sigma(x)
    assert O.silu(0.0) == 0.0


def test_rope_is_complex_rotation_rotate_half_pairs():
    theta = 100.0
    d = 4
    v = np.array([0.3, -1.2, 0.7, 2.0])
    for pos in (0, 1, 5, 37):
        got = O.rope(v, 1, d, pos, theta)
        # pairs (i, i+d/2) as complex numbers v_i + 1j v_{i+d/2}, frequency theta^(-2i/d)
        for i in range(d // 2):
            w = complex(v[i], v[i + d // 2]) * cmath.exp(1j * pos * theta ** (-2.0 * i / d))
            assert abs(got[i] - w.real) < 1e-12 and abs(got[i + d // 2] - w.imag) < 1e-12
    assert np.array_equal(O.rope(v, 1, d, 0, theta), v)


def test_rope_relative_position_and_norm():
    rng = np.random.default_rng(2)
    d, theta = 16, 1e4
    q, k = rng.standard_normal(d), rng.standard_normal(d)
    dots = [np.dot(O.rope(q, 1, d, m + s, theta), O.rope(k, 1, d, n + s, theta))
            for (m, n, s) in ((7, 3, 0), (7, 3, 11), (7, 3, 1000))]
    assert np.allclose(dots, dots[0], atol=1e-9)
    assert abs(np.linalg.norm(O.rope(q, 1, d, 123, theta)) - np.linalg.norm(q)) < 1e-12
    # two heads rotate independently and identically
    two = O.rope(np.concatenate([q, k]), 2, d, 9, theta)
    assert np.allclose(two[:d], O.rope(q, 1, d, 9, theta)) and np.allclose(two[d:], O.rope(k, 1, d, 9, theta))


def test_attention_single_entry_returns_value():
    rng = np.random.default_rng(3)
    d, nq, nkv = 8, 4, 2
    q = rng.standard_normal(nq * d)
    K = rng.standard_normal((1, nkv * d))
    V = rng.standard_normal((1, nkv * d))
    out = O.attend(q, K, V, nq, nkv, d).reshape(nq, d)
    # GQA: query heads 0,1 read kv head 0; heads 2,3 read kv head 1
    for h in range(nq):
        g = h // (nq // nkv)
        assert np.allclose(out[h], V[0, g * d:(g + 1) * d], atol=1e-15)


def test_attention_softmax_scale_is_inverse_sqrt_d():
    # scores ln3 apart after scaling by 1/sqrt(d): weights 3/4 and 1/4
    d = 16
    q = np.zeros(d); q[0] = 1.0
    K = np.zeros((2, d)); K[0, 0] = LN3 * math.sqrt(d); K[1, 0] = 0.0
    V = np.zeros((2, d)); V[0, :] = 1.0; V[1, :] = -3.0
    out = O.attend(q, K, V, 1, 1, d)
    assert np.allclose(out, 0.75 * 1.0 + 0.25 * -3.0, atol=1e-14)


def test_argmax_lowest_index_on_ties_and_margin():
    i, m = O.argmax([0.1, 0.9, 0.3, 0.9, -2.0])
    assert i == 1 and m == 0.0
    i, m = O.argmax([0.1, 0.2, 0.7, 0.4])
    assert i == 2 and abs(m - 0.3) < 1e-15


# ------------------------------------------------------- model construction

def small_shape(**kw):
    base = dict(name="pin", H=8, L=1, n_q=4, n_kv=2, d_h=2, F=12, V=8,
                compressor="linear", mtp_block=0, dtype="f32", rope_theta=1e4, tau=0.5)
    base.update(kw)
    return synth.ModelShape(**base)


def zero_model(s):
    """All projections zero and all gains one: every block is the identity."""
    w = {}
    for name, shape in synth.tensor_shapes(s).items():
        w[name] = torch.ones(shape) if synth.is_gain(name) else torch.zeros(shape)
    return w


def onehot_model(s, perm):
    """E = I (V = H), compressor [I I], MTP W_fc = [0 P], zero blocks,
    confidence W2 = 0 (so c = sigma(0) = 1/2)."""
    assert s.V == s.H
    w = zero_model(s)
    H = s.H
    w["E"] = torch.eye(H)
    w["comp.W"] = torch.cat([torch.eye(H), torch.eye(H)], 1)
    P = torch.zeros(H, H)
    for i, j in enumerate(perm):
        P[j, i] = 1.0
    w["mtp.W_fc"] = torch.cat([torch.zeros(H, H), P], 1)
    return w


def test_compressor_identity_pair_is_sum():
    # Eq. 1 / App. A.1: Linear W [a;b] + b with W = [I I], b = 0 gives a + b
    s = small_shape(V=16)
    w = zero_model(s)
    rng = torch.Generator().manual_seed(0)
    w["E"] = torch.randn(s.V, s.H, generator=rng)
    w["x_pad"] = torch.randn(s.H, generator=rng)
    w["comp.W"] = torch.cat([torch.eye(s.H), torch.eye(s.H)], 1)
    m = O.Model(s, w)
    z = O.compress(m, 3, 11)
    assert np.allclose(z, (w["E"][3] + w["E"][11]).double().numpy(), atol=1e-6)
    # the bias is added once
    w["comp.b"] = torch.arange(s.H, dtype=torch.float32)
    m = O.Model(s, w)
    assert np.allclose(O.compress(m, 3, 11), (w["E"][3] + w["E"][11] + w["comp.b"]).double().numpy(), atol=1e-6)
    # PAD in the second slot reads x_pad
    assert np.allclose(O.compress(m, 3, -1), (w["E"][3] + w["x_pad"] + w["comp.b"]).double().numpy(), atol=1e-6)
    # order matters: W = [I 0] keeps the first slot
    w["comp.W"] = torch.cat([torch.eye(s.H), torch.zeros(s.H, s.H)], 1)
    w["comp.b"] = torch.zeros(s.H)
    m = O.Model(s, w)
    assert np.allclose(O.compress(m, 3, 11), w["E"][3].double().numpy(), atol=1e-7)


def test_compressor_mlp_closed_form():
    # MLP variant W2 SiLU(W1 [a;b]): with W1 = [I I], W2 = 2I and a + b = ln3
    # per element, every output is 2 * ln3 * 3/4
    s = small_shape(compressor="mlp", V=4)
    w = zero_model(s)
    E = torch.zeros(s.V, s.H)
    E[1] = 0.25 * LN3
    E[2] = 0.75 * LN3
    w["E"] = E.to(torch.float32)
    w["comp.W1"] = torch.cat([torch.eye(s.H), torch.eye(s.H)], 1)
    w["comp.W2"] = 2 * torch.eye(s.H)
    m = O.Model(s, w)
    z = O.compress(m, 1, 2)
    expect = 2 * (float(E[1, 0]) + float(E[2, 0])) * 0.75  # ln3 in fp32, times sigma(ln3)
    x = float(E[1, 0]) + float(E[2, 0])
    expect = 2 * x / (1 + math.exp(-x))
    assert np.allclose(z, expect, atol=1e-12)
    assert abs(expect - 1.5 * LN3) < 1e-6
    # the nonlinearity sits between W1 and W2: a + b = 0 gives exactly 0
    assert np.all(O.compress(m, 0, 0) == 0)


def test_compressor_residual_form():
    """The residual MLP compressor (comp_residual): z = a + b + W2 SiLU(W1 [a;b]).
    With the branch zeroed (W2 = 0) it is exactly a + b, the paper's
    initial state of the compressor; otherwise it differs from the literal MLP
    by exactly a + b; a PAD slot contributes x_pad."""
    s = small_shape(compressor="mlp", V=16, comp_residual=1)
    w = zero_model(s)
    rng = torch.Generator().manual_seed(3)
    w["E"] = torch.randn(s.V, s.H, generator=rng)
    w["x_pad"] = torch.randn(s.H, generator=rng)
    w["comp.W1"] = torch.randn(s.H, 2 * s.H, generator=rng)
    m = O.Model(s, w)
    a, b, pad = (w["E"][5].double().numpy(), w["E"][9].double().numpy(), w["x_pad"].double().numpy())
    assert np.array_equal(O.compress(m, 5, 9), a + b)
    assert np.array_equal(O.compress(m, 5, -1), a + pad)
    w["comp.W2"] = torch.randn(s.H, s.H, generator=rng)
    res = O.compress(O.Model(s, w), 5, 9)
    lit = O.compress(O.Model(s.with_(comp_residual=0), w), 5, 9)
    assert np.allclose(res - lit, a + b, rtol=0, atol=1e-12)
    assert not np.allclose(lit, a + b)


def test_onehot_model_closed_form_tokens_and_acceptance():
    """With E = I, a [I I] compressor and identity blocks, h_b = e_t0 + e_t1,
    so the LM head's argmax is min(t0, t1) (a tie, lowest index wins); the MTP
    head sees RMSNorm(E[x_b]) through W_fc = [0 P], so x_d = P(x_b); with
    W2 = 0 the confidence is exactly 1/2 and tau = 1/2 accepts (c >= tau)."""
    s = small_shape(L=1)
    perm = [3, 6, 0, 7, 1, 5, 2, 4]
    m = O.Model(s, onehot_model(s, perm))
    st = O.State(m, 1)
    o = st.prefill([[5, 2]], tau=0.5)
    assert o["tokens"][0, 0] == 2 and o["tokens"][0, 1] == perm[2]
    assert o["conf"][0] == 0.5 and o["n_acc"][0] == 1
    assert st.seq(0) == dict(p0=2, p1=perm[2], n=1, emitted=2)
    # next step consumes (2, 0): argmax min(2, 0) = 0, draft perm[0] = 3
    o = st.step(tau=0.5)
    assert list(o["tokens"][0]) == [0, perm[0]]
    # tau just above 1/2 rejects; the pending pair then has PAD in slot 1
    o = st.step(tau=0.5 + 1e-12)
    assert list(o["tokens"][0]) == [min(0, 3), -1] and o["n_acc"][0] == 0
    assert st.seq(0)["p1"] == -1
    # PAD input: x_pad = 0, so z = e_{p0} alone and the argmax is p0
    o = st.step(tau=0.5)
    assert o["tokens"][0, 0] == 0
    assert st.seq(0)["n"] == 4 and st.seq(0)["emitted"] == 2 + 2 + 1 + 2


def test_mtp_input_order_and_block_identity():
    # W_fc = [I 0] reads RMSNorm(h_b) (first half), not the token embedding
    s = small_shape(L=1)
    w = onehot_model(s, list(range(8)))
    w["mtp.W_fc"] = torch.cat([torch.eye(s.H), torch.zeros(s.H, s.H)], 1)
    m = O.Model(s, w)
    st = O.State(m, 1)
    o = st.prefill([[6, 4]])
    # h_d = RMSNorm(e6 + e4): argmax over {4, 6} -> 4, the same as the backbone
    assert o["x_b"][0] == 4 and o["x_d"][0] == 4
    assert np.allclose(o["h_d"][0], O.rmsnorm(o["h_b"][0], np.ones(8)), atol=1e-12)


def test_confidence_joint_norm_over_2H():
    """App. A.3 normalises the concatenation [h_b; h_d] with one RMSNorm over
    2H.  With W1 = I on the h_b half and W2 = 1, the pre-sigmoid value is
    sum SiLU(h_b / rms([h_b; h_d])), which a per-half norm would not give."""
    s = small_shape(H=4, V=4, n_q=2, n_kv=1, d_h=2, F=4)
    w = zero_model(s)
    w["conf.W1"] = torch.cat([torch.eye(4), torch.zeros(4, 4)], 1)
    w["conf.W2"] = torch.ones(1, 4)
    m = O.Model(s, w)
    hb = np.array([1.0, 1.0, 1.0, 1.0])
    hd = np.array([3.0, 3.0, 3.0, 3.0])
    rms = math.sqrt((4 * 1 + 4 * 9) / 8 + 1e-6)
    x = 1.0 / rms
    expect = 1 / (1 + math.exp(-4 * x / (1 + math.exp(-x))))
    assert abs(O.confidence(m, hb, hd) - expect) < 1e-12
    # W2 = 0 gives exactly 1/2
    w["conf.W2"] = torch.zeros(1, 4)
    assert O.confidence(O.Model(s, w), hb, hd) == 0.5


def test_block_residual_paths():
    """A block with W_o = 0 and W_down = 0 is the identity (both residuals);
    with only W_down = 0, h changes by W_o a where a is the attention output,
    which at the first position is v itself (single entry)."""
    s = small_shape(L=1, V=8, H=8)
    w = onehot_model(s, list(range(8)))
    m = O.Model(s, w)
    st = O.State(m, 1)
    o = st.prefill([[1, 2]])
    assert np.allclose(o["h_b"][0], np.eye(8)[1] + np.eye(8)[2])
    # now W_v = I-slice, W_o = I-slice: at position 0 a = v = W_v RMSNorm(x)
    rng = torch.Generator().manual_seed(5)
    w["blk.Wv"][0] = torch.randn(s.n_kv * s.d_h, s.H, generator=rng)
    w["blk.Wo"][0] = torch.randn(s.H, s.n_q * s.d_h, generator=rng)
    m = O.Model(s, w)
    st = O.State(m, 1)
    o = st.prefill([[1, 2]])
    x = np.eye(8)[1] + np.eye(8)[2]
    y = O.rmsnorm(x, np.ones(8))
    v = w["blk.Wv"][0].double().numpy() @ y
    a = np.concatenate([v[(h // 2) * 2:(h // 2) * 2 + 2] for h in range(4)])
    assert np.allclose(o["h_b"][0], x + w["blk.Wo"][0].double().numpy() @ a, atol=1e-6)


def test_swiglu_gate_and_up_are_not_swapped():
    """FFN = W_down(SiLU(W_gate y) * W_up y).  With W_gate rows picking y_0,
    W_up rows picking 2 y_0 and W_down summing, the output is
    SiLU(y0) * 2 y0, which differs from y0 * SiLU(2 y0)."""
    s = small_shape(L=1, V=8, H=8, F=1)
    w = onehot_model(s, list(range(8)))
    w["blk.Wgate"][0] = torch.zeros(1, 8); w["blk.Wgate"][0][0, 0] = 1.0
    w["blk.Wup"][0] = torch.zeros(1, 8); w["blk.Wup"][0][0, 0] = 2.0
    w["blk.Wdown"][0] = torch.zeros(8, 1); w["blk.Wdown"][0][7, 0] = 1.0
    m = O.Model(s, w)
    o = O.State(m, 1).prefill([[0, 0]])
    x = 2 * np.eye(8)[0]
    y0 = O.rmsnorm(x, np.ones(8))[0]
    expect = x.copy(); expect[7] += (y0 / (1 + math.exp(-y0))) * 2 * y0
    assert np.allclose(o["h_b"][0], expect, atol=1e-12)


# ------------------------------------------------------------ gain wiring
#
# Every RMSNorm of the model has its own gain vector (backbone attention and
# FFN norms per layer, the final norm, the MTP input norms of h_b and of the
# token embedding, the MTP block's norms, the MTP post-norm, the joint
# confidence norm over 2H).  The pins below give every gain distinct values
# and fix the results in closed form or by a single-position numpy
# evaluation of the definitions, so a gain taken from the wrong norm, the
# wrong layer or the wrong half of the confidence norm fails one of them.

def _r(x, eps=1e-6):
    """x / sqrt(mean(x^2) + eps), the normalisation of an RMSNorm."""
    x = np.asarray(x, dtype=np.float64)
    return x / math.sqrt(np.mean(x * x) + eps)


def _silu(x):
    return x / (1.0 + np.exp(-x))


def _distinct_gains(w, rng):
    """Overwrite every gain with its own uniform draw in [0.5, 1.5]."""
    for name in list(w):
        if synth.is_gain(name):
            w[name] = torch.from_numpy(rng.uniform(0.5, 1.5, tuple(w[name].shape)).astype(np.float32))
    return w


@pytest.mark.parametrize("t0,t1", [(5, 2), (1, 6), (4, 4)])
def test_head_gains_final_post_and_mtp_inputs(t0, t1):
    """Eq. 3-5 and App. A.2 with E = I (V = H), a [I I] compressor and
    identity blocks, so h_b = e_t0 + e_t1 (2 e_t0 when t0 = t1):
      logits_b = E (g_final * r(h_b))            = g_final * r(h_b)
      W_fc = [0 P]:  h_d = P (g_e * r(E[x_b]))   (no MTP block)
      W_fc = [I 0]:  h_d = g_h * r(h_b)
      logits_d = g_post * r(h_d).
    Swapping the final and post gains, or the two MTP input gains, changes
    these values."""
    s = small_shape(L=1)
    perm = [3, 6, 0, 7, 1, 5, 2, 4]
    w = _distinct_gains(onehot_model(s, perm), np.random.default_rng(11))
    g = {k: w[k].double().numpy() for k in ("final_norm", "mtp.norm_h", "mtp.norm_e", "mtp.norm_post")}
    hb = np.zeros(8); hb[t0] += 1; hb[t1] += 1
    lb = g["final_norm"] * _r(hb)
    xb = int(np.argmax(lb))
    P = w["mtp.W_fc"][:, 8:].double().numpy()
    for wfc, hd in ((None, P @ (g["mtp.norm_e"] * _r(np.eye(8)[xb]))),
                    (torch.cat([torch.eye(8), torch.zeros(8, 8)], 1), g["mtp.norm_h"] * _r(hb))):
        if wfc is not None:
            w["mtp.W_fc"] = wfc
        o = O.State(O.Model(s, w), 1).prefill([[t0, t1]], tau=0.5)
        assert np.allclose(o["h_b"][0], hb, rtol=0, atol=1e-15)
        assert np.allclose(o["logits_b"][0], lb, rtol=0, atol=1e-12)
        assert o["x_b"][0] == xb
        assert np.allclose(o["h_d"][0], hd, rtol=0, atol=1e-12)
        assert np.allclose(o["logits_d"][0], g["mtp.norm_post"] * _r(hd), rtol=0, atol=1e-12)


def test_confidence_gain_halves():
    """App. A.3: one RMSNorm over [h_b; h_d] with a 2H gain, its first half on
    h_b and its second half on h_d.  With h_b = 1, h_d = 3 (H = 4), the joint
    rms is sqrt(5 + eps); gains 2 (first half) and 1/2 (second half); W2 = 1:
      W1 = [I 0]:  c = sigma(4 SiLU(2 / rms))
      W1 = [0 I]:  c = sigma(4 SiLU(1.5 / rms)).
    Dropping the second half of the gain, or reusing the first half for both,
    changes the second value."""
    s = small_shape(H=4, V=4, n_q=2, n_kv=1, d_h=2, F=4)
    w = zero_model(s)
    w["conf.norm"] = torch.tensor([2.0] * 4 + [0.5] * 4)
    w["conf.W2"] = torch.ones(1, 4)
    hb, hd = np.ones(4), np.full(4, 3.0)
    rms = math.sqrt(5.0 + 1e-6)
    sig = lambda x: 1.0 / (1.0 + math.exp(-x))
    for W1, inner in ((torch.cat([torch.eye(4), torch.zeros(4, 4)], 1), 2.0 / rms),
                      (torch.cat([torch.zeros(4, 4), torch.eye(4)], 1), 1.5 / rms)):
        w["conf.W1"] = W1
        expect = sig(4 * inner * sig(inner))
        assert abs(O.confidence(O.Model(s, w), hb, hd) - expect) < 1e-14


def _block_pos0(x, wts, pre, l, nq, nkv, d, eps=1e-6):
    """One pre-norm decoder block at the first position of a sequence: the
    only cached entry is the position's own, so attention returns its value
    vector v (softmax over one score is 1; RoPE does not touch v)."""
    W = lambda k: wts[f"{pre}.{k}"][l].double().numpy()
    y = W("attn_norm") * _r(x, eps)
    v = W("Wv") @ y
    grp = nq // nkv
    a = np.concatenate([v[(h // grp) * d:(h // grp + 1) * d] for h in range(nq)])
    x = x + W("Wo") @ a
    y = W("ffn_norm") * _r(x, eps)
    return x + W("Wdown") @ (_silu(W("Wgate") @ y) * (W("Wup") @ y))


@pytest.mark.parametrize("comp", ["linear", "mlp"])
def test_every_gain_at_the_first_position(comp):
    """The whole step at position 0 evaluated from the definitions (Eq. 1-6,
    App. A.1-A.3) with random weights and a distinct gain per norm and per
    layer: compressor, two backbone blocks (attention returns v at a single
    entry), final-norm LM head, MTP input and block, post-norm LM head and the
    joint-norm confidence.  A gain taken from another norm or another layer
    changes h_b, h_d, the logits or c."""
    s = small_shape(L=2, H=8, V=8, F=6, mtp_block=1, compressor=comp)
    rng = np.random.default_rng(21)
    w = {}
    for name, shape in synth.tensor_shapes(s).items():
        w[name] = torch.from_numpy(rng.standard_normal(shape).astype(np.float32) * 0.5)
    w = _distinct_gains(w, rng)
    W = lambda k: w[k].double().numpy()
    t0, t1 = 3, 6
    ab = np.concatenate([W("E")[t0], W("E")[t1]])
    if comp == "linear":
        x = W("comp.W") @ ab + W("comp.b")
    else:
        x = W("comp.W2") @ _silu(W("comp.W1") @ ab)
    for l in range(s.L):
        x = _block_pos0(x, w, "blk", l, s.n_q, s.n_kv, s.d_h)
    hb = x
    lb = W("E") @ (W("final_norm") * _r(hb))
    xb = int(np.argmax(lb))
    u = W("mtp.W_fc") @ np.concatenate([W("mtp.norm_h") * _r(hb), W("mtp.norm_e") * _r(W("E")[xb])])
    hd = _block_pos0(u, w, "mtp", 0, s.n_q, s.n_kv, s.d_h)
    ld = W("E") @ (W("mtp.norm_post") * _r(hd))
    t = W("conf.W1") @ (W("conf.norm") * _r(np.concatenate([hb, hd])))
    c = 1.0 / (1.0 + math.exp(-float(W("conf.W2")[0] @ _silu(t))))
    o = O.State(O.Model(s, w), 1).prefill([[t0, t1]], tau=0.5)
    assert np.allclose(o["h_b"][0], hb, rtol=0, atol=1e-12)
    assert np.allclose(o["logits_b"][0], lb, rtol=0, atol=1e-12)
    assert o["x_b"][0] == xb and np.sort(lb)[-1] - np.sort(lb)[-2] > 1e-6
    assert np.allclose(o["h_d"][0], hd, rtol=0, atol=1e-12)
    assert np.allclose(o["logits_d"][0], ld, rtol=0, atol=1e-12)
    assert abs(o["conf"][0] - c) < 1e-13


def test_seeded_gains_are_distinct_per_norm():
    """The generator gives every norm (and every layer of a stacked norm) its
    own gains, none of them unit, so the GPU parity runs can see a gain
    applied to the wrong norm."""
    s = TINY_SMALL.with_(L=3)
    w = synth.gen_weights(s, seed=0)
    gains = {k: v.double().numpy() for k, v in w.items() if synth.is_gain(k)}
    rows = []
    for k, v in gains.items():
        rows += [v[i] for i in range(v.shape[0])] if v.ndim == 2 else [v[: s.H], v[s.H:]] if k == "conf.norm" else [v]
    assert len(rows) == 2 * 3 + 1 + 2 + 2 + 1 + 2
    for i in range(len(rows)):
        assert np.all(np.abs(rows[i] - 1.0) < 0.35) and np.std(rows[i]) > 0.05
        for j in range(i):
            assert np.abs(rows[i] - rows[j]).max() > 0.05
    assert np.all(synth.gen_weights(s, seed=0, gain_std=0.0)["final_norm"].numpy() == 1.0)


# ------------------------------------------------------ seeded small models

def seeded(s, seed=0):
    w = synth.gen_weights(s, seed=seed)
    return w


TINY_SMALL = synth.TINY.with_(name="t", H=32, L=2, n_q=4, n_kv=2, d_h=8, F=48, V=64)


@pytest.mark.parametrize("comp,mtp,kvb", [("linear", 1, 0), ("mlp", 1, 1), ("mlp", 0, 0), ("linear", 0, 1)])
def test_cached_steps_equal_bruteforce_recompute(comp, mtp, kvb):
    s = TINY_SMALL.with_(compressor=comp, mtp_block=mtp)
    w = seeded(s, 3)
    w["x_pad"] = w["x_pad"] * 30  # make PAD inputs matter
    m = O.Model(s, w, max_ctx=32, kv_bf16=bool(kvb))
    st = O.State(m, 1)
    prompt = synth.gen_prompts(1, 9, s.V, seed=4).numpy()  # odd: last pair has PAD
    o = st.prefill(prompt, tau=0.5)
    pairs = [[int(prompt[0, 2 * j]), int(prompt[0, 2 * j + 1]) if 2 * j + 1 < 9 else -1] for j in range(5)]
    mtok = [int(prompt[0, 2 * j + 2]) for j in range(4)]
    force = 0
    for it in range(6):
        bf = O.bruteforce(m, pairs, mtok, tau=0.5, force=force)
        for k in ("logits_b", "logits_d", "h_b", "h_d", "conf"):
            assert np.allclose(o[k][0], bf[k][0], rtol=0, atol=1e-11), (it, k)
        assert list(o["tokens"][0]) == list(bf["tokens"][0])
        # extend the history with what this position produced
        mtok.append(int(o["x_b"][0]))
        pairs.append([int(o["tokens"][0, 0]), int(o["tokens"][0, 1])])
        force = [0, 2, 1][it % 3]
        o = st.step(tau=0.5, force=force)


def test_prompt_pairs_halve_the_length():
    s = TINY_SMALL
    m = O.Model(s, seeded(s), max_ctx=64)
    for n_tok, n_lat in ((2, 1), (10, 5), (11, 6), (1, 1)):
        st = O.State(m, 1)
        st.prefill(synth.gen_prompts(1, n_tok, s.V).numpy())
        assert st.seq(0)["n"] == n_lat


def test_reject_all_gives_one_token_per_pair_and_accept_all_two():
    s = TINY_SMALL
    m = O.Model(s, seeded(s), max_ctx=64)
    st = O.State(m, 2)
    st.prefill(synth.gen_prompts(2, 12, s.V).numpy(), force=2)
    for _ in range(5):
        o = st.step(force=2)
        assert np.all(o["n_acc"] == 0) and np.all(o["tokens"][:, 1] == -1)
        assert all(st.seq(b)["p1"] == -1 for b in range(2))
    assert [st.seq(b)["emitted"] for b in range(2)] == [1 + 5, 1 + 5]
    st2 = O.State(m, 2)
    st2.prefill(synth.gen_prompts(2, 12, s.V).numpy(), force=1)
    for _ in range(5):
        o = st2.step(force=1)
        assert np.all(o["n_acc"] == 1) and np.all(o["tokens"][:, 1] == o["x_d"])
    assert [st2.seq(b)["emitted"] for b in range(2)] == [2 + 10, 2 + 10]
    # tau = 0 accepts every draft (c > 0), the same trajectory as forced accept
    st3 = O.State(m, 2)
    st3.prefill(synth.gen_prompts(2, 12, s.V).numpy(), tau=0.0)
    st4 = O.State(m, 2)
    st4.prefill(synth.gen_prompts(2, 12, s.V).numpy(), force=1)
    for _ in range(3):
        a, b = st3.step(tau=0.0), st4.step(force=1)
        assert np.array_equal(a["tokens"], b["tokens"])


def test_rollback_equals_never_appending():
    s = TINY_SMALL
    m = O.Model(s, seeded(s), max_ctx=40)
    st = O.State(m, 2)
    st.prefill(synth.gen_prompts(2, 14, s.V).numpy())
    snap = [st.seq(b) for b in range(2)]
    caches = [[st.cache(b, l, 40) for l in range(s.L + 1)] for b in range(2)]
    ref = O.State(m, 2)
    ref.prefill(synth.gen_prompts(2, 14, s.V).numpy())
    for _ in range(4):
        st.step()
    st.rollback([snap[0]["n"], snap[1]["n"]])
    st.set_pending([[snap[b]["p0"], snap[b]["p1"]] for b in range(2)])
    for b in range(2):
        assert st.seq(b)["n"] == snap[b]["n"]
        for l in range(s.L + 1):
            K, V = st.cache(b, l, 40)
            assert np.array_equal(K, caches[b][l][0]) and np.array_equal(V, caches[b][l][1])
    a, r = st.step(), ref.step()
    assert np.array_equal(a["tokens"], r["tokens"]) and np.array_equal(a["logits_b"], r["logits_b"])


def test_batch_equals_independent_sequences():
    s = TINY_SMALL
    m = O.Model(s, seeded(s), max_ctx=40)
    prompts = synth.gen_prompts(3, 10, s.V, seed=9).numpy()
    st = O.State(m, 3)
    ob = [st.prefill(prompts)] + [st.step() for _ in range(3)]
    for b in range(3):
        one = O.State(m, 1)
        o1 = [one.prefill(prompts[b:b + 1])] + [one.step() for _ in range(3)]
        for x, y in zip(ob, o1):
            assert np.array_equal(x["tokens"][b], y["tokens"][0])
            assert np.array_equal(x["logits_d"][b], y["logits_d"][0])


@pytest.mark.parametrize("odd", [False, True])
def test_reprefill_of_history_reproduces_state(odd):
    """prefill(prompt) then k steps equals prefill(prompt + the consumed pairs):
    same caches in every layer, same next outputs (pair-level interface of
    Sec. 3.1).  With odd=True the last consumed pair carries PAD in its second
    slot, which a prompt of odd length expresses (PAD at the odd slot, App. B.2)."""
    s = TINY_SMALL
    m = O.Model(s, seeded(s, 5), max_ctx=40)
    prompt = synth.gen_prompts(1, 8, s.V, seed=2).numpy()
    st = O.State(m, 1)
    st.prefill(prompt, force=1)
    consumed = []
    forces = [1, 1, 2, 0] if odd else [1, 1, 1, 1]
    for f in forces:
        consumed.append((st.seq(0)["p0"], st.seq(0)["p1"]))
        o = st.step(force=f)
    n_now = st.seq(0)["n"]
    toks = list(prompt[0])
    for i, (a, b) in enumerate(consumed):
        toks.append(a)
        if b >= 0:
            toks.append(b)
        else:
            assert odd and i == len(consumed) - 1
    st2 = O.State(m, 1)
    o2 = st2.prefill(np.array([toks], np.int32), force=forces[-1])
    assert st2.seq(0)["n"] == n_now
    assert (st2.seq(0)["p0"], st2.seq(0)["p1"]) == (st.seq(0)["p0"], st.seq(0)["p1"])
    assert np.array_equal(o["tokens"], o2["tokens"]) and np.array_equal(o["logits_d"], o2["logits_d"])
    for l in range(s.L + 1):
        K1, V1 = st.cache(0, l, n_now)
        K2, V2 = st2.cache(0, l, n_now)
        assert np.array_equal(K1, K2) and np.array_equal(V1, V2)
    a, b = st.step(), st2.step()
    assert np.array_equal(a["logits_b"], b["logits_b"]) and np.array_equal(a["tokens"], b["tokens"])


def test_capacity_and_bad_ids_are_errors():
    s = TINY_SMALL
    m = O.Model(s, seeded(s), max_ctx=4)
    st = O.State(m, 1)
    with pytest.raises(ValueError):
        st.prefill([[s.V, 1]])
    st.prefill(synth.gen_prompts(1, 8, s.V).numpy())
    with pytest.raises(ValueError):
        st.step()


def test_bf16_cache_rounding_cascade():
    """Rounding the cache to bf16 (the storage of the bf16 configurations)
    turns a small difference into an ulp-level one over depth.  A relative
    1.2e-4 change of E flips a few cached bf16 values in layer 0.  Each flip
    moves the next layer's inputs enough to flip more, until a large share
    of every layer's cached values differ, and h_b differs by ~1e-3 relative.
    Without cache rounding the same change stays near its own size.  An fp32
    GPU path and the fp64 oracle round the cache independently, so at full
    depth their agreement is bounded by this cascade, whatever the kernels'
    precision."""
    s = synth.ModelShape("cascade", H=256, L=36, n_q=4, n_kv=2, d_h=64, F=768, V=512, compressor="mlp",
                         mtp_block=1, dtype="f32", rope_theta=1e6)
    w = {k: v.to(torch.bfloat16).float() for k, v in synth.gen_weights(s.with_(dtype="bf16"), seed=0).items()}
    wp = dict(w)
    E = w["E"].clone()
    E.view(torch.int32).add_(2048)  # +2048 fp32 ulps: about 1.2e-4 relative
    wp["E"] = E
    prompts = synth.gen_prompts(4, 4, s.V, seed=7).numpy()
    kd = 2 * s.n_kv * s.d_h  # cached values per layer and position (K and V)

    def run(weights, kvb):
        st = O.State(O.Model(s, weights, max_ctx=4, kv_bf16=kvb), 4)
        o = st.prefill(prompts, tau=0.5)
        return o, [[st.cache(b, l, 2) for l in range(s.L + 1)] for b in range(4)]

    (oa, ca), (ob, cb) = run(w, True), run(wp, True)
    (na, _), (nb, _) = run(w, False), run(wp, False)
    for b in range(4):
        flips = [int((ca[b][l][0] != cb[b][l][0]).sum() + (ca[b][l][1] != cb[b][l][1]).sum()) for l in range(s.L)]
        assert 0 < flips[0] < 0.1 * 2 * kd            # a few flips in the first layer
        assert min(flips[-6:]) > 0.3 * 2 * kd         # a large share of the last layers
        rel = np.abs(oa["h_b"][b] - ob["h_b"][b]).max() / np.abs(oa["h_b"][b]).max()
        rel_exact = np.abs(na["h_b"][b] - nb["h_b"][b]).max() / np.abs(na["h_b"][b]).max()
        assert rel > 5e-4 and rel > 10 * rel_exact, (rel, rel_exact)
