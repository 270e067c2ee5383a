"""Pins of the oracle's sampling primitive (the paper's evaluation sampler:
temperature, top-k, top-p, repetition penalty, one draw u in [0, 1)) against
closed forms on small vocabularies.  CPU only."""
import math

import numpy as np
import pytest

from oracle import oracle as O

LOG1234 = np.log([1.0, 2.0, 3.0, 4.0])  # softmax: 0.1, 0.2, 0.3, 0.4


def plain(logits, u, **kw):
    args = dict(temperature=1.0, top_k=0, top_p=1.0, rep_penalty=1.0)
    args.update(kw)
    return O.sample(logits, u, **args)


def test_full_distribution_inverse_cdf_in_descending_order():
    # order 3 (0.4), 2 (0.3), 1 (0.2), 0 (0.1); cumulative 0.4, 0.7, 0.9, 1.0
    for u, want in ((0.0, 3), (0.39, 3), (0.41, 2), (0.69, 2), (0.71, 1), (0.89, 1), (0.91, 0), (0.999, 0)):
        assert plain(LOG1234, u) == want, u


def test_top_k_renormalises_the_k_largest():
    # keep 3 and 2: 4/7, 3/7
    assert plain(LOG1234, 0.57, top_k=2) == 3      # 0.57 < 4/7 = 0.5714
    assert plain(LOG1234, 0.58, top_k=2) == 2
    assert plain(LOG1234, 0.999, top_k=2) == 2     # never 1 or 0


def test_top_p_keeps_the_shortest_prefix_reaching_p():
    # cumulative 0.4, 0.7, 0.9: p = 0.65 keeps {3, 2} (4/7, 3/7), p = 0.75 keeps {3, 2, 1}
    assert plain(LOG1234, 0.58, top_p=0.65) == 2
    assert plain(LOG1234, 0.999, top_p=0.65) == 2
    # {3, 2, 1}: 4/9, 3/9, 2/9 -> u = 0.8 lands in id 1 (cumulative 7/9 = 0.778)
    assert plain(LOG1234, 0.8, top_p=0.75) == 1
    assert plain(LOG1234, 0.999, top_p=0.75) == 1
    # a p below the largest probability keeps only the argmax
    assert plain(LOG1234, 0.999, top_p=0.3) == 3


def test_temperature_scales_logits():
    # T = 2 on log [1, 4]: probs proportional to [1, 2] -> 1/3, 2/3
    lg = np.log([1.0, 4.0])
    assert plain(lg, 0.66, temperature=2.0) == 1
    assert plain(lg, 0.67, temperature=2.0) == 0
    # a small temperature is greedy
    assert plain(LOG1234, 0.999, temperature=1e-3) == 3
    # temperature acts before the nucleus cut: at T = 0.5 the probs are
    # proportional to 1, 4, 9, 16 (/30): p = 0.5 keeps {3} (16/30 >= 0.5)
    assert plain(LOG1234, 0.999, temperature=0.5, top_p=0.5) == 3
    assert plain(LOG1234, 0.999, temperature=1.0, top_p=0.5) == 2


def test_greedy_is_top_k_one_with_lower_id_on_ties():
    assert O.sample([0.5, 2.0, 2.0, 1.0], 0.999, top_k=1, top_p=0.95, rep_penalty=1.0) == 1
    rng = np.random.default_rng(0)
    for _ in range(20):
        lg = rng.standard_normal(50)
        assert O.sample(lg, rng.random(), top_k=1, rep_penalty=1.0) == int(np.argmax(lg))


def test_repetition_penalty_divides_positive_and_multiplies_negative_logits_once():
    # positive: 1.0 -> 1/1.5 = 0.667 < 0.8 flips the argmax to id 1
    assert O.sample([1.0, 0.8], 0.0, hist=[0], top_k=1, rep_penalty=1.5) == 1
    assert O.sample([1.0, 0.8], 0.0, hist=[], top_k=1, rep_penalty=1.5) == 0
    # negative: -0.5 -> -0.75 < -0.6 flips the argmax to id 1
    assert O.sample([-0.5, -0.6], 0.0, hist=[0], top_k=1, rep_penalty=1.5) == 1
    # an id that repeats in the history is penalised once: 1.0 -> 0.667 > 0.5
    assert O.sample([1.0, 0.5], 0.0, hist=[0, 0, 0], top_k=1, rep_penalty=1.5) == 0
    # the penalised distribution: [2/1.5, ln 1] = [4/3, 0] -> p(0) = e^(4/3) / (e^(4/3) + 1)
    p0 = math.exp(4 / 3) / (math.exp(4 / 3) + 1)
    assert O.sample([2.0, 0.0], p0 - 1e-9, hist=[0], top_k=0, top_p=1.0, rep_penalty=1.5) == 0
    assert O.sample([2.0, 0.0], p0 + 1e-9, hist=[0], top_k=0, top_p=1.0, rep_penalty=1.5) == 1


def test_paper_settings_stay_in_the_top_twenty():
    rng = np.random.default_rng(1)
    lg = rng.standard_normal(500) * 3
    top20 = set(np.argsort(-lg)[:20].tolist())
    for i in range(200):
        t = O.sample(lg, rng.random())  # T = 1, k = 20, p = 0.95, penalty 1.5
        assert t in top20


# ---- the decision margin -------------------------------------------------

def test_decision_margin_closed_forms():
    # order 3 (0.4), 2 (0.3), 1 (0.2), 0 (0.1); u = 0.5 lands in id 2's interval [0.4, 0.7)
    t, m = O.sample_ex(LOG1234, 0.5, top_k=0, top_p=1.0, rep_penalty=1.0)
    assert t == 2 and m == pytest.approx(0.1)  # u is 0.1 from 0.4 and 0.2 from 0.7; logit gaps log(4/3), log(3/2)
    t, m = O.sample_ex(LOG1234, 0.41, top_k=0, top_p=1.0, rep_penalty=1.0)
    assert t == 2 and m == pytest.approx(0.01)
    # the first id: only its upper end counts (0.4 - 0.05 = 0.35), against the gap log(4/3) = 0.288
    t, m = O.sample_ex(LOG1234, 0.05, top_k=0, top_p=1.0, rep_penalty=1.0)
    assert t == 3 and m == pytest.approx(np.log(4 / 3))
    t, m = O.sample_ex(LOG1234, 0.2, top_k=0, top_p=1.0, rep_penalty=1.0, temperature=1e-1)
    assert t == 3  # T = 0.1 sharpens: p(3) = 4^10 / (1 + 2^10 + 3^10 + 4^10) = 0.947
    assert m == pytest.approx(min(10 * np.log(4 / 3), 4.0 ** 10 / (1 + 2.0 ** 10 + 3.0 ** 10 + 4.0 ** 10) - 0.2))
    # k = 1: the top-1 / top-2 logit gap whatever u is
    for u in (0.0, 0.5, 0.999):
        t, m = O.sample_ex(LOG1234, u, top_k=1, top_p=1.0, rep_penalty=1.0)
        assert t == 3 and m == pytest.approx(np.log(4 / 3))
    # top-p = 0.65 keeps {3, 2} (cumulative 0.7): the cut is 0.05 above p and 0.25 below the first id's 0.4
    t, m = O.sample_ex(LOG1234, 0.99, top_k=0, top_p=0.65, rep_penalty=1.0)
    assert t == 2 and m == pytest.approx(0.05)
    # top-k = 2 with the nucleus taking both: the boundary gap log(3/2) between the 2nd and 3rd
    t, m = O.sample_ex(LOG1234, 0.99, top_k=2, top_p=1.0, rep_penalty=1.0)
    assert t == 2 and m == pytest.approx(min(np.log(4 / 3), np.log(3 / 2), 0.99 - 4 / 7))


# ---- the sampler in both heads of the pair step --------------------------

from paper_2605_27255_gb300 import synth  # noqa: E402


def _tiny_states(B=2, seed=0):
    s = synth.TINY
    w = synth.gen_weights(s, seed=seed, device="cpu")
    return s, w


def test_top1_sampling_is_the_greedy_step():
    s, w = _tiny_states()
    prompts = synth.gen_prompts(2, 21, s.V, seed=3).numpy()
    rng = np.random.default_rng(5)
    greedy = O.State(O.Model(s, w, max_ctx=32), 2)
    samp = O.State(O.Model(s, w, max_ctx=32), 2)
    samp.set_sampler(temperature=1.0, top_k=1, top_p=0.95, rep_penalty=1.0)
    outs = [(greedy.prefill(prompts), samp.prefill(prompts, u=rng.random((2, 2))))]
    for _ in range(5):
        outs.append((greedy.step(), samp.step(u=rng.random((2, 2)))))
    for a, b in outs:
        for key in ("tokens", "n_acc", "logits_b", "logits_d", "conf", "x_b", "x_d"):
            assert np.array_equal(a[key], b[key]), key


def test_sampled_heads_follow_the_primitive_and_the_history():
    """x_b is drawn from the backbone head's logits with the tokens so far as
    the repetition history, x_d from the draft head's with that history and
    x_b; the history then keeps x_b and, when accepted, x_d."""
    s, w = _tiny_states(seed=1)
    B = 2
    prompts = synth.gen_prompts(B, 19, s.V, seed=4).numpy()
    rng = np.random.default_rng(6)
    st = O.State(O.Model(s, w, max_ctx=32), B)
    cfg = dict(temperature=0.8, top_k=20, top_p=0.9, rep_penalty=1.5)
    st.set_sampler(**cfg)
    hist = [list(prompts[b]) for b in range(B)]
    u = rng.random((B, 2))
    o = st.prefill(prompts, u=u, tau=0.5)
    for step in range(7):
        for b in range(B):
            xb = O.sample(o["logits_b"][b], u[b, 0], hist=hist[b], **cfg)
            assert o["x_b"][b] == xb == o["tokens"][b, 0]
            xd = O.sample(o["logits_d"][b], u[b, 1], hist=hist[b] + [xb], **cfg)
            assert o["x_d"][b] == xd
            hist[b] += [xb] + ([xd] if o["n_acc"][b] else [])
            assert o["tokens"][b, 1] == (xd if o["n_acc"][b] else -1)
            assert list(st.history(b)) == hist[b]
            assert (st.seq(b)["p0"], st.seq(b)["p1"]) == (xb, xd if o["n_acc"][b] else -1)
        u = rng.random((B, 2))
        o = st.step(u=u, tau=0.5)


def test_large_penalty_top1_never_repeats_a_token_with_positive_logits():
    s, w = _tiny_states(seed=2)
    prompts = synth.gen_prompts(1, 9, s.V, seed=7).numpy()
    st = O.State(O.Model(s, w, max_ctx=40), 1)
    st.set_sampler(temperature=1.0, top_k=1, top_p=1.0, rep_penalty=1e6)
    o = st.prefill(prompts, u=np.zeros((1, 2)), force=1)
    for _ in range(12):
        before = list(st.history(0))
        o = st.step(u=np.zeros((1, 2)), force=1)
        xb, xd = int(o["x_b"][0]), int(o["x_d"][0])
        seen_b, seen_d = set(before), set(before) | {xb}
        if max(v for i, v in enumerate(o["logits_b"][0]) if i not in seen_b) > 0:
            assert xb not in seen_b
        if max(v for i, v in enumerate(o["logits_d"][0]) if i not in seen_d) > 0:
            assert xd not in seen_d


def test_sampler_needs_draws_and_valid_settings():
    s, w = _tiny_states()
    st = O.State(O.Model(s, w, max_ctx=16), 1)
    st.set_sampler()
    with pytest.raises(ValueError):
        st.prefill(synth.gen_prompts(1, 6, s.V, seed=1).numpy())  # no draws
    with pytest.raises(ValueError):
        st.set_sampler(top_p=0.0)
    st.set_sampler(temperature=0.0)  # greedy again: no draws needed
    st.prefill(synth.gen_prompts(1, 6, s.V, seed=1).numpy())


def test_regular_decoding_history_is_prompt_then_outputs():
    s, w = _tiny_states()
    prompts = synth.gen_prompts(1, 7, s.V, seed=2).numpy()
    st = O.State(O.Model(s, w, max_ctx=16), 1)
    toks = [int(st.regular_prefill(prompts)["tokens"][0, 0])]
    for _ in range(3):
        toks.append(int(st.regular_step()["tokens"][0, 0]))
    assert list(st.history(0)) == list(prompts[0]) + toks
