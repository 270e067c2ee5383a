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
