"""Pins of oracle.sampler: top-k order, softmax closed forms, and the acceptance rule's
losslessness (Sec. 2.2 / Sec. 3.2: keep d with prob min(1, p/q), else resample from
norm(max(0, p - q)); the emitted code is then distributed exactly as p)."""
import math

import numpy as np
import pytest
from scipy import stats

from oracle import philox
from oracle.enumeration import alpha
from oracle.sampler import (Dist, accept, draw, greedy_dist, residual_draw,
                            residual_weights, topk_dist, topk_order)


def test_topk_ties_go_to_lower_id():
    l = np.array([1.0, 3.0, 3.0, 2.0, 3.0], dtype=np.float32)
    assert topk_order(l, 2) == [1, 2]
    assert topk_order(l, 4) == [1, 2, 4, 3]
    assert topk_order(l, 99) == [1, 2, 4, 3, 0]          # k >= V keeps all


def test_topk_signed_zero_is_a_tie():
    l = np.array([-0.0, 0.0, -1.0], dtype=np.float32)
    assert topk_order(l, 2) == [0, 1]


def test_topk_matches_lexsort_brute_force():
    rng = np.random.default_rng(0)
    for _ in range(50):
        V = int(rng.integers(1, 40))
        l = np.round(rng.standard_normal(V) * 2).astype(np.float32)   # many ties
        k = int(rng.integers(1, V + 3))
        ref = list(np.lexsort((np.arange(V), -l.astype(np.float64))))[:k]
        assert topk_order(l, k) == [int(i) for i in ref]


def test_softmax_two_entry_closed_form():
    l = np.array([0.25, 1.5], dtype=np.float32)
    T = 0.9
    d = topk_dist(l, 2, T)
    Tf = float(np.float32(T))
    p1 = 1.0 / (1.0 + math.exp((0.25 - 1.5) / Tf))
    assert d.ids == [1, 0]
    assert math.isclose(d.prob(1), p1, rel_tol=1e-15)
    assert math.isclose(d.prob(0), 1.0 - p1, rel_tol=1e-14)
    assert d.prob(7) == 0.0


def test_softmax_temperature_and_truncation():
    rng = np.random.default_rng(1)
    l = rng.standard_normal(64).astype(np.float32)
    d = topk_dist(l, 8, 0.5)
    ids = np.argsort(-l.astype(np.float64), kind="stable")[:8]
    w = np.exp((l[ids].astype(np.float64) - l[ids[0]]) / float(np.float32(0.5)))
    ref = w / w.sum()
    assert d.ids == list(ids)
    assert np.allclose([d.prob(i) for i in ids], ref, rtol=1e-13, atol=0)
    assert math.isclose(sum(d.prob(i) for i in range(64)), 1.0, rel_tol=1e-14)


def test_draw_endpoints_and_frequencies():
    d = Dist(ids=[4, 2, 9], e=[0.5, 0.3, 0.2], S=1.0)
    assert draw(d, 0.0) == 4
    assert draw(d, 0.4999999) == 4 and draw(d, 0.5) == 2
    assert draw(d, 1.0 - 2.0 ** -53) == 9
    n = 20000
    c = {4: 0, 2: 0, 9: 0}
    for i in range(n):
        c[draw(d, philox.uniform(2, 0, i, 0, 1, 0))] += 1
    chi = stats.chisquare([c[4], c[2], c[9]], [n * 0.5, n * 0.3, n * 0.2])
    assert chi.pvalue > 1e-4


def test_greedy_is_one_hot_on_argmax():
    l = np.array([0.0, 2.0, 2.0, 1.0], dtype=np.float32)
    g = greedy_dist(l)
    assert g.ids == [1] and g.prob(1) == 1.0 and g.prob(2) == 0.0


def test_accept_rule_special_cases():
    p = Dist(ids=[0, 1], e=[0.6, 0.4], S=1.0)
    q = Dist(ids=[0, 2], e=[0.5, 0.5], S=1.0)
    # p(0) >= q(0): always kept, even at the largest uniform
    assert accept(p, q, 0, 1.0 - 2.0 ** -53)
    # p(2) = 0: never kept, even at u = 0 (strict comparison)
    assert not accept(p, q, 2, 0.0)


def _emission_law(p: Dist, q: Dist):
    """Exact law of the code emitted for one draft: q(d) min(1,p/q) on accept + residual."""
    law = {}
    a = 0.0
    for d in q.ids:
        keep = min(1.0, p.prob(d) / q.prob(d))
        law[d] = law.get(d, 0.0) + q.prob(d) * keep
        a += q.prob(d) * keep
    xs, r, R = residual_weights(p, q)
    for x, rx in zip(xs, r):
        law[x] = law.get(x, 0.0) + (1.0 - a) * rx / R
    return law, a


def _random_pair(rng, V, k):
    lp = rng.standard_normal(V).astype(np.float32)
    lq = (lp + rng.standard_normal(V)).astype(np.float32)
    return topk_dist(lp, k, 0.9), topk_dist(lq, k, 0.9)


@pytest.mark.parametrize("V,k", [(4, 4), (6, 6), (8, 5), (16, 6)])
def test_acceptance_rule_is_lossless_exactly(V, k):
    rng = np.random.default_rng(V * 31 + k)
    for _ in range(20):
        p, q = _random_pair(rng, V, k)
        law, a = _emission_law(p, q)
        for x in range(V):
            assert abs(law.get(x, 0.0) - p.prob(x)) < 1e-15
        assert math.isclose(a, alpha(p, q), rel_tol=1e-13, abs_tol=1e-15)


def test_acceptance_rule_is_lossless_statistically():
    rng = np.random.default_rng(7)
    p, q = _random_pair(rng, 8, 6)
    n = 20000
    counts = np.zeros(8)
    kept = 0
    for i in range(n):
        d = draw(q, philox.uniform(4, 0, i, 0, 2, philox.PURPOSE_DRAFT))
        if accept(p, q, d, philox.uniform(4, 0, i, 0, 2, philox.PURPOSE_ACCEPT)):
            counts[d] += 1
            kept += 1
        else:
            counts[residual_draw(p, q, philox.uniform(4, 0, i, 0, 2, philox.PURPOSE_TARGET))] += 1
    exp = np.array([p.prob(x) for x in range(8)]) * n
    m = exp > 0
    assert counts[~m].sum() == 0
    assert stats.chisquare(counts[m], exp[m]).pvalue > 1e-4
    a = alpha(p, q)
    assert abs(kept / n - a) < 4 * math.sqrt(a * (1 - a) / n) + 1e-9


def test_residual_support_is_where_p_exceeds_q():
    p = Dist(ids=[0, 1, 2], e=[0.5, 0.3, 0.2], S=1.0)
    q = Dist(ids=[0, 3], e=[0.9, 0.1], S=1.0)
    xs, r, R = residual_weights(p, q)
    assert xs == [0, 1, 2]
    assert r[0] == 0.0 and r[1] == 0.3 and r[2] == 0.2
    assert residual_draw(p, q, 0.0) == 1
    assert residual_draw(p, q, 0.99) == 2
    # p == q: R = 0 falls back to p (the accept test keeps every draft then)
    assert residual_draw(p, p, 0.0) == 0
