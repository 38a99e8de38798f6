"""Pins of oracle.sampler: the fp32 exponential, top-k order, integer-weight softmax, and
the acceptance rule's losslessness (Sec. 2.2 / Sec. 3.2: keep d with prob min(1, p/q),
else resample from norm(max(0, p - q)); the emitted code is then distributed exactly as p).
"""
import math
import struct
from fractions import Fraction

import numpy as np
import pytest
from scipy import stats

from oracle import philox
from oracle.enumeration import alpha
from oracle.sampler import (TAYLOR, Dist, accept, draw, exp32, greedy_dist, residual_draw,
                            residual_weights, topk_dist, topk_order)


def bits(f):
    return struct.unpack("<I", struct.pack("<f", float(np.float32(f))))[0]


# ---- exp32 (Cody-Waite range reduction + Taylor polynomial) ---------------------------
def test_exp32_constants_are_the_rounded_taylor_coefficients():
    # the CUDA implementation hard-codes these fp32 bit patterns
    assert [bits(c) for c in TAYLOR] == [0x39500D01, 0x3AB60B61, 0x3C088889, 0x3D2AAAAB,
                                          0x3E2AAAAB, 0x3F000000, 0x3F800000, 0x3F800000]


def test_exp32_matches_libm_within_a_few_ulp():
    xs = np.concatenate([-np.logspace(-8, math.log10(87), 4000), np.linspace(-87, 0, 4001)]).astype(np.float32)
    for x in xs:
        got = float(exp32(x))
        ref = math.exp(float(x))
        assert abs(got - ref) <= 4 * 2.0 ** -24 * ref, (x, got, ref)
    assert exp32(np.float32(0)) == np.float32(1)
    assert exp32(np.float32(-88)) == 0 and exp32(np.float32(-1000)) == 0


def test_exp32_special_values():
    # exact powers of two: d = -n ln2 reduces to r ~ 0
    assert abs(float(exp32(np.float32(-math.log(2)))) - 0.5) <= 2 ** -24
    assert abs(float(exp32(np.float32(-10 * math.log(2)))) - 2.0 ** -10) <= 2 ** -33


# ---- top-k order -----------------------------------------------------------------------
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


# ---- integer-weight softmax ------------------------------------------------------------
def test_weights_two_entry_closed_form():
    l = np.array([0.25, 1.5], dtype=np.float32)
    T = 0.9
    d = topk_dist(l, 2, T)
    Tf = float(np.float32(T))
    assert d.ids == [0, 1]                                   # listed in ascending id order
    assert d.weight(1) == 2 ** 24                            # the maximum has e = 1 exactly
    p1 = 1.0 / (1.0 + math.exp((0.25 - 1.5) / Tf))
    assert abs(d.prob(1) - p1) < 1e-6
    assert d.frac(0) + d.frac(1) == 1 and d.frac(7) == 0


def test_weights_follow_temperature_softmax():
    rng = np.random.default_rng(1)
    l = rng.standard_normal(64).astype(np.float32)
    d = topk_dist(l, 8, 0.5)
    ids = np.argsort(-l.astype(np.float64), kind="stable")[:8]
    w = np.exp((l[ids].astype(np.float64) - l[ids[0]]) / float(np.float32(0.5)))
    assert d.ids == sorted(int(i) for i in ids)
    assert np.allclose([d.prob(i) for i in ids], w / w.sum(), rtol=2e-6, atol=0)
    assert sum(d.frac(i) for i in range(64)) == 1


def test_weights_are_floor_of_scaled_exp32():
    l = np.array([3.0, 1.0, -2.0, 0.5], dtype=np.float32)
    d = topk_dist(l, 4, 1.3)
    T = np.float32(1.3)
    assert d.ids == [0, 1, 2, 3]
    z_max = l[0] / T
    assert d.W == [math.floor(float(exp32(l[i] / T - z_max)) * 2 ** 24) for i in d.ids]
    # ties at the boundary: the lower ids are kept, then listed ascending
    t = topk_dist(np.array([1.0, 2.0, 1.0, 1.0, 0.0], dtype=np.float32), 3, 1.0)
    assert t.ids == [0, 1, 2]


# ---- draws and acceptance ---------------------------------------------------------------
def test_draw_boundaries_are_exact():
    d = Dist(ids=[4, 2, 9], W=[5, 3, 2])                     # p = 1/2, 3/10, 1/5
    top = 2 ** 53
    assert draw(d, 0) == 4
    assert draw(d, top // 2 - 1) == 4 and draw(d, top // 2) == 2
    assert draw(d, (top * 8) // 10 - 1) == 2 and draw(d, -(-top * 8 // 10)) == 9
    assert draw(d, top - 1) == 9
    n = 20000
    c = {4: 0, 2: 0, 9: 0}
    for i in range(n):
        c[draw(d, philox.uniform_int(2, 0, i, 0, 1, 0))] += 1
    assert stats.chisquare([c[4], c[2], c[9]], [n * 0.5, n * 0.3, n * 0.2]).pvalue > 1e-4


def test_greedy_is_one_hot_on_argmax():
    l = np.array([0.0, 2.0, 2.0, 1.0], dtype=np.float32)
    g = greedy_dist(l)
    assert g.ids == [1] and g.frac(1) == 1 and g.frac(2) == 0


def test_accept_rule_special_cases():
    p = Dist(ids=[0, 1], W=[6, 4])
    q = Dist(ids=[0, 2], W=[5, 5])
    assert accept(p, q, 0, 2 ** 53 - 1)          # p(0) >= q(0): always kept
    assert not accept(p, q, 2, 0)                # p(2) = 0: never kept (strict)
    # keep probability exactly p/q: 0.4/0.5 = 4/5 of the uniform range
    p2 = Dist(ids=[0, 5], W=[4, 6])
    edge = -(-(2 ** 53 * 4) // 5)                # ceil(0.8 * 2^53): first rejected U
    assert accept(p2, q, 0, edge - 1) and not accept(p2, q, 0, edge)


def _emission_law(p: Dist, q: Dist):
    """Exact law of the code emitted for one draft: q(d) min(1,p/q) on accept + residual."""
    law = {}
    a = Fraction(0)
    for d in q.ids:
        keep = min(Fraction(1), p.frac(d) / q.frac(d))
        law[d] = law.get(d, Fraction(0)) + q.frac(d) * keep
        a += q.frac(d) * keep
    xs, r, R = residual_weights(p, q)
    for x, rx in zip(xs, r):
        law[x] = law.get(x, Fraction(0)) + (1 - a) * Fraction(rx, R)
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
            assert law.get(x, Fraction(0)) == p.frac(x)
        assert a == alpha(p, q)


def test_acceptance_rule_is_lossless_statistically():
    rng = np.random.default_rng(7)
    p, q = _random_pair(rng, 8, 6)
    n = 20000
    counts = np.zeros(8)
    kept = 0
    for i in range(n):
        d = draw(q, philox.uniform_int(4, 0, i, 0, 2, philox.PURPOSE_DRAFT))
        if accept(p, q, d, philox.uniform_int(4, 0, i, 0, 2, philox.PURPOSE_ACCEPT)):
            counts[d] += 1
            kept += 1
        else:
            counts[residual_draw(p, q, philox.uniform_int(4, 0, i, 0, 2, philox.PURPOSE_TARGET))] += 1
    exp = np.array([p.prob(x) for x in range(8)]) * n
    m = exp > 0
    assert counts[~m].sum() == 0
    assert stats.chisquare(counts[m], exp[m] * counts[m].sum() / exp[m].sum()).pvalue > 1e-4
    a = float(alpha(p, q))
    assert abs(kept / n - a) < 4 * math.sqrt(a * (1 - a) / n) + 1e-9


def test_residual_support_is_where_p_exceeds_q():
    p = Dist(ids=[0, 1, 2], W=[5, 3, 2])
    q = Dist(ids=[0, 3], W=[9, 1])
    xs, r, R = residual_weights(p, q)
    assert xs == [0, 1, 2]                       # p's sampling order
    # N_x = S_p S_q max(0, p - q): S_p = S_q = 10
    assert r == [0, 30, 20] and R == 50
    assert residual_draw(p, q, 0) == 1
    assert residual_draw(p, q, 2 ** 53 - 1) == 2
    assert residual_draw(p, p, 0) == 0           # p == q: R = 0 falls back to p
    # the walk follows p's sampling order, not id order
    p3 = Dist(ids=[7, 1], W=[2, 2])
    q3 = Dist(ids=[5], W=[1])
    assert residual_draw(p3, q3, 0) == 7
