"""Pins of oracle.philox: published known answers and distributional checks."""
import math

import numpy as np
import pytest
from scipy import stats

from conftest import read_golden
from oracle import philox


def test_philox_known_answers():
    rows = read_golden("philox4x32_10_kat.txt")
    assert len(rows) == 3
    for row in rows:
        w = [int(t, 16) for t in row.split()]
        assert philox.philox4x32_10(w[0:4], w[4:6]) == tuple(w[6:10])


def test_res53_endpoints_and_exactness():
    assert philox.res53(0, 0) == 0.0
    top = philox.res53(0xFFFFFFFF, 0xFFFFFFFF)
    assert top == 1.0 - 2.0 ** -53 and top < 1.0
    # 2^26 * (w0>>5) + (w1>>6) is the 53-bit integer numerator
    assert philox.res53(1 << 31, 0) == 0.5
    assert philox.res53(0, 1 << 6) == 2.0 ** -53


def test_integer_uniform_is_the_res53_numerator():
    for w0, w1 in ((0, 0), (0xFFFFFFFF, 0xFFFFFFFF), (0x12345678, 0x9ABCDEF0), (1 << 31, 1 << 6)):
        assert philox.int53(w0, w1) / 2.0 ** 53 == philox.res53(w0, w1)
        assert 0 <= philox.int53(w0, w1) < 2 ** 53
    assert philox.uniform_int(1, 2, 3, 4, 5, 0) / 2.0 ** 53 == philox.uniform(1, 2, 3, 4, 5, 0)


def test_counter_layout_separates_decisions():
    seen = set()
    for rnd in range(3):
        for pos in range(16):
            for purpose in range(4):
                seen.add(philox.counter(5, 9, rnd, pos, purpose))
    assert len(seen) == 3 * 16 * 4
    assert philox.counter(1, 2, 3, 4, 5) == (1, 2, (3 << 8) | 4, 5)
    assert philox.key_of((7 << 32) | 11) == (11, 7)


def test_uniform_is_uniform():
    u = np.array([philox.uniform(1, 0, f, 0, 1, 0) for f in range(20000)])
    assert abs(u.mean() - 0.5) < 0.01
    assert abs(u.var() - 1.0 / 12.0) < 0.005
    assert stats.kstest(u, "uniform").pvalue > 1e-4


def test_normal_pairs_are_standard_normal():
    z = np.array([v for f in range(5000) for v in philox.normal_pair(3, 1, f, 2, 5, 0)])
    assert abs(z.mean()) < 0.05
    assert abs(z.std() - 1.0) < 0.05
    assert stats.kstest(z, "norm").pvalue > 1e-4
    # the pair is (r cos t, r sin t): r^2 = -2 ln(1 - u1) is Exp(1/2)
    a, b = philox.normal_pair(3, 1, 0, 2, 5, 0)
    w = philox.philox4x32_10(philox.counter(1, 0, 2, 5, philox.PURPOSE_NOISE), philox.key_of(3))
    u1 = philox.res53(w[0], w[1])
    assert math.isclose(a * a + b * b, -2.0 * math.log(1.0 - u1), rel_tol=1e-12)
