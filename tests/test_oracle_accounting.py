"""Pins of oracle.accounting against numbers the paper prints (tests/golden/paper_numbers.txt)."""
import math

import pytest

from conftest import read_golden
from oracle import accounting as A


def _golden():
    out = {}
    for row in read_golden("paper_numbers.txt"):
        name, value, tol, *_ = row.split()
        out[name] = (float(value), float(tol))
    return out


G = _golden()


def _check(name, got):
    v, tol = G[name]
    assert abs(got - v) <= tol + 1e-9 * abs(v), (name, got, v)


def test_real_time_rates():
    _check("tokens_per_second", A.tokens_per_second())
    _check("inner_calls_per_second", A.inner_calls_per_second_ar())
    _check("sequential_calls_per_second_at_2.47", A.sequential_calls_per_second(2.47))
    _check("inner_calls_at_2.47", A.inner_calls_per_second_ar() / 2.47)


def test_parameter_counts():
    _check("offset_parameters", A.offset_parameters(3, 1024))
    _check("offset_percent_of_0.6B", 100.0 * A.offset_parameters(3, 1024) / 0.6e9)
    _check("medusa_parameters_millions", A.medusa_head_parameters(45, 1024, 2048) / 1e6)


def test_inner_loop_cost_per_audio_second():
    _check("ar_inner_ms_iphone12", A.inner_ms_per_audio_second(4.77))
    _check("ar_inner_ms_iphone17", A.inner_ms_per_audio_second(2.05))
    _check("spec_inner_ms_iphone17", A.inner_ms_per_audio_second(2.05) / 2.34)
