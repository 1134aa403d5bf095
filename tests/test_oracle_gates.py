"""Pins of oracle/gates.py against values the mathematics fixes (not a retyped formula).

* sigmoid: sigma(0) = 1/2; sigma(x) + sigma(-x) = 1; sigma(+-ln n) = n/(n+1), 1/(n+1) (exact
  rationals, since e^-x = 1/n there); against 1/(1 + e^-x) at a handful of points; limits.
* softplus: softplus(0) = ln 2; softplus(x) - softplus(-x) = x; softplus(x) -> x and -> 0;
  d softplus / dx = sigma(x) (central difference).
* forget_gate: alpha(0, A) = 2^-A (since softplus(0) = ln 2); alpha -> 1 as the logit -> -inf
  and -> 0 as it -> +inf for A > 0; alpha in (0, 1]; alpha(f, A1 + A2) = alpha(f, A1) alpha(f, A2).
* write_strength in (0, 1) and equal to sigma.
* cumulative_clock: a constant increment gives lambda_t = lambda0 + t delta; order preserving
  (Prop. 5: positive increments give a strictly increasing clock).
"""
import math
from fractions import Fraction

import numpy as np
import pytest

from oracle import gates as OG


def test_sigmoid_fixed_points_and_symmetry():
    assert OG.sigmoid(0.0) == 0.5
    x = np.linspace(-30, 30, 601)
    np.testing.assert_allclose(OG.sigmoid(x) + OG.sigmoid(-x), 1.0, rtol=0, atol=1e-15)
    assert np.all(np.diff(OG.sigmoid(x)) >= 0)
    assert OG.sigmoid(-800.0) >= 0.0 and OG.sigmoid(-800.0) < 1e-300
    assert OG.sigmoid(800.0) == 1.0


@pytest.mark.parametrize('n', [1, 2, 3, 5, 10])
def test_sigmoid_at_log_points(n):
    # at x = ln n: e^-x = 1/n exactly, so sigma = n / (n + 1); at x = -ln n: 1 / (n + 1)
    want = Fraction(n, n + 1)
    assert abs(float(OG.sigmoid(math.log(n))) - float(want)) < 1e-15
    assert abs(float(OG.sigmoid(-math.log(n))) - float(1 - want)) < 1e-15


def test_sigmoid_against_logistic_definition():
    x = np.array([-7.25, -2.0, -0.5, 0.125, 1.0, 3.5, 9.0])
    want = np.array([1.0 / (1.0 + math.exp(-v)) for v in x])
    np.testing.assert_allclose(OG.sigmoid(x), want, rtol=1e-14, atol=0)


def test_softplus_fixed_points_and_identity():
    assert abs(float(OG.softplus(0.0)) - math.log(2.0)) < 1e-16
    x = np.linspace(-40, 40, 801)
    np.testing.assert_allclose(OG.softplus(x) - OG.softplus(-x), x, rtol=0, atol=1e-12)
    assert np.all(OG.softplus(x) > 0)
    np.testing.assert_allclose(OG.softplus(np.array([50.0, 100.0])), [50.0, 100.0], rtol=1e-15)
    assert OG.softplus(-50.0) < 2e-22
    # softplus(ln n) = ln(1 + n)
    for n in (1, 3, 7):
        assert abs(float(OG.softplus(math.log(n))) - math.log(1 + n)) < 1e-15


def test_softplus_derivative_is_sigmoid():
    x = np.linspace(-6, 6, 25)
    h = 1e-5
    fd = (OG.softplus(x + h) - OG.softplus(x - h)) / (2 * h)
    np.testing.assert_allclose(fd, OG.sigmoid(x), rtol=0, atol=1e-9)


@pytest.mark.parametrize('A', [1.0, 0.5, 1.0 / 256, 3.0])
def test_forget_gate_at_zero_logit(A):
    # softplus(0) = ln 2, so alpha = exp(-A ln 2) = 2^-A
    assert abs(float(OG.forget_gate(0.0, A)) - 2.0 ** (-A)) < 1e-15


def test_forget_gate_limits_and_range():
    A = np.array([1.0, 0.25, 1.0 / 256])
    assert np.all(np.abs(OG.forget_gate(-60.0, A) - 1.0) < 1e-15)
    assert np.all(OG.forget_gate(800.0, A[:1]) == 0.0)
    assert float(OG.forget_gate(40.0, 1.0)) < 1e-17
    f = np.linspace(-20, 20, 81)
    for a in A:
        al = OG.forget_gate(f, a)
        assert np.all((al > 0) & (al <= 1))
        assert np.all(np.diff(al) < 0)          # a larger logit forgets more
    # exp(-(A1 + A2) s) = exp(-A1 s) exp(-A2 s)
    np.testing.assert_allclose(OG.forget_gate(f, 0.75),
                               OG.forget_gate(f, 0.5) * OG.forget_gate(f, 0.25), rtol=1e-14)
    # broadcasting of a per-sequence A against [N, T] logits
    ff = np.zeros((2, 3))
    got = OG.forget_gate(ff, np.array([1.0, 2.0])[:, None])
    np.testing.assert_allclose(got, [[0.5] * 3, [0.25] * 3], rtol=1e-15)


def test_write_strength_range():
    x = np.linspace(-30, 30, 121)
    b = OG.write_strength(x)
    assert np.all((b > 0) & (b < 1))
    np.testing.assert_array_equal(b, OG.sigmoid(x))
    assert OG.clock_increment(0.0) == 0.5


def test_cumulative_clock_closed_form_and_order():
    T = 50
    delta = np.full((2, T), 0.375)
    lam = OG.cumulative_clock(delta, np.array([[1.5], [-4.0]]), axis=1)
    np.testing.assert_allclose(lam[0], 1.5 + 0.375 * np.arange(1, T + 1), rtol=0, atol=1e-13)
    np.testing.assert_allclose(lam[1], -4.0 + 0.375 * np.arange(1, T + 1), rtol=0, atol=1e-13)
    rng = np.random.default_rng(0)
    d = OG.clock_increment(rng.standard_normal(200))
    assert np.all(np.diff(OG.cumulative_clock(d)) > 0)
