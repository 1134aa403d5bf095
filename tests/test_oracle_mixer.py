"""Pins of oracle/mixer.py (ShortConv, SiLU, RMSNorm, output gate) against values the mathematics
fixes, and of its gradients against central finite differences."""
import numpy as np
import pytest

from oracle import mixer as MX


def test_short_conv_identity_delay_and_convolve():
    rng = np.random.default_rng(0)
    x = rng.standard_normal((2, 9, 3))
    ident = np.zeros((3, 4))
    ident[:, 3] = 1.0                     # last tap reads the current token
    np.testing.assert_array_equal(MX.short_conv(x, ident), x)
    delay = np.zeros((3, 4))
    delay[:, 2] = 1.0                     # one token back, zero before the first
    want = np.concatenate([np.zeros((2, 1, 3)), x[:, :-1]], axis=1)
    np.testing.assert_array_equal(MX.short_conv(x, delay), want)
    w = rng.standard_normal((3, 4))
    got = MX.short_conv(x, w)
    for n in range(2):
        for c in range(3):
            # causal: full convolution with the reversed filter, first T outputs
            ref = np.convolve(x[n, :, c], w[c, ::-1])[:9]
            np.testing.assert_allclose(got[n, :, c], ref, rtol=0, atol=1e-13)
    # shorter sequences than the filter
    np.testing.assert_allclose(MX.short_conv(x[:, :2], w), got[:, :2], atol=1e-14)


def test_silu_values():
    assert MX.silu(np.array(0.0)) == 0.0
    # the oracle's sigmoid is accurate to ~1e-16 absolute (not relative) in the far negative tail
    np.testing.assert_allclose(MX.silu(np.array([30.0, -30.0])), [30.0, -30.0 / (1 + np.exp(30))],
                               rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(MX.silu(np.log(3.0)), np.log(3.0) * 0.75, rtol=1e-15)
    assert abs(float(MX.silu_grad(np.array(0.0))) - 0.5) < 1e-15
    x = np.linspace(-5, 5, 21)
    h = 1e-6
    np.testing.assert_allclose(MX.silu_grad(x), (MX.silu(x + h) - MX.silu(x - h)) / (2 * h),
                               atol=1e-8)


def test_rms_norm_unit_rms_and_scale_invariance():
    rng = np.random.default_rng(1)
    a = rng.standard_normal((4, 5, 16)) * 3
    y = MX.rms_norm(a, np.ones(16), 0.0)
    np.testing.assert_allclose(np.sqrt(np.mean(y * y, axis=-1)), 1.0, rtol=1e-13)
    np.testing.assert_allclose(MX.rms_norm(7.5 * a, np.ones(16), 0.0), y, rtol=1e-13)
    g = rng.standard_normal(16)
    np.testing.assert_allclose(MX.rms_norm(a, g, 0.0), y * g, rtol=1e-13)
    # eps: a zero row stays zero; a constant row c gives c / sqrt(c^2 + eps)
    assert np.all(MX.rms_norm(np.zeros((1, 16)), g, 1e-6) == 0)
    np.testing.assert_allclose(MX.rms_norm(np.full((1, 16), 0.01), np.ones(16), 1e-4),
                               0.01 / np.sqrt(1e-4 + 1e-4), rtol=1e-13)


def test_mixer_post_reduces_to_its_parts():
    rng = np.random.default_rng(2)
    o = rng.standard_normal((3, 8))
    g = rng.standard_normal(8)
    np.testing.assert_allclose(MX.mixer_post(o, np.zeros((3, 8)), g, 1e-6),
                               0.5 * MX.rms_norm(o, g, 1e-6), rtol=1e-15)
    np.testing.assert_allclose(MX.mixer_post(o, np.full((3, 8), 50.0), g, 1e-6),
                               MX.rms_norm(o, g, 1e-6), rtol=1e-15)


def _fd(f, x, h=1e-6):
    g = np.zeros_like(x)
    it = np.nditer(x, flags=['multi_index'])
    for _ in it:
        i = it.multi_index
        x0 = x[i]
        x[i] = x0 + h
        fp = f()
        x[i] = x0 - h
        fm = f()
        x[i] = x0
        g[i] = (fp - fm) / (2 * h)
    return g


def test_mixer_pre_backward_finite_differences():
    rng = np.random.default_rng(3)
    N, T, H, d, K = 1, 6, 2, 4, 4
    C = H * d
    xq, xk, xv = (rng.standard_normal((N, T, C)) for _ in range(3))
    wq, wk, wv = (rng.standard_normal((C, K)) * 0.7 for _ in range(3))
    gq, gk = rng.standard_normal(d), rng.standard_normal(d)
    dq, dk, dv = (rng.standard_normal((N, T, C)) for _ in range(3))
    eps = 1e-3

    def loss():
        q, k, v = MX.mixer_pre(xq, xk, xv, wq, wk, wv, gq, gk, eps, H)
        return np.sum(q * dq) + np.sum(k * dk) + np.sum(v * dv)

    got = MX.mixer_pre_backward(xq, xk, xv, wq, wk, wv, gq, gk, eps, H, dq, dk, dv)
    for name, arr in (('dxq', xq), ('dxk', xk), ('dxv', xv), ('dwq', wq), ('dwk', wk),
                      ('dwv', wv), ('dgq', gq), ('dgk', gk)):
        np.testing.assert_allclose(got[name], _fd(loss, arr), rtol=1e-6, atol=1e-7, err_msg=name)


def test_mixer_post_backward_finite_differences():
    rng = np.random.default_rng(4)
    o = rng.standard_normal((2, 3, 8))
    z = rng.standard_normal((2, 3, 8))
    g = rng.standard_normal(8)
    dy = rng.standard_normal((2, 3, 8))
    eps = 1e-3

    def loss():
        return np.sum(MX.mixer_post(o, z, g, eps) * dy)

    do, dz, dg = MX.mixer_post_backward(o, z, g, eps, dy)
    np.testing.assert_allclose(do, _fd(loss, o), rtol=1e-6, atol=1e-7)
    np.testing.assert_allclose(dz, _fd(loss, z), rtol=1e-6, atol=1e-7)
    np.testing.assert_allclose(dg, _fd(loss, g), rtol=1e-6, atol=1e-7)
