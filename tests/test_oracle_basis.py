"""Pins of the oracle's cyclic-transport objects against what the paper fixes.

Sec. 3.1 and App. A.1-A.2: Phi orthogonal, P(1) the printed permutation, b
the printed vector, group law / inverse / period, the Prop. 2 kernel in its
three forms, cardinality, partition of unity, the frame orbit.
"""
import os

import numpy as np
import pytest

from oracle import basis

GOLD = os.path.join(os.path.dirname(__file__), 'golden')
ODD_M = [1, 3, 5, 7, 9, 127]


def _load(name):
    return np.loadtxt(os.path.join(GOLD, name), comments='#', ndmin=1)


@pytest.mark.parametrize('m', ODD_M)
def test_phi_orthogonal(m):
    phi = basis.fourier_basis(m)
    np.testing.assert_allclose(phi.T @ phi, np.eye(m), atol=1e-12)
    np.testing.assert_allclose(phi @ phi.T, np.eye(m), atol=1e-12)


def test_even_m_rejected():
    with pytest.raises(ValueError):
        basis.fourier_basis(4)


def test_unit_shift_matches_printed_matrix():
    gold = _load('cyclic_shift_m5.txt')
    np.testing.assert_allclose(basis.shift_matrix(1.0, 5), gold, atol=1e-12)
    np.testing.assert_allclose(basis.shift_matrix_kernel(1.0, 5), gold, atol=1e-12)
    np.testing.assert_array_equal(basis.cyclic_permutation(5), gold)


@pytest.mark.parametrize('m', [3, 7, 127])
def test_unit_shift_is_cyclic_permutation(m):
    # (P x)_r = x_{r-1 mod m}
    x = np.random.default_rng(m).standard_normal(m)
    np.testing.assert_allclose(basis.shift_matrix(1.0, m) @ x, np.roll(x, 1), atol=1e-12)


def test_b_matches_printed_vector():
    np.testing.assert_allclose(basis.b_vector(5), _load('b_vector_m5.txt'), atol=1e-15)


@pytest.mark.parametrize('m', [7, 127])
def test_b_structure(m):
    b = basis.b_vector(m)
    assert abs(b[0] - 1 / np.sqrt(m)) < 1e-15
    np.testing.assert_allclose(b[1::2], np.sqrt(2 / m), atol=1e-15)
    np.testing.assert_allclose(b[2::2], 0.0, atol=1e-15)


@pytest.mark.parametrize('m', [5, 7, 127])
def test_group_law_inverse_period(m):
    rng = np.random.default_rng(1)
    for _ in range(3):
        t1, t2 = rng.uniform(-300, 300, size=2)
        P1, P2 = basis.shift_matrix(t1, m), basis.shift_matrix(t2, m)
        np.testing.assert_allclose(P1 @ P2, basis.shift_matrix(t1 + t2, m), atol=1e-10)
        np.testing.assert_allclose(P1 @ basis.shift_matrix(-t1, m), np.eye(m), atol=1e-10)
        np.testing.assert_allclose(basis.shift_matrix(t1 + m, m), P1, atol=1e-10)
        np.testing.assert_allclose(P1.T @ P1, np.eye(m), atol=1e-10)
        np.testing.assert_allclose(basis.U(t1, m).T, basis.U(-t1, m), atol=1e-12)
    np.testing.assert_allclose(basis.shift_matrix(0.0, m), np.eye(m), atol=1e-12)


@pytest.mark.parametrize('m', [5, 9, 127])
def test_kernel_three_forms(m):
    rng = np.random.default_rng(2)
    tau = rng.uniform(-5, 5)
    P = basis.shift_matrix(tau, m)
    r = np.arange(m)[:, None]
    s = np.arange(m)[None, :]
    x = tau + s - r
    np.testing.assert_allclose(basis.shift_kernel_sum(x, m), P, atol=1e-11)
    np.testing.assert_allclose(basis.shift_kernel_closed(x, m), P, atol=1e-11)
    # the closed form at its removable singularities (x a multiple of m)
    xs = np.array([0.0, float(m), -2.0 * m, 3.0])
    np.testing.assert_allclose(basis.shift_kernel_closed(xs, m), basis.shift_kernel_sum(xs, m),
                               atol=1e-11)


@pytest.mark.parametrize('m', [5, 7, 127])
def test_cardinality_and_partition_of_unity(m):
    for a in [0, 1, 2, m - 1, m + 3, -4]:
        P = basis.shift_matrix(float(a), m)
        for sl in [0, 1, m - 1]:
            e = np.zeros(m)
            e[(sl + a) % m] = 1.0
            np.testing.assert_allclose(P[:, sl], e, atol=1e-11)
    rng = np.random.default_rng(3)
    for tau in rng.uniform(-10, 10, size=4):
        P = basis.shift_matrix(tau, m)
        np.testing.assert_allclose(P.sum(axis=0), 1.0, atol=1e-11)       # 1^T P e_s = 1
        np.testing.assert_allclose(P.T @ P, np.eye(m), atol=1e-11)      # profile orthonormality


@pytest.mark.parametrize('m', [5, 127])
def test_frame_orbit(m):
    # Phi^T e_r = U(r) b, Eq. app-frame-orbit
    phi = basis.fourier_basis(m)
    b = basis.b_vector(m)
    for r in [0, 1, 3, m - 1]:
        np.testing.assert_allclose(phi[r, :], basis.U(float(r), m) @ b, atol=1e-12)


@pytest.mark.parametrize('m', [5, 127])
def test_omega_is_generator(m):
    tau, h = 0.37, 1e-6
    dU = (basis.U(tau + h, m) - basis.U(tau - h, m)) / (2 * h)
    np.testing.assert_allclose(dU, basis.omega(m) @ basis.U(tau, m), atol=1e-7)


@pytest.mark.parametrize('m', [5, 127, 255])
def test_U_commutes_with_its_generator(m):
    # U(tau) = exp(tau Omega): U commutes with Omega, so the bilinear forms <x, y> and
    # <x, Omega y> are the same before and after one rotation of both vectors (the CUDA-core
    # readout gradient takes them before its final rotation by U(-lam))
    rng = np.random.default_rng(4)
    tau = rng.uniform(-300, 300)
    Ut, W = basis.U(tau, m), basis.omega(m)
    np.testing.assert_allclose(Ut @ W, W @ Ut, atol=1e-12)
    np.testing.assert_allclose(W.T, -W, atol=0)
    x, y = rng.standard_normal(m), rng.standard_normal(m)
    assert abs((Ut @ x) @ (Ut @ y) - x @ y) < 1e-10
    assert abs((Ut @ x) @ (W @ (Ut @ y)) - x @ (W @ y)) < 1e-9


def test_state_size_accounting():
    H, ms, dk, dv, entries = _load('state_size.txt').astype(int)
    assert H * ms * (dk + dv) == entries
