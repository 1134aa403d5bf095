"""Cyclic-transport objects of CyFA in float64 -- test infrastructure only.

All functions take the number of active relative-time slots ``m`` (odd) and
return plain numpy float64 arrays of size m (no padding row).

Pins (tests/test_oracle_basis.py): Phi orthogonal (Prop. 1); P(1) equal to the
printed cyclic permutation (Eq. cyfa-cyclic-permutation, golden fixture);
b equal to the printed vector (Eq. app-b-explicit, golden fixture); group law,
inverse and period (Eq. app-group-properties); the cosine-sum kernel equal to
the closed Dirichlet form (Eq. app-kernel-closed) and to Phi U Phi^T entries
(Eq. app-kernel-inner-product); cardinality and partition of unity.
"""
import numpy as np


def _check_m(m):
    if m < 1 or m % 2 == 0:
        raise ValueError("CyFA uses an odd number of active slots, got m=%d" % m)


def fourier_basis(m):
    """Real orthogonal Fourier basis Phi (m x m), App. A.1 Eq. app-real-fourier.

    Column 0 is the DC column 1/sqrt(m); columns 2j-1 and 2j hold
    sqrt(2/m) cos(2 pi j r / m) and sqrt(2/m) sin(2 pi j r / m), r = row index.
    """
    _check_m(m)
    r = np.arange(m, dtype=np.float64)
    phi = np.empty((m, m), dtype=np.float64)
    phi[:, 0] = 1.0 / np.sqrt(m)
    for j in range(1, (m - 1) // 2 + 1):
        phi[:, 2 * j - 1] = np.sqrt(2.0 / m) * np.cos(2.0 * np.pi * j * r / m)
        phi[:, 2 * j] = np.sqrt(2.0 / m) * np.sin(2.0 * np.pi * j * r / m)
    return phi


def rotation(theta):
    """Rot(theta), Sec. 3.1 Eq. cyfa-rotation-block."""
    c, s = np.cos(theta), np.sin(theta)
    return np.array([[c, -s], [s, c]], dtype=np.float64)


def U(tau, m):
    """U(tau) = 1 (+) blockdiag_j Rot(2 pi j tau / m), Eq. cyfa-fractional-shift."""
    _check_m(m)
    u = np.zeros((m, m), dtype=np.float64)
    u[0, 0] = 1.0
    for j in range(1, (m - 1) // 2 + 1):
        u[2 * j - 1:2 * j + 1, 2 * j - 1:2 * j + 1] = rotation(2.0 * np.pi * j * tau / m)
    return u


def omega(m):
    """Generator of U: dU(tau)/dtau = Omega U(tau).

    Differentiating each block Rot(2 pi j tau / m) of Eq. cyfa-fractional-shift
    gives (2 pi j / m) [[0, -1], [1, 0]] Rot(...); the DC entry is constant.
    """
    _check_m(m)
    w = np.zeros((m, m), dtype=np.float64)
    for j in range(1, (m - 1) // 2 + 1):
        f = 2.0 * np.pi * j / m
        w[2 * j - 1, 2 * j] = -f
        w[2 * j, 2 * j - 1] = f
    return w


def shift_matrix(tau, m):
    """P(tau) = Phi U(tau) Phi^T, Eq. cyfa-fractional-shift."""
    phi = fourier_basis(m)
    return phi @ U(tau, m) @ phi.T


def b_vector(m):
    """b = Phi^T e_0, Eq. cyfa-fourier-coordinates (explicit form Eq. app-b-explicit)."""
    return fourier_basis(m)[0, :].copy()


def shift_kernel_sum(x, m):
    """(1/m) [1 + 2 sum_{j=1}^{(m-1)/2} cos(2 pi j x / m)], Eq. app-kernel-sum.

    Prop. 2: e_r^T P(tau) e_s equals this with x = tau + s - r.  Accepts an
    array ``x`` and works elementwise.
    """
    _check_m(m)
    x = np.asarray(x, dtype=np.float64)
    acc = np.ones_like(x)
    for j in range(1, (m - 1) // 2 + 1):
        acc = acc + 2.0 * np.cos(2.0 * np.pi * j * x / m)
    return acc / m


def shift_kernel_closed(x, m):
    """sin(pi x) / (m sin(pi x / m)), Eq. app-kernel-closed.

    Where the denominator vanishes (x a multiple of m) the ratio is taken by
    continuity: its limit is cos(pi x) / cos(pi x / m), which is +-1 there.
    """
    _check_m(m)
    x = np.asarray(x, dtype=np.float64)
    den = m * np.sin(np.pi * x / m)
    # distance to the nearest multiple of m decides which branch is used
    near = np.abs(x / m - np.round(x / m)) < 1e-9
    safe = np.where(near, 1.0, den)
    val = np.sin(np.pi * x) / safe
    lim = np.cos(np.pi * x) / np.cos(np.pi * x / m)
    return np.where(near, lim, val)


def shift_matrix_kernel(tau, m):
    """P(tau) assembled entry by entry from the cosine-sum kernel (Prop. 2).

    Never touches Phi or U: this is the form the relative-time recurrence of
    the oracle uses, so that its agreement with the absolute-clock form is a
    check of both.
    """
    r = np.arange(m)[:, None]
    s = np.arange(m)[None, :]
    return shift_kernel_sum(tau + s - r, m)


def cyclic_permutation(m):
    """The unit cyclic shift P = Z + e_0 e_{m-1}^T of Eq. cyfa-cyclic-permutation."""
    p = np.zeros((m, m), dtype=np.float64)
    for r in range(m - 1):
        p[r + 1, r] = 1.0
    p[0, m - 1] = 1.0
    return p
