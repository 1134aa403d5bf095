"""Pins of the oracle's forward forms (Sec. 3.1-3.3, App. A.3-A.6, App. B).

The four forms are written independently (cosine-sum kernel, Phi/U/b,
closed Dirichlet form, chunk matrices); they must agree to 1e-10.  Special
cases reduce to textbook objects.
"""
import numpy as np
import pytest

from oracle import basis, forward as F, gates as G


def _case(N, T, d, m, seed, A=0.5, jitter=0.3):
    rng = np.random.default_rng(seed)
    q = rng.standard_normal((N, T, d))
    k = rng.standard_normal((N, T, d))
    v = rng.standard_normal((N, T, d))
    delta = G.clock_increment(rng.standard_normal((N, T)))
    alpha = G.forget_gate(rng.standard_normal((N, T)), A)
    beta = G.write_strength(rng.standard_normal((N, T)))
    R = np.eye(m)[None] + jitter * rng.standard_normal((N, m, m))
    return q, k, v, delta, alpha, beta, R


@pytest.mark.parametrize('m,T,d', [(5, 17, 3), (7, 12, 4), (127, 9, 5), (255, 7, 3)])
def test_four_forms_agree(m, T, d):
    q, k, v, delta, alpha, beta, R = _case(2, T, d, m, seed=m)
    s = 0.9
    o_rel, K_rel, V_rel = F.relative_time(q, k, v, delta, alpha, beta, R, s)
    o_abs, Kb, Vb, lam_T = F.absolute_clock(q, k, v, delta, alpha, beta, R, s)
    o_quad = F.quadratic(q, k, v, delta, alpha, beta, R, s)
    np.testing.assert_allclose(o_abs, o_rel, atol=1e-10, rtol=0)
    np.testing.assert_allclose(o_quad, o_rel, atol=1e-10, rtol=0)
    for C in (1, 4, 64):
        o_ch, Kc, Vc = F.chunkwise(q, k, v, delta, alpha, beta, R, s, C)
        np.testing.assert_allclose(o_ch, o_rel, atol=1e-10, rtol=0)
        np.testing.assert_allclose(Kc, Kb, atol=1e-10, rtol=0)
        np.testing.assert_allclose(Vc, Vb, atol=1e-10, rtol=0)
    # Eq. cyfa-relative-reconstruction: K_t = Phi U(lambda_t) Kbar_t
    phi = basis.fourier_basis(m)
    for n in range(2):
        np.testing.assert_allclose(phi @ basis.U(lam_T[n], m) @ Kb[n], K_rel[n], atol=1e-10)
        np.testing.assert_allclose(phi @ basis.U(lam_T[n], m) @ Vb[n], V_rel[n], atol=1e-10)


def test_textbook_softmax_attention():
    """Unit integer clock, no decay, full writes, R = I, T <= m.

    Cardinality (App. A.2) puts token i in slot t - i exactly, so the readout
    is causal softmax attention over the t written slots plus m - t empty
    slots with logit 0:  o_t = sum_i e^{s q_t.k_i} v_i / (sum_i e^{s q_t.k_i} + m - t).
    """
    m, T, d, s = 7, 6, 3, 0.8
    rng = np.random.default_rng(5)
    q = rng.standard_normal((1, T, d))
    k = rng.standard_normal((1, T, d))
    v = rng.standard_normal((1, T, d))
    one = np.ones((1, T))
    R = np.eye(m)[None]
    want = np.zeros((T, d))
    for t in range(T):
        w = np.exp(s * k[0, :t + 1] @ q[0, t])
        want[t] = (w @ v[0, :t + 1]) / (w.sum() + (m - (t + 1)))
    for o in (F.relative_time(q, k, v, one, one, one, R, s)[0],
              F.absolute_clock(q, k, v, one, one, one, R, s)[0],
              F.chunkwise(q, k, v, one, one, one, R, s, 4)[0],
              F.quadratic(q, k, v, one, one, one, R, s)):
        np.testing.assert_allclose(o[0], want, atol=1e-12)


def test_single_slot_is_decayed_cumsum():
    """m = 1: the softmax has one entry, so o_t = R sum_i beta_i prod_{j>i} alpha_j v_i."""
    q, k, v, delta, alpha, beta, _ = _case(1, 11, 3, 1, seed=9)
    R = np.array([[[1.7]]])
    want = np.zeros((11, 3))
    acc = np.zeros(3)
    for t in range(11):
        acc = alpha[0, t] * acc + beta[0, t] * v[0, t]
        want[t] = 1.7 * acc
    for o in (F.relative_time(q, k, v, delta, alpha, beta, R, 1.0)[0],
              F.absolute_clock(q, k, v, delta, alpha, beta, R, 1.0)[0],
              F.chunkwise(q, k, v, delta, alpha, beta, R, 1.0, 4)[0]):
        np.testing.assert_allclose(o[0], want, atol=1e-12)


def test_clock_origin_invariance():
    """Prop. 6: lambda -> lambda + c changes Kbar by U(-c) and leaves o unchanged."""
    m = 9
    q, k, v, delta, alpha, beta, R = _case(2, 10, 4, m, seed=11)
    o0, K0, V0, _ = F.absolute_clock(q, k, v, delta, alpha, beta, R, 0.7)
    for c in (0.3, 5.0, -123.456):
        o1, K1, V1, _ = F.absolute_clock(q, k, v, delta, alpha, beta, R, 0.7,
                                         lambda0=np.full(2, c))
        np.testing.assert_allclose(o1, o0, atol=1e-11)
        for n in range(2):
            np.testing.assert_allclose(K1[n], basis.U(-c, m) @ K0[n], atol=1e-11)


def test_fixed_rate_profile():
    """App. A.6: delta = 1/rho gives the Fourier-Dirichlet profile of Eq. app-constant-rate-profile."""
    m, rho, T = 7, 3.0, 15
    d = 1
    k = np.zeros((1, T, d))
    k[0, 0, 0] = 1.0                      # only token 1 writes a key
    q = np.zeros((1, T, d))
    v = np.zeros((1, T, d))
    delta = np.full((1, T), 1.0 / rho)
    one = np.ones((1, T))
    R = np.eye(m)[None]
    Tcyc = rho * m
    for t in range(T):
        _, K, _ = F.relative_time(q[:, :t + 1], k[:, :t + 1], v[:, :t + 1], delta[:, :t + 1],
                                  one[:, :t + 1], one[:, :t + 1], R, 1.0)
        r = np.arange(m)
        hh = np.arange(1, (m - 1) // 2 + 1)[:, None]
        prof = (1 + 2 * np.cos(2 * np.pi * hh * (t - 0 - rho * r) / Tcyc).sum(0)) / m
        np.testing.assert_allclose(K[0, :, 0], prof, atol=1e-12)


def test_profile_overlap_depends_only_on_clock_gap():
    """Prop. 4 / Cor. 1: profile inner products are constant in t and follow the closed form."""
    m = 11
    rng = np.random.default_rng(4)
    lam = np.cumsum(rng.uniform(0, 1, size=8))
    i, j = 2, 5
    for t in range(5, 8):
        pi = basis.shift_matrix(lam[t] - lam[i], m)[:, 0]
        pj = basis.shift_matrix(lam[t] - lam[j], m)[:, 0]
        np.testing.assert_allclose(pi @ pj, basis.shift_kernel_closed(lam[i] - lam[j], m),
                                   atol=1e-12)


def test_initial_state_continuation():
    """Splitting a sequence and carrying (Kbar, Vbar, lambda) gives the unsplit result."""
    q, k, v, delta, alpha, beta, R = _case(2, 14, 3, 7, seed=13)
    o, Kb, Vb, lam = F.absolute_clock(q, k, v, delta, alpha, beta, R, 0.6)
    o1, K1, V1, l1 = F.absolute_clock(q[:, :9], k[:, :9], v[:, :9], delta[:, :9], alpha[:, :9],
                                      beta[:, :9], R, 0.6)
    o2, K2, V2, l2 = F.absolute_clock(q[:, 9:], k[:, 9:], v[:, 9:], delta[:, 9:], alpha[:, 9:],
                                      beta[:, 9:], R, 0.6, lambda0=l1, Kbar0=K1, Vbar0=V1)
    np.testing.assert_allclose(np.concatenate([o1, o2], 1), o, atol=1e-12)
    np.testing.assert_allclose(K2, Kb, atol=1e-12)
    np.testing.assert_allclose(l2, lam, atol=1e-12)


def test_clock_is_order_preserving():
    """Prop. 5: lambda_j - lambda_i lies in (0, j - i) for i < j."""
    delta = G.clock_increment(np.random.default_rng(0).standard_normal(50) * 4)
    lam = G.cumulative_clock(delta)
    for i in range(0, 50, 7):
        for j in range(i + 1, 50, 5):
            gap = lam[j] - lam[i]
            assert 0 < gap < j - i


@pytest.mark.parametrize('m', [7, 127])
def test_chunk_form_over_128_token_chunks(m):
    """App. B at the blocking of the tensor-core path: two full 128-token chunks and a ragged
    tail, with slow decay (A = 0.02) so the state carried across chunk boundaries matters."""
    q, k, v, delta, alpha, beta, R = _case(1, 300, 4, m, seed=300 + m, A=0.02)
    s = 0.7
    o_rel = F.relative_time(q, k, v, delta, alpha, beta, R, s)[0]
    o_abs, Kb, Vb, _ = F.absolute_clock(q, k, v, delta, alpha, beta, R, s)
    o_ch, Kc, Vc = F.chunkwise(q, k, v, delta, alpha, beta, R, s, 128)
    np.testing.assert_allclose(o_ch, o_rel, atol=1e-10, rtol=0)
    np.testing.assert_allclose(o_ch, o_abs, atol=1e-10, rtol=0)
    np.testing.assert_allclose(Kc, Kb, atol=1e-10, rtol=0)
    np.testing.assert_allclose(Vc, Vb, atol=1e-10, rtol=0)
    # the state carried into the last chunk still weighs: its decay over the first two chunks
    decay = np.prod(alpha[0, :256])
    assert decay > 1e-3, decay
