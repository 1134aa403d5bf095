"""Four independent float64 forward forms of the CyFA operator -- test infrastructure only.

Shapes (N independent (batch, head) sequences, m active slots, no padding):
    q, k : [N, T, dk]      v : [N, T, dv]
    delta, alpha, beta : [N, T]   (post-activation gates, see ``gates``)
    R : [N, m, m]          scale : float (the dot-product scale s; q enters as s*q)
Output o : [N, T, dv].

The dot-product scale is left out of the paper's notation (Sec. 3.1, footnote
to Eq. cyfa-physical-readout); here the query is multiplied by ``scale``
before the key pass, which is the same as scaling the slot logits R K q.

Forms:
* ``relative_time``  -- the defining recurrence, Sec. 3.1 Eq.
  cyfa-physical-recurrence, with P(delta) built from the cosine-sum kernel of
  Prop. 2 (never from Phi or U), and readout Eq. cyfa-physical-readout.
* ``absolute_clock`` -- Sec. 3.2 Eq. cyfa-absolute-recurrence with the temporal
  write vector U(-lambda) b and readout Eq. cyfa-absolute-readout.
* ``quadratic``      -- Prop. 3 (Eq. app-unrolled-K / app-unrolled-V): the
  relative-time states as an explicit sum over writes, each profile
  P(lambda_t - lambda_i) e_0 taken from the closed Dirichlet form
  (Eq. app-kernel-closed).  O(T^2) per sequence; tiny inputs only.
* ``chunkwise``      -- App. B: Eqs. app-chunk-decay, app-chunk-rescale,
  app-temporal-writes, app-cyfa-key-chunk, app-cyfa-value-chunk, with the
  token-wise middle line of Eq. cyfa-two-pass between the passes.

Pins (tests/test_oracle_forms.py): all four agree to 1e-10; the textbook
special case (integer unit clock, no decay, R = I) equals causal softmax
attention with empty zero-logit slots; m = 1 reduces to a decayed cumulative
sum; the clock origin does not change the output (Prop. 6); the fixed-rate
clock reproduces the Fourier-Dirichlet profile (Eq. app-constant-rate-profile).
"""
import numpy as np

from . import basis


def _softmax(x):
    x = x - np.max(x, axis=-1, keepdims=True)
    e = np.exp(x)
    return e / np.sum(e, axis=-1, keepdims=True)


def relative_readout(R, K, V, qs):
    """o = (R V)^T softmax(R K qs), Eq. cyfa-physical-readout (batched over N)."""
    logits = np.einsum('nij,njd,nd->ni', R, K, qs)
    w = _softmax(logits)
    return np.einsum('nij,njd,ni->nd', R, V, w)


def relative_time(q, k, v, delta, alpha, beta, R, scale, K0=None, V0=None):
    """Step-by-step relative-time recurrence (Sec. 3.1).

    K_t = alpha_t P(delta_t) K_{t-1} + beta_t e_0 k_t^T (same for V), then the
    readout from K_t, V_t: the write of token t is visible at step t.
    P(delta) is circulant: entry (r, s) is the Prop. 2 kernel at delta + s - r,
    which is periodic in its argument with period m, so one row of m values
    indexed by (s - r) mod m fills the whole matrix.
    Returns (o, K_T, V_T).
    """
    N, T, dk = q.shape
    dv = v.shape[2]
    m = R.shape[1]
    K = np.zeros((N, m, dk)) if K0 is None else np.array(K0, dtype=np.float64)
    V = np.zeros((N, m, dv)) if V0 is None else np.array(V0, dtype=np.float64)
    o = np.zeros((N, T, dv))
    idx = (np.arange(m)[None, :] - np.arange(m)[:, None]) % m     # (s - r) mod m
    for t in range(T):
        row = basis.shift_kernel_sum(delta[:, t, None] + np.arange(m)[None, :], m)  # [N, m]
        P = row[:, idx]                                                       # [N, m, m]
        K = alpha[:, t, None, None] * np.einsum('nrs,nsd->nrd', P, K)
        V = alpha[:, t, None, None] * np.einsum('nrs,nsd->nrd', P, V)
        K[:, 0, :] += beta[:, t, None] * k[:, t, :]
        V[:, 0, :] += beta[:, t, None] * v[:, t, :]
        o[:, t, :] = relative_readout(R, K, V, scale * q[:, t, :])
    return o, K, V


def _rotation_angles(lam, m):
    """theta_j = 2 pi j lam / m for j = 1..(m-1)/2, shape [..., (m-1)/2]."""
    j = np.arange(1, (m - 1) // 2 + 1, dtype=np.float64)
    return 2.0 * np.pi * np.asarray(lam, dtype=np.float64)[..., None] * j / m


def apply_U(tau, x):
    """U(tau) x for a batch: tau [N], x [N, m]  (Eq. cyfa-fractional-shift)."""
    m = x.shape[-1]
    th = _rotation_angles(tau, m)
    c, s = np.cos(th), np.sin(th)
    y = x.copy()
    xc, xs = x[..., 1::2], x[..., 2::2]           # (cos_j, sin_j) pair entries
    y[..., 1::2] = c * xc - s * xs
    y[..., 2::2] = s * xc + c * xs
    return y


def write_vectors(lam, beta, m):
    """Temporal write vectors a_t = beta_t U(-lambda_t) b, [N, T, m] (Sec. 3.2)."""
    N, T = lam.shape
    b = basis.b_vector(m)
    bb = np.broadcast_to(b, (N * T, m))
    w = apply_U(-lam.reshape(-1), bb).reshape(N, T, m)
    return beta[..., None] * w


def middle_readout(o1, lam, M):
    """Middle line of Eq. cyfa-two-pass for a batch of rows.

    o1 [N, m] (key-pass output), lam [N], M = R Phi [N, m, m]:
    o'' = U(-lam) Phi^T R^T softmax(R Phi U(lam) o1).
    """
    z = apply_U(lam, o1)
    w = _softmax(np.einsum('nij,nj->ni', M, z))
    y = np.einsum('nij,ni->nj', M, w)
    return apply_U(-lam, y)


def absolute_clock(q, k, v, delta, alpha, beta, R, scale, lambda0=None,
                   Kbar0=None, Vbar0=None, return_trace=False):
    """Absolute-clock token recurrence (Sec. 3.2).

    lambda_t = lambda0 + sum_{u<=t} delta_u; a_t = beta_t U(-lambda_t) b;
    Kbar_t = alpha_t Kbar_{t-1} + a_t k_t^T; Vbar_t = alpha_t Vbar_{t-1} + a_t v_t^T;
    o_t = Vbar_t^T U(-lambda_t) Phi^T R^T softmax(R Phi U(lambda_t) Kbar_t (s q_t)).
    Returns (o, Kbar_T, Vbar_T, lambda_T) and, with ``return_trace``, a dict of
    per-token intermediates used by the backward oracle.
    """
    N, T, dk = q.shape
    dv = v.shape[2]
    m = R.shape[1]
    phi = basis.fourier_basis(m)
    M = np.einsum('nij,jk->nik', R, phi)
    lam0 = np.zeros(N) if lambda0 is None else np.asarray(lambda0, dtype=np.float64)
    lam = lam0[:, None] + np.cumsum(delta, axis=1)
    a = write_vectors(lam, beta, m)
    Kb = np.zeros((N, m, dk)) if Kbar0 is None else np.array(Kbar0, dtype=np.float64)
    Vb = np.zeros((N, m, dv)) if Vbar0 is None else np.array(Vbar0, dtype=np.float64)
    o = np.zeros((N, T, dv))
    o1s = np.zeros((N, T, m)) if return_trace else None
    o2s = np.zeros((N, T, m)) if return_trace else None
    for t in range(T):
        Kb = alpha[:, t, None, None] * Kb + a[:, t, :, None] * k[:, t, None, :]
        Vb = alpha[:, t, None, None] * Vb + a[:, t, :, None] * v[:, t, None, :]
        o1 = np.einsum('nrd,nd->nr', Kb, scale * q[:, t, :])
        o2 = middle_readout(o1, lam[:, t], M)
        o[:, t, :] = np.einsum('nrd,nr->nd', Vb, o2)
        if return_trace:
            o1s[:, t] = o1
            o2s[:, t] = o2
    out = (o, Kb, Vb, lam[:, -1] if T > 0 else lam0)
    if return_trace:
        return out + ({'lam': lam, 'a': a, 'M': M, 'o1': o1s, 'o2': o2s},)
    return out


def quadratic(q, k, v, delta, alpha, beta, R, scale):
    """Unrolled relative-time states (Prop. 3), evaluated independently per t.

    K_t = sum_{i<=t} beta_i (prod_{j=i+1}^t alpha_j) P(lambda_t - lambda_i) e_0 k_i^T
    with [P(tau) e_0]_r = sin(pi (tau - r)) / (m sin(pi (tau - r) / m))
    (Eq. app-kernel-closed with s = 0), then the Eq. cyfa-physical-readout.
    """
    N, T, dk = q.shape
    m = R.shape[1]
    lam = np.cumsum(delta, axis=1)
    r = np.arange(m, dtype=np.float64)
    o = np.zeros((N, T, v.shape[2]))
    for t in range(T):
        decay = np.ones((N, t + 1))
        for i in range(t + 1):
            decay[:, i] = np.prod(alpha[:, i + 1:t + 1], axis=1)
        coef = beta[:, :t + 1] * decay                                     # [N, t+1]
        age = lam[:, t, None] - lam[:, :t + 1]                             # [N, t+1]
        prof = basis.shift_kernel_closed(age[..., None] - r, m)            # [N, t+1, m]
        K = np.einsum('ni,nir,nid->nrd', coef, prof, k[:, :t + 1])
        V = np.einsum('ni,nir,nid->nrd', coef, prof, v[:, :t + 1])
        o[:, t] = relative_readout(R, K, V, scale * q[:, t])
    return o


def chunkwise(q, k, v, delta, alpha, beta, R, scale, C):
    """Chunk-wise two-pass form of App. B (fp64, exact up to rounding).

    Per chunk [i+1] of C tokens: gamma^r = prod_{j<=r} alpha, Gamma_rs =
    gamma^r / gamma^s (r >= s), X<- scales row r by gamma^r, X-> by
    gamma^C / gamma^r; A holds the rows beta U(-lambda) b.
        Kbar_{[i+1]} = gamma^C Kbar_{[i]} + A->^T K
        O'  = Q<- Kbar_{[i]}^T + (Q K^T o Gamma) A
        O'' = middle line of Eq. cyfa-two-pass, row by row
        Vbar_{[i+1]} = gamma^C Vbar_{[i]} + A^T V->
        O   = O''<- Vbar_{[i]} + (O'' A^T o Gamma) V
    A trailing partial chunk is handled with its own length.
    """
    N, T, dk = q.shape
    dv = v.shape[2]
    m = R.shape[1]
    phi = basis.fourier_basis(m)
    M = np.einsum('nij,jk->nik', R, phi)
    lam = np.cumsum(delta, axis=1)
    A_all = write_vectors(lam, beta, m)
    Kb = np.zeros((N, m, dk))
    Vb = np.zeros((N, m, dv))
    o = np.zeros((N, T, dv))
    for c0 in range(0, T, C):
        c1 = min(T, c0 + C)
        L = c1 - c0
        gam = np.cumprod(alpha[:, c0:c1], axis=1)                          # gamma^r, r=1..L
        Gam = np.tril(gam[:, :, None] / gam[:, None, :])                   # [N, L, L]
        Qc = scale * q[:, c0:c1]
        Kc, Vc, Ac = k[:, c0:c1], v[:, c0:c1], A_all[:, c0:c1]
        back = gam                                                          # <- factors
        fwd = gam[:, -1:] / gam                                             # -> factors
        O1 = (np.einsum('nr,nrd,nmd->nrm', back, Qc, Kb)
              + np.einsum('nrs,nsm->nrm', np.einsum('nrd,nsd->nrs', Qc, Kc) * Gam, Ac))
        O2 = np.stack([middle_readout(O1[:, r], lam[:, c0 + r], M) for r in range(L)], axis=1)
        o[:, c0:c1] = (np.einsum('nr,nrm,nmd->nrd', back, O2, Vb)
                       + np.einsum('nrs,nsd->nrd', np.einsum('nrm,nsm->nrs', O2, Ac) * Gam, Vc))
        Kb = gam[:, -1, None, None] * Kb + np.einsum('nsm,nsd->nmd', fwd[..., None] * Ac, Kc)
        Vb = gam[:, -1, None, None] * Vb + np.einsum('nsm,nsd->nmd', Ac, fwd[..., None] * Vc)
    return o, Kb, Vb
