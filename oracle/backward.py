"""Reverse-mode gradient of the CyFA operator in float64 -- test infrastructure only.

Differentiates the absolute-clock token recurrence of Sec. 3.2 (the same
function as ``forward.absolute_clock``, which is pinned equal to the defining
relative-time recurrence) from the raw per-token logits:

    delta = sigmoid(c), alpha = exp(-A softplus(f)), beta = sigmoid(g_b),
    lambda_t = lambda0 + sum_{u<=t} delta_u, a_t = beta_t U(-lambda_t) b,
    Kbar_t = alpha_t Kbar_{t-1} + a_t k_t^T,  Vbar_t = alpha_t Vbar_{t-1} + a_t v_t^T,
    o'_t = Kbar_t (s q_t),  z_t = U(lambda_t) o'_t,  p_t = softmax(M z_t),
    o''_t = U(-lambda_t) M^T p_t,  o_t = Vbar_t^T o''_t,   M = R Phi.

The paper gives no gradient formula except the clock accumulation
dL/d delta_s = sum_{t>=s} dL/d lambda_t (App. D.1, Eq.
app-clock-gradient-accumulation), which is used as written.  Every other
step is the chain rule applied to the lines above in reverse order; the
derivative of U is dU(tau)/dtau = Omega U(tau) (see ``basis.omega``).
States are checkpointed every ``ckpt`` tokens and recomputed per segment.

Pins (tests/test_oracle_grad.py): central finite differences of the
independent relative-time forward (``forward.relative_time``) for every
input, at m = 5 and m = 127; the reverse-cumsum identity of the clock.
"""
import numpy as np

from . import basis, gates
from .forward import apply_U, write_vectors


def _softmax(x):
    x = x - np.max(x, axis=-1, keepdims=True)
    e = np.exp(x)
    return e / np.sum(e, axis=-1, keepdims=True)


def backward(q, k, v, clock_logit, decay_logit, beta_logit, A, R, scale, dO,
             lambda0=None, ckpt=64):
    """Gradients of sum(o * dO) for N independent sequences.

    q, k [N,T,dk]; v, dO [N,T,dv]; logits [N,T]; A [N]; R [N,m,m].
    Returns a dict with dq, dk, dv, d_clock, d_decay, d_beta ([N,T]), dR
    [N,m,m], dA [N], plus the intermediate d_lambda, d_delta, d_logalpha,
    d_betaval.
    """
    N, T, dk = q.shape
    dv = v.shape[2]
    m = R.shape[1]
    A = np.asarray(A, dtype=np.float64).reshape(N)
    delta = gates.clock_increment(clock_logit)
    alpha = gates.forget_gate(decay_logit, A[:, None])
    beta = gates.write_strength(beta_logit)
    lam0 = np.zeros(N) if lambda0 is None else np.asarray(lambda0, dtype=np.float64)
    lam = lam0[:, None] + np.cumsum(delta, axis=1)
    a = write_vectors(lam, beta, m)
    phi = basis.fourier_basis(m)
    M = np.einsum('nij,jk->nik', R, phi)
    Om = basis.omega(m)

    # forward sweep: checkpoint the state before every segment
    starts = list(range(0, T, ckpt))
    ck_K, ck_V = [], []
    Kb = np.zeros((N, m, dk))
    Vb = np.zeros((N, m, dv))
    for s0 in starts:
        ck_K.append(Kb.copy())
        ck_V.append(Vb.copy())
        for t in range(s0, min(T, s0 + ckpt)):
            Kb = alpha[:, t, None, None] * Kb + a[:, t, :, None] * k[:, t, None, :]
            Vb = alpha[:, t, None, None] * Vb + a[:, t, :, None] * v[:, t, None, :]

    dq = np.zeros_like(q)
    dkk = np.zeros_like(k)
    dvv = np.zeros_like(v)
    d_lam = np.zeros((N, T))
    d_alpha = np.zeros((N, T))
    d_betaval = np.zeros((N, T))
    dM = np.zeros((N, m, m))
    GK = np.zeros((N, m, dk))       # dL/dKbar_t accumulated from steps >= t
    GV = np.zeros((N, m, dv))
    for si in reversed(range(len(starts))):
        s0 = starts[si]
        s1 = min(T, s0 + ckpt)
        # recompute the states of this segment; Ks[i] is the state after token s0+i-1
        Ks = [ck_K[si]]
        Vs = [ck_V[si]]
        for t in range(s0, s1):
            Ks.append(alpha[:, t, None, None] * Ks[-1] + a[:, t, :, None] * k[:, t, None, :])
            Vs.append(alpha[:, t, None, None] * Vs[-1] + a[:, t, :, None] * v[:, t, None, :])
        for t in reversed(range(s0, s1)):
            Kt, Vt = Ks[t - s0 + 1], Vs[t - s0 + 1]
            Kp, Vp = Ks[t - s0], Vs[t - s0]
            lt = lam[:, t]
            qs = scale * q[:, t]
            o1 = np.einsum('nrd,nd->nr', Kt, qs)
            z = apply_U(lt, o1)
            p = _softmax(np.einsum('nij,nj->ni', M, z))
            y = np.einsum('nij,ni->nj', M, p)
            o2 = apply_U(-lt, y)
            # value pass readout o = Vbar^T o''
            do2 = np.einsum('nrd,nd->nr', Vt, dO[:, t])
            GV = GV + o2[:, :, None] * dO[:, t, None, :]
            # o'' = U(-lam) y
            dy = apply_U(lt, do2)
            d_lam[:, t] -= np.einsum('nr,rs,ns->n', do2, Om, o2)
            # y = M^T p
            dp = np.einsum('nij,nj->ni', M, dy)
            dM += p[:, :, None] * dy[:, None, :]
            # p = softmax(l)
            dl = p * (dp - np.sum(p * dp, axis=1, keepdims=True))
            # l = M z
            dM += dl[:, :, None] * z[:, None, :]
            dz = np.einsum('nij,ni->nj', M, dl)
            # z = U(lam) o'
            d_lam[:, t] += np.einsum('nr,rs,ns->n', dz, Om, z)
            do1 = apply_U(-lt, dz)
            # o' = Kbar q_s
            GK = GK + do1[:, :, None] * qs[:, None, :]
            dq[:, t] = scale * np.einsum('nrd,nr->nd', Kt, do1)
            # Kbar_t = alpha Kbar_{t-1} + a k^T (and V)
            da = np.einsum('nrd,nd->nr', GK, k[:, t]) + np.einsum('nrd,nd->nr', GV, v[:, t])
            dkk[:, t] = np.einsum('nrd,nr->nd', GK, a[:, t])
            dvv[:, t] = np.einsum('nrd,nr->nd', GV, a[:, t])
            d_alpha[:, t] = np.einsum('nrd,nrd->n', GK, Kp) + np.einsum('nrd,nrd->n', GV, Vp)
            # a = beta U(-lam) b
            d_betaval[:, t] = np.sum(da * a[:, t], axis=1) / beta[:, t]
            d_lam[:, t] -= np.einsum('nr,rs,ns->n', da, Om, a[:, t])
            GK = alpha[:, t, None, None] * GK
            GV = alpha[:, t, None, None] * GV

    # Eq. app-clock-gradient-accumulation: dL/d delta_s = sum_{t>=s} dL/d lambda_t
    d_delta = np.cumsum(d_lam[:, ::-1], axis=1)[:, ::-1]
    d_logalpha = alpha * d_alpha
    sp = gates.softplus(decay_logit)
    return {
        'dq': dq, 'dk': dkk, 'dv': dvv,
        'd_clock': d_delta * delta * (1.0 - delta),
        'd_decay': d_logalpha * (-A[:, None] * gates.sigmoid(decay_logit)),
        'd_beta': d_betaval * beta * (1.0 - beta),
        'dR': np.einsum('nij,kj->nik', dM, phi),
        'dA': np.sum(d_logalpha * (-sp), axis=1),
        'd_lambda': d_lam, 'd_delta': d_delta, 'd_logalpha': d_logalpha,
        'd_betaval': d_betaval,
    }
