"""Pins of the oracle's backward against central finite differences.

The finite differences are taken of ``forward.relative_time`` (the defining
recurrence of Sec. 3.1 with the cosine-sum kernel), an independent code path
from the absolute-clock recurrence the backward differentiates.
"""
import numpy as np
import pytest

from oracle import backward as Bk, forward as F, gates as G


def _inputs(N, T, d, m, seed):
    rng = np.random.default_rng(seed)
    return dict(q=rng.standard_normal((N, T, d)), k=rng.standard_normal((N, T, d)),
                v=rng.standard_normal((N, T, d)), c=rng.standard_normal((N, T)),
                f=rng.standard_normal((N, T)), bl=rng.standard_normal((N, T)),
                A=rng.uniform(0.2, 1.0, size=N),
                R=np.eye(m)[None] + 0.3 * rng.standard_normal((N, m, m))), rng.standard_normal((N, T, d))


def _loss(x, dO, s):
    o, _, _ = F.relative_time(x['q'], x['k'], x['v'], G.clock_increment(x['c']),
                              G.forget_gate(x['f'], x['A'][:, None]), G.write_strength(x['bl']),
                              x['R'], s)
    return float(np.sum(o * dO))


NAMES = {'q': 'dq', 'k': 'dk', 'v': 'dv', 'c': 'd_clock', 'f': 'd_decay', 'bl': 'd_beta',
         'A': 'dA', 'R': 'dR'}


@pytest.mark.parametrize('m,T,d,ckpt,entries', [(5, 9, 3, 4, None), (127, 6, 2, 4, 6)])
def test_backward_matches_finite_differences(m, T, d, ckpt, entries):
    x, dO = _inputs(2, T, d, m, seed=m)
    s = 1.3
    g = Bk.backward(x['q'], x['k'], x['v'], x['c'], x['f'], x['bl'], x['A'], x['R'], s, dO,
                    ckpt=ckpt)
    h = 1e-6
    rng = np.random.default_rng(0)
    for nm, gname in NAMES.items():
        arr = x[nm]
        idxs = list(np.ndindex(arr.shape))
        if entries is not None and len(idxs) > entries:
            idxs = [idxs[i] for i in rng.choice(len(idxs), size=entries, replace=False)]
        for idx in idxs:
            xp = {kk: vv.copy() for kk, vv in x.items()}
            xm = {kk: vv.copy() for kk, vv in x.items()}
            xp[nm][idx] += h
            xm[nm][idx] -= h
            fd = (_loss(xp, dO, s) - _loss(xm, dO, s)) / (2 * h)
            assert abs(fd - g[gname][idx]) <= 1e-6 * (1 + abs(fd)), (nm, idx, fd, g[gname][idx])


def test_clock_origin_gradient_vanishes():
    """Prop. 6 makes o independent of a common clock shift, so sum_t dL/d lambda_t = 0."""
    x, dO = _inputs(2, 12, 3, 7, seed=3)
    g = Bk.backward(x['q'], x['k'], x['v'], x['c'], x['f'], x['bl'], x['A'], x['R'], 0.8, dO)
    np.testing.assert_allclose(g['d_lambda'].sum(axis=1), 0.0, atol=1e-10)
    # App. D.1 Eq. app-clock-gradient-accumulation, read back: d_delta_s - d_delta_{s+1} = d_lambda_s
    np.testing.assert_allclose(g['d_delta'][:, :-1] - g['d_delta'][:, 1:], g['d_lambda'][:, :-1],
                               atol=1e-12)


def test_checkpoint_length_does_not_matter():
    x, dO = _inputs(1, 13, 3, 5, seed=4)
    g1 = Bk.backward(x['q'], x['k'], x['v'], x['c'], x['f'], x['bl'], x['A'], x['R'], 1.0, dO, ckpt=1)
    g2 = Bk.backward(x['q'], x['k'], x['v'], x['c'], x['f'], x['bl'], x['A'], x['R'], 1.0, dO, ckpt=64)
    for key in NAMES.values():
        np.testing.assert_allclose(g1[key], g2[key], atol=1e-12)
