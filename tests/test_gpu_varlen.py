"""Packed variable-length sequences (cyfa_prepare_varlen) and the fixed-rate clock
(cyfa_prepare_fixed_rate), through the C ABI, against the fp64 oracle run on every sequence on
its own (App. A, Fixed-Rate Specialization; App. B chunk form with per-sequence zero states).

Sequence j occupies tokens [cu[j], cu[j+1]) of a [1, T, H, d] stream; the oracle sees it as a
separate (b, h) sequence with zero initial states and its own clock origin lambda0[j].
"""
import math

import numpy as np
import pytest
import torch

from oracle import backward as OB, basis, forward as OF, gates as OG
from paper_2609_36259_gb300 import cyfa, synth

from _harness import (BF16_MAX_ABS, assert_close_batch_sum, assert_close_bf16, assert_close_fp32,
                      assert_close_rel, rel_l2, to_device)

pytestmark = pytest.mark.gpu

M = 127
SEQ_KEYS = ('q', 'k', 'v', 'clock_logit', 'decay_logit', 'beta_logit', 'dO')


def _seq(x, c0, c1, h):
    """Tokens [c0, c1) of head h of a [1, T, H, ...] tensor as float64 numpy [1, L, ...]."""
    return x[0, c0:c1, h].detach().to('cpu', torch.float64).numpy()[None]


def _oracle_seq(inp, c0, c1, h, lam0, rho=None, dO=None):
    """The oracle's forward (and backward with dO) of one sequence of one head."""
    q, k, v = (_seq(inp[n], c0, c1, h) for n in ('q', 'k', 'v'))
    f, bl = _seq(inp['decay_logit'], c0, c1, h), _seq(inp['beta_logit'], c0, c1, h)
    if rho is None:
        c = _seq(inp['clock_logit'], c0, c1, h)
        delta = OG.clock_increment(c)
    else:   # delta = 1/rho exactly; as a logit, -ln(rho - 1) (+inf at rho = 1)
        delta = np.full(f.shape, 1.0 / rho)
        c = np.full(f.shape, -math.log(rho - 1.0) if rho > 1.0 else np.inf)
    A = inp['A'].double().cpu().numpy()[[h]]
    R = inp['R'].double().cpu().numpy()[[h]]
    alpha = OG.forget_gate(f, A[:, None])
    beta = OG.write_strength(bl)
    o, Kb, Vb, lamT = OF.absolute_clock(q, k, v, delta, alpha, beta, R, inp['scale'],
                                        lambda0=np.array([lam0]))
    grads = None
    if dO is not None:
        grads = OB.backward(q, k, v, c, f, bl, A, R, inp['scale'], _seq(dO, c0, c1, h),
                            lambda0=np.array([lam0]))
    return o[0], Kb[0], Vb[0], lamT[0], grads


def _packed(lengths, H, D, seed, dtype=torch.bfloat16, with_dO=True):
    T = int(sum(lengths))
    inp = to_device(synth.make_inputs(1, T, H, D, seed=seed, dtype=dtype, with_dO=with_dO))
    cu = torch.tensor(np.concatenate([[0], np.cumsum(lengths)]), dtype=torch.int32, device='cuda')
    lam0 = torch.tensor([[3.25 * j + 0.5 * h for h in range(H)] for j in range(len(lengths))],
                        dtype=torch.float64, device='cuda')
    return inp, cu, lam0, T


def _backward(d, inp, lam, g, beta, fixed, saved=None):
    q, k, v = inp['q'], inp['k'], inp['v']
    out = dict(dq=torch.empty_like(q), dk=torch.empty_like(k), dv=torch.empty_like(v),
               d_clock=None if fixed else torch.empty_like(lam), d_decay=torch.empty_like(lam),
               d_beta=torch.empty_like(lam), dA=torch.empty_like(inp['A']),
               dR=torch.empty_like(inp['R']))
    ws = cyfa.workspace(d, cyfa.CYFA_WS_BWD, q.device)
    cyfa.cyfa_chunk_bwd(d, q, k, v, lam, g, beta, inp['R'], None if fixed else inp['clock_logit'],
                        inp['decay_logit'], inp['A'], inp['dO'], out['dq'], out['dk'], out['dv'],
                        out['d_clock'], out['d_decay'], out['d_beta'], out['dR'], out['dA'], ws,
                        saved=saved)
    return out


LENGTHS_BF16 = [1, 0, 37, 128, 300, 5, 0, 203, 350]      # 1024 tokens: ragged, empty, length 1
LENGTHS_FP32 = [10, 0, 100, 1, 145]                       # 256 tokens


@pytest.mark.parametrize('fixed_rho', [None, 2.5])
@pytest.mark.parametrize('dtype,cuda_cores', [(torch.bfloat16, False), (torch.bfloat16, True),
                                              (torch.float32, True)])
def test_varlen_forward_backward(dtype, cuda_cores, fixed_rho):
    """Every output, clock and gradient of every packed sequence against the oracle run on that
    sequence alone; dA and dR against the sums over the sequences."""
    H = 2
    D = 128 if dtype == torch.bfloat16 else 64
    lengths = LENGTHS_BF16 if dtype == torch.bfloat16 else LENGTHS_FP32
    inp, cu, lam0, T = _packed(lengths, H, D, seed=31, dtype=dtype)
    d = cyfa.dims(1, T, H, D, chunk=64, dtype=dtype, cuda_cores=cuda_cores)
    fixed = fixed_rho is not None
    lam, g, beta, lend = cyfa.prepare_varlen(d, cu, inp['decay_logit'], inp['beta_logit'],
                                             inp['A'], None if fixed else inp['clock_logit'],
                                             fixed_rho or 0.0, lambda0=lam0, want_lambda_end=True)
    o, Ko, Vo = cyfa.forward(d, inp['q'], inp['k'], inp['v'], lam, g, beta, inp['R'],
                             want_state=True)
    out = _backward(d, inp, lam, g, beta, fixed)
    cyfa.cyfa_check()
    cuh = cu.cpu().numpy()
    want = {k: np.zeros((T, H) + ((D,) if k in ('o', 'dq', 'dk', 'dv') else ()))
            for k in ('o', 'dq', 'dk', 'dv', 'd_clock', 'd_decay', 'd_beta')}
    dA_ref, dR_ref = np.zeros(H), np.zeros((H, M, M))
    terms = [[] for _ in range(H)]
    last = None
    for j in range(len(lengths)):
        c0, c1 = int(cuh[j]), int(cuh[j + 1])
        for h in range(H):
            l0 = float(lam0[j, h])
            if c1 == c0:   # an empty sequence keeps its clock origin
                assert float(lend[j, h]) == l0
                continue
            o_r, Kb, Vb, lamT, gr = _oracle_seq(inp, c0, c1, h, l0, fixed_rho, inp['dO'])
            want['o'][c0:c1, h] = o_r
            for key in ('dq', 'dk', 'dv', 'd_clock', 'd_decay', 'd_beta'):
                want[key][c0:c1, h] = gr[key][0]
            dA_ref[h] += gr['dA'][0]
            f = _seq(inp['decay_logit'], c0, c1, h)[0]
            terms[h].append(-np.logaddexp(0.0, f) * gr['d_logalpha'][0])
            dR_ref[h] += gr['dR'][0]
            assert abs(float(lend[j, h]) - lamT) < 1e-6 + 4e-9 * (c1 - c0), (j, h)
            if c1 == T:
                last = last or {}
                last[h] = (Kb, Vb)
    close = assert_close_bf16 if dtype == torch.bfloat16 else assert_close_fp32
    close(o[0].double().cpu().numpy(), want['o'], 'o')
    for key in ('dq', 'dk', 'dv', 'd_decay', 'd_beta') + (() if fixed else ('d_clock',)):
        close(out[key][0].double().cpu().numpy(), want[key], key)
    # the last sequence's final states
    for h in range(H):
        close(Ko[0, h, :M].double().cpu().numpy(), last[h][0], 'Kbar_out')
        close(Vo[0, h, :M].double().cpu().numpy(), last[h][1], 'Vbar_out')
    dA = out['dA'].double().cpu().numpy()
    if dtype == torch.bfloat16:
        assert_close_batch_sum(dA, dA_ref, [np.concatenate(t) for t in terms], 'dA')
        assert_close_rel(out['dR'].double().cpu().numpy(), dR_ref, 'dR')
    else:
        assert rel_l2(dA, dA_ref) <= 1e-4, (dA, dA_ref)
        assert rel_l2(out['dR'].double().cpu().numpy(), dR_ref) <= 1e-4


def test_varlen_of_equal_lengths_is_the_batch():
    """Packing B equal-length sequences gives the batched call's results (clock origin 0)."""
    B, Tb, H, D = 3, 256, 2, 128
    inp = to_device(synth.make_inputs(B, Tb, H, D, seed=33))
    d = cyfa.dims(B, Tb, H, D, chunk=64)
    lam, g, beta, _ = cyfa.prepare(d, inp['clock_logit'], inp['decay_logit'],
                                   inp['beta_logit'], inp['A'])
    o_batch = cyfa.forward(d, inp['q'], inp['k'], inp['v'], lam, g, beta, inp['R'])[0]
    flat = {k: (v.reshape(1, B * Tb, *v.shape[2:]) if k in SEQ_KEYS else v)
            for k, v in inp.items()}
    cu = torch.arange(0, B * Tb + 1, Tb, dtype=torch.int32, device='cuda')
    dp = cyfa.dims(1, B * Tb, H, D, chunk=64)
    lam2, g2, beta2, _ = cyfa.prepare_varlen(dp, cu, flat['decay_logit'], flat['beta_logit'],
                                             flat['A'], flat['clock_logit'])
    o_pack = cyfa.forward(dp, flat['q'], flat['k'], flat['v'], lam2, g2, beta2, flat['R'])[0]
    cyfa.cyfa_check()
    # the clock and the chunk-local log-decays of the first sequence are those of the batch call
    np.testing.assert_allclose(lam2[0, :Tb].cpu().numpy(), lam[0].cpu().numpy(), atol=1e-5)
    np.testing.assert_allclose(g2[0, :Tb].cpu().numpy(), g[0].cpu().numpy(), atol=1e-6)
    # the fp32 results agree far more closely; a bf16 rounding may still land one unit apart
    err = (o_pack.reshape(B, Tb, H, D).float() - o_batch.float()).abs().max().item()
    assert err <= BF16_MAX_ABS, err


def test_varlen_rejects_bad_offsets():
    """Offsets that do not cover [0, T] in order are reported by cyfa_check as CYFA_ERR_ARG."""
    H, D, T = 1, 128, 256
    inp = to_device(synth.make_inputs(1, T, H, D, seed=34))
    d = cyfa.dims(1, T, H, D, chunk=64)
    for bad in ([0, 100, 50, 256], [0, 100, 200], [5, 100, 256]):
        cu = torch.tensor(bad, dtype=torch.int32, device='cuda')
        cyfa.prepare_varlen(d, cu, inp['decay_logit'], inp['beta_logit'], inp['A'],
                            inp['clock_logit'])
        with pytest.raises(cyfa.CyfaError) as e:
            cyfa.cyfa_check()
        assert e.value.code == cyfa.CYFA_ERR_ARG, bad
    cu = torch.tensor([0, 100, 256], dtype=torch.int32, device='cuda')   # valid again
    cyfa.prepare_varlen(d, cu, inp['decay_logit'], inp['beta_logit'], inp['A'],
                        inp['clock_logit'])
    cyfa.cyfa_check()


@pytest.mark.parametrize('rho', [1.0, 2.5, 7.0])
@pytest.mark.parametrize('cuda_cores', [False, True])
def test_fixed_rate_matches_oracle(rho, cuda_cores):
    """cyfa_prepare_fixed_rate + chunk calls against the oracle with delta = 1/rho: clock,
    outputs and every gradient (no clock gradient)."""
    B, T, H, D = 2, 384, 2, 128
    inp = to_device(synth.make_inputs(B, T, H, D, seed=35, with_dO=True))
    d = cyfa.dims(B, T, H, D, chunk=64, cuda_cores=cuda_cores)
    lam0 = torch.tensor([[1.5, 40.0], [100.25, 0.0]], dtype=torch.float64, device='cuda')
    lam, g, beta, lend = cyfa.prepare_fixed_rate(d, rho, inp['decay_logit'], inp['beta_logit'],
                                                 inp['A'], lambda0=lam0, want_lambda_end=True)
    o = cyfa.forward(d, inp['q'], inp['k'], inp['v'], lam, g, beta, inp['R'])[0]
    out = _backward(d, inp, lam, g, beta, True)
    cyfa.cyfa_check()
    for b in range(B):
        for h in range(H):
            one = {k: (v[b:b + 1] if k in SEQ_KEYS else v) for k, v in inp.items()}
            o_r, _, _, lamT, gr = _oracle_seq(one, 0, T, h, float(lam0[b, h]), rho, one['dO'])
            want_lam = np.mod(float(lam0[b, h]) + np.arange(1, T + 1) / rho, M)
            got_lam = lam[b, :, h].double().cpu().numpy()
            dist = np.abs(got_lam - want_lam)
            assert np.minimum(dist, M - dist).max() < 2e-5
            assert abs(float(lend[b, h]) - lamT) < 1e-9
            assert_close_bf16(o[b, :, h].double().cpu().numpy(), o_r, 'o')
            for key in ('dq', 'dk', 'dv', 'd_decay', 'd_beta'):
                assert_close_bf16(out[key][b, :, h].double().cpu().numpy(), gr[key][0], key)


def test_fixed_rate_state_is_the_dirichlet_profile():
    """With alpha = beta = 1 the relative-time key state after T tokens of a fixed-rate clock is
    sum_i P((T - i)/rho) e_0 k_i^T, whose entries are the Fourier-Dirichlet profile of Eq.
    app-constant-rate-profile; the library exports the absolute-clock state Kbar, and Phi
    U(lambda_T) Kbar is that relative-time state (Sec. 3.2)."""
    T, H, D, rho = 256, 1, 64, 3.0
    inp = to_device(synth.make_inputs(1, T, H, D, seed=36, dtype=torch.float32))
    inp['decay_logit'].fill_(-float('inf'))    # softplus = 0: alpha = 1
    inp['beta_logit'].fill_(float('inf'))      # beta = 1
    d = cyfa.dims(1, T, H, D, chunk=64, dtype=torch.float32)
    lam, g, beta, lend = cyfa.prepare_fixed_rate(d, rho, inp['decay_logit'], inp['beta_logit'],
                                                 inp['A'], want_lambda_end=True)
    _, Ko, _ = cyfa.forward(d, inp['q'], inp['k'], inp['v'], lam, g, beta, inp['R'],
                            want_state=True)
    cyfa.cyfa_check()
    Kb = Ko[0, 0, :M].double().cpu().numpy()
    K_rel = basis.fourier_basis(M) @ basis.U(T / rho, M) @ Kb
    k = inp['k'][0, :, 0].double().cpu().numpy()
    r = np.arange(M)
    hh = np.arange(1, (M - 1) // 2 + 1)[:, None, None]
    i = np.arange(1, T + 1)[None, :, None]
    prof = (1 + 2 * np.cos(2 * np.pi * hh * ((T - i) - rho * r[None, None, :]) / (rho * M))
            .sum(0)) / M                                            # [T, m]
    want = prof.T @ k                                               # [m, D]
    err = np.abs(K_rel - want).max() / max(1.0, np.abs(want).max())
    assert err < 1e-4, err


def test_varlen_full_size_sampled():
    """The 1.4B-shaped layer's 65,536 tokens (H16 d128) as one packed stream of sequences of
    mixed length around 2,048 tokens (the paper's training context), forward and backward in one
    call each; sampled (sequence, head) pairs, the first and the last sequence among them, against
    the oracle run on each alone."""
    H, D = 16, 128
    lengths = synth.varlen_lengths(65536, 2048, seed=3)
    inp, cu, lam0, T = _packed(lengths, H, D, seed=37)
    d = cyfa.dims(1, T, H, D, chunk=64)
    lam, g, beta, lend = cyfa.prepare_varlen(d, cu, inp['decay_logit'], inp['beta_logit'],
                                             inp['A'], inp['clock_logit'], lambda0=lam0,
                                             want_lambda_end=True)
    saved = cyfa.saved_buffer(d, inp['q'].device)
    o = cyfa.forward(d, inp['q'], inp['k'], inp['v'], lam, g, beta, inp['R'], saved=saved)[0]
    out = _backward(d, inp, lam, g, beta, False, saved=saved)
    cyfa.cyfa_check()
    cuh = cu.cpu().numpy()
    n = len(lengths)
    picks = [(0, 0), (n // 2, 7), (n - 1, H - 1)]
    for j, h in picks:
        c0, c1 = int(cuh[j]), int(cuh[j + 1])
        o_r, _, _, lamT, gr = _oracle_seq(inp, c0, c1, h, float(lam0[j, h]), None, inp['dO'])
        what = 'seq %d (%d tokens) head %d' % (j, c1 - c0, h)
        assert_close_bf16(o[0, c0:c1, h].double().cpu().numpy(), o_r, what + ' o')
        for key in ('dq', 'dk', 'dv', 'd_clock', 'd_decay', 'd_beta'):
            assert_close_bf16(out[key][0, c0:c1, h].double().cpu().numpy(), gr[key][0],
                              what + ' ' + key)
        assert abs(float(lend[j, h]) - lamT) < 1e-6 + 4e-9 * (c1 - c0)
