"""GPU parity of cyfa_chunk_bwd against the fp64 oracle's reverse-mode gradient."""
import numpy as np
import pytest
import torch

from paper_2609_36259_gb300 import cyfa, synth

from _harness import (assert_close_bf16, assert_close_fp32, assert_close_rel, assert_close_sum,
                      gpu_prepare,
                      oracle_backward,
                      oracle_inputs, pairs_np, sample_pairs, to_device)

pytestmark = pytest.mark.gpu

GRADS = (('dq', 'dq'), ('dk', 'dk'), ('dv', 'dv'), ('d_clock', 'd_clock'),
         ('d_decay', 'd_decay'), ('d_beta', 'd_beta'))


def gpu_backward(d, inp, want_dA=True, use_saved=False, want_dR=False):
    lam, g, beta, _ = gpu_prepare(d, inp)
    q, k, v, dO = inp['q'], inp['k'], inp['v'], inp['dO']
    saved = None
    if use_saved:   # a forward that saves its chunk-start states for this backward
        saved = cyfa.saved_buffer(d, q.device)
        assert saved is not None
        o_plain = cyfa.forward(d, q, k, v, lam, g, beta, inp['R'])[0]
        o_saving = cyfa.forward(d, q, k, v, lam, g, beta, inp['R'], saved=saved)[0]
        assert torch.equal(o_plain, o_saving)   # saving does not change the forward
    out = dict(dq=torch.empty_like(q), dk=torch.empty_like(k), dv=torch.empty_like(v),
               d_clock=torch.empty_like(inp['clock_logit']),
               d_decay=torch.empty_like(inp['clock_logit']),
               d_beta=torch.empty_like(inp['clock_logit']),
               dA=torch.empty_like(inp['A']) if want_dA else None,
               dR=torch.empty_like(inp['R']) if want_dR else None)
    ws = cyfa.workspace(d, cyfa.CYFA_WS_BWD, q.device)
    cyfa.cyfa_chunk_bwd(d, q, k, v, lam, g, beta, inp['R'], inp['clock_logit'],
                        inp['decay_logit'], inp['A'], dO, out['dq'], out['dk'], out['dv'],
                        out['d_clock'], out['d_decay'], out['d_beta'], out['dR'], out['dA'], ws,
                        saved=saved)
    torch.cuda.synchronize()
    return out


def _compare(out, ref, pairs, close, what=''):
    for gk, rk in GRADS:
        close(pairs_np(out[gk].float(), pairs), ref[rk], '%s %s' % (what, gk))


@pytest.mark.parametrize('cuda_cores', [False, True])
@pytest.mark.parametrize('B,T,H,D,C', [(2, 256, 2, 128, 64), (1, 384, 3, 64, 64),
                                       (1, 512, 2, 128, 128), (1, 2304, 2, 128, 64)])
def test_backward_small_bf16(B, T, H, D, C, cuda_cores):
    """Tensor-core kernels (bf16, d = 128, T a multiple of 128) and the CUDA-core kernels;
    T = 2304 spans several 1024-token segments plus a partial one."""
    inp = to_device(synth.make_inputs(B, T, H, D, seed=8, with_dO=True))
    d = cyfa.dims(B, T, H, D, chunk=C, cuda_cores=cuda_cores)
    out = gpu_backward(d, inp, want_dR=True)
    pairs = [(b, h) for b in range(B) for h in range(H)]
    ref = oracle_backward(oracle_inputs(inp, pairs), pairs_np(inp['dO'], pairs))
    _compare(out, ref, pairs, assert_close_bf16)
    dR_ref = np.zeros((H, 127, 127))
    for n, (b, h) in enumerate(pairs):
        dR_ref[h] += ref['dR'][n]
    assert_close_rel(out['dR'].double().cpu().numpy(), dR_ref, 'dR')
    dA_ref, l1 = np.zeros(H), np.zeros(H)
    f = pairs_np(inp['decay_logit'], pairs)
    softplus = np.logaddexp(0.0, f)
    for n, (b, h) in enumerate(pairs):
        dA_ref[h] += ref['dA'][n]
        l1[h] += np.abs(ref['d_logalpha'][n] * softplus[n]).sum()
    assert_close_sum(out['dA'].double().cpu().numpy(), dA_ref, l1, 'dA')


def test_backward_fp32():
    B, T, H, D = 1, 256, 2, 64
    inp = to_device(synth.make_inputs(B, T, H, D, seed=9, with_dO=True, dtype=torch.float32))
    d = cyfa.dims(B, T, H, D, chunk=64, dtype=torch.float32)
    out = gpu_backward(d, inp, want_dR=True)
    pairs = [(0, 0), (0, 1)]
    ref = oracle_backward(oracle_inputs(inp, pairs), pairs_np(inp['dO'], pairs))
    for gk, rk in GRADS:
        got = pairs_np(out[gk], pairs)
        scale = max(1.0, float(np.abs(ref[rk]).max()))
        err = float(np.abs(got - ref[rk]).max())
        assert err <= 1e-4 * scale, (gk, err, scale)
    got = out['dR'].double().cpu().numpy()   # both heads of the single batch row
    scale = max(1.0, float(np.abs(ref['dR']).max()))
    err = float(np.abs(got - ref['dR']).max())
    assert err <= 1e-4 * scale, ('dR', err, scale)


@pytest.mark.parametrize('B,T,H,C,cuda_cores', [(4, 8192, 16, 64, False), (4, 8192, 16, 64, True),
                                                 (2, 32768, 16, 64, False),
                                                 (2, 32768, 16, 128, True)])
def test_backward_full_size_sampled(B, T, H, C, cuda_cores):
    """The B4 H16 T8192 and the 1.4B-shaped B2 H16 T32768 layers: all gradients of sampled
    (b, h) sequences against the oracle."""
    inp = synth.make_inputs(B, T, H, 128, seed=0, device='cuda', with_dO=True)
    d = cyfa.dims(B, T, H, 128, chunk=C, cuda_cores=cuda_cores)
    out = gpu_backward(d, inp, want_dA=False)
    pairs = sample_pairs(B, H, 2)
    ref = oracle_backward(oracle_inputs(inp, pairs), pairs_np(inp['dO'], pairs))
    _compare(out, ref, pairs, assert_close_bf16, 'B%d T%d' % (B, T))


@pytest.mark.parametrize('B,T,H', [(2, 256, 2), (1, 2304, 2), (2, 1152, 3)])
def test_backward_saved_states(B, T, H):
    """The backward reading the forward's saved chunk-start states instead of recomputing them
    (one segment, several segments plus a partial one, odd head count)."""
    inp = to_device(synth.make_inputs(B, T, H, 128, seed=11, with_dO=True))
    d = cyfa.dims(B, T, H, 128, chunk=64)
    out = gpu_backward(d, inp, use_saved=True)
    pairs = [(b, h) for b in range(B) for h in range(H)]
    ref = oracle_backward(oracle_inputs(inp, pairs), pairs_np(inp['dO'], pairs))
    _compare(out, ref, pairs, assert_close_bf16, 'saved')


def test_backward_saved_full_size_sampled():
    """The 1.4B-shaped layer (B2 H16 T32768) with saved states, as the bench step runs it."""
    B, T, H = 2, 32768, 16
    inp = synth.make_inputs(B, T, H, 128, seed=1, device='cuda', with_dO=True)
    d = cyfa.dims(B, T, H, 128, chunk=64)
    out = gpu_backward(d, inp, want_dA=False, use_saved=True)
    pairs = sample_pairs(B, H, 2)
    ref = oracle_backward(oracle_inputs(inp, pairs), pairs_np(inp['dO'], pairs))
    _compare(out, ref, pairs, assert_close_bf16, 'saved full')
