"""GPU parity of cyfa_chunk_bwd against the fp64 oracle's reverse-mode gradient."""
import numpy as np
import pytest
import torch

from paper_2609_36259_gb300 import cyfa, synth

from _harness import (CLOCK_FAST_HEAD_REL_L2, Guards, assert_close_batch_sum, assert_close_bf16,
                      assert_close_rel, gpu_prepare, oracle_backward, oracle_inputs, pairs_np,
                      rel_l2, sample_pairs, to_device)

pytestmark = pytest.mark.gpu

GRADS = (('dq', 'dq'), ('dk', 'dk'), ('dv', 'dv'), ('d_clock', 'd_clock'),
         ('d_decay', 'd_decay'), ('d_beta', 'd_beta'))


def gpu_backward(d, inp, want_dA=True, use_saved=False, want_dR=False):
    lam, g, beta, _ = gpu_prepare(d, inp)
    q, k, v, dO = inp['q'], inp['k'], inp['v'], inp['dO']
    saved = None
    if use_saved:   # a forward that saves its chunk-start states for this backward
        n = cyfa.cyfa_saved_size(d)
        assert n > 0
        sg = Guards()
        saved = sg.empty((n,), torch.uint8, q.device)
        o_plain = cyfa.forward(d, q, k, v, lam, g, beta, inp['R'])[0]
        o_saving = cyfa.forward(d, q, k, v, lam, g, beta, inp['R'], saved=saved)[0]
        assert torch.equal(o_plain, o_saving)   # saving does not change the forward
        sg.check('cyfa_chunk_fwd saved states')
    gd = Guards()
    out = dict(dq=gd.empty_like(q), dk=gd.empty_like(k), dv=gd.empty_like(v),
               d_clock=gd.empty_like(inp['clock_logit']),
               d_decay=gd.empty_like(inp['clock_logit']),
               d_beta=gd.empty_like(inp['clock_logit']),
               dA=gd.empty_like(inp['A']) if want_dA else None,
               dR=gd.empty_like(inp['R']) if want_dR else None)
    ws = cyfa.workspace(d, cyfa.CYFA_WS_BWD, q.device)
    cyfa.cyfa_chunk_bwd(d, q, k, v, lam, g, beta, inp['R'], inp['clock_logit'],
                        inp['decay_logit'], inp['A'], dO, out['dq'], out['dk'], out['dv'],
                        out['d_clock'], out['d_decay'], out['d_beta'], out['dR'], out['dA'], ws,
                        saved=saved)
    gd.check('cyfa_chunk_bwd')
    return out


def _compare(out, ref, pairs, close, what='', clock_rel=None):
    for gk, rk in GRADS:
        if gk == 'd_clock' and clock_rel is not None:
            close(pairs_np(out[gk].float(), pairs), ref[rk], '%s %s' % (what, gk), rel_bar=clock_rel)
        else:
            close(pairs_np(out[gk].float(), pairs), ref[rk], '%s %s' % (what, gk))
    # the decay gradient of each head on its own (A_h scales it by up to 256x between heads)
    got = pairs_np(out['d_decay'].float(), pairs)
    for h in sorted({h for _, h in pairs}):
        idx = [n for n, (_, hh) in enumerate(pairs) if hh == h]
        print('measured %s d_decay head %d: rel-L2 %.3e'
              % (what, h, rel_l2(got[idx], ref['d_decay'][idx])))


def _dA_terms(inp, ref, pairs, H):
    """The oracle's dA per head and its terms w_t d log alpha_t (w_t = -softplus(f_t))."""
    f = pairs_np(inp['decay_logit'], pairs)
    dA_ref = np.zeros(H)
    terms = [[] for _ in range(H)]
    for n, (b, h) in enumerate(pairs):
        dA_ref[h] += ref['dA'][n]
        terms[h].append(-np.logaddexp(0.0, f[n]) * ref['d_logalpha'][n])
    return dA_ref, [np.concatenate(t) if t else np.zeros(1) for t in terms]


@pytest.mark.parametrize('cuda_cores', [False, True])
@pytest.mark.parametrize('B,T,H,D,C', [(2, 256, 2, 128, 64), (1, 384, 3, 64, 64),
                                       (1, 512, 2, 128, 128), (1, 2304, 2, 128, 64),
                                       (1, 256, 2, 256, 64), (1, 64, 1, 128, 64),
                                       (1, 128, 1, 128, 128)])
def test_backward_small_bf16(B, T, H, D, C, cuda_cores):
    """Tensor-core kernels (bf16, d = 128, T a multiple of 128) and the CUDA-core kernels;
    T = 2304 spans several 1024-token segments plus a partial one; B = H = 1 with a single chunk
    (T = C = 64 on the CUDA-core kernels, T = C = 128 on both)."""
    inp = to_device(synth.make_inputs(B, T, H, D, seed=8, with_dO=True))
    d = cyfa.dims(B, T, H, D, chunk=C, cuda_cores=cuda_cores)
    out = gpu_backward(d, inp, want_dR=True)
    pairs = [(b, h) for b in range(B) for h in range(H)]
    ref = oracle_backward(oracle_inputs(inp, pairs), pairs_np(inp['dO'], pairs))
    # one head only (A = 1, the fast-decay head) on the tensor-core kernels: the d_clock reading
    tc_fast = H == 1 and not cuda_cores and D == 128 and T % 128 == 0
    _compare(out, ref, pairs, assert_close_bf16,
             clock_rel=CLOCK_FAST_HEAD_REL_L2 if tc_fast else None)
    dR_ref = np.zeros((H, 127, 127))
    for n, (b, h) in enumerate(pairs):
        dR_ref[h] += ref['dR'][n]
    assert_close_rel(out['dR'].double().cpu().numpy(), dR_ref, 'dR')
    dA_ref, terms = _dA_terms(inp, ref, pairs, H)
    assert_close_batch_sum(out['dA'].double().cpu().numpy(), dA_ref, terms, 'dA')


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
    pairs = sample_pairs(B, H, 4)
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


@pytest.mark.parametrize('dtype,D,cuda_cores', [(torch.float32, 64, True),
                                                (torch.bfloat16, 256, False),
                                                (torch.bfloat16, 128, True)])
def test_backward_saved_states_cuda_cores(dtype, D, cuda_cores):
    """The CUDA-core backward reading the forward's fp32 chunk-start states (64-token chunks)
    gives bit-identical gradients to the one that recomputes them (the same state pass computes
    them either way)."""
    B, T, H = 2, 512, 2
    inp = to_device(synth.make_inputs(B, T, H, D, seed=13, dtype=dtype, with_dO=True))
    d = cyfa.dims(B, T, H, D, chunk=64, dtype=dtype, cuda_cores=cuda_cores)
    assert cyfa.cyfa_saved_size(d) == B * H * (T // 64) * 128 * 2 * D * 4
    got = gpu_backward(d, inp, use_saved=True, want_dR=True)
    want = gpu_backward(d, inp, want_dR=True)
    for k, t in want.items():
        assert torch.equal(got[k], t), k


def test_backward_saved_full_size_sampled():
    """The 1.4B-shaped layer (B2 H16 T32768) with saved states, as the bench step runs it."""
    B, T, H = 2, 32768, 16
    inp = synth.make_inputs(B, T, H, 128, seed=1, device='cuda', with_dO=True)
    d = cyfa.dims(B, T, H, 128, chunk=64)
    out = gpu_backward(d, inp, want_dA=False, use_saved=True)
    pairs = sample_pairs(B, H, 4)
    ref = oracle_backward(oracle_inputs(inp, pairs), pairs_np(inp['dO'], pairs))
    _compare(out, ref, pairs, assert_close_bf16, 'saved full')


@pytest.mark.parametrize('B,T,H,saved', [(4, 8192, 16, False), (2, 32768, 16, True)])
def test_backward_full_size_dA_dR(B, T, H, saved):
    """dA and dR at full size, in the launch configuration the bench step uses (dR requested,
    saved states on the 1.4B layer).  Both are sums over the batch, so the upstream gradient is
    kept on a few sampled (b, h) sequences and zeroed on every other one: the others then add
    exactly zero to every gradient, and dA[h], dR[h] equal the oracle's sums over the sampled
    sequences of head h (heads without a sampled sequence must come out zero)."""
    inp = synth.make_inputs(B, T, H, 128, seed=3, device='cuda', with_dO=True)
    pairs = sample_pairs(B, H, 3, seed=5)
    keep = torch.zeros(B, 1, H, 1, device='cuda')
    for b, h in pairs:
        keep[b, 0, h, 0] = 1.0
    inp['dO'] = (inp['dO'].float() * keep).to(inp['dO'].dtype)
    d = cyfa.dims(B, T, H, 128, chunk=64)
    out = gpu_backward(d, inp, want_dA=True, use_saved=saved, want_dR=True)
    ref = oracle_backward(oracle_inputs(inp, pairs), pairs_np(inp['dO'], pairs))
    _compare(out, ref, pairs, assert_close_bf16, 'masked dO B%d T%d' % (B, T))
    dR_ref = np.zeros((H, 127, 127))
    for n, (b, h) in enumerate(pairs):
        dR_ref[h] += ref['dR'][n]
    dA_ref, terms = _dA_terms(inp, ref, pairs, H)
    hs = sorted({h for _, h in pairs})
    dA = out['dA'].double().cpu().numpy()
    dR = out['dR'].double().cpu().numpy()
    assert_close_batch_sum(dA[hs], dA_ref[hs], [terms[h] for h in hs], 'dA')
    assert_close_rel(dR[hs], dR_ref[hs], 'dR')
    others = [h for h in range(H) if h not in hs]
    assert np.all(dA[others] == 0) and np.all(dR[others] == 0)


def test_backward_paper_kernel_shape_sampled():
    """The paper's kernel-latency shape (H = 4, d_k = d_v = 256, T = 2048, B = 32): all
    gradients of sampled (b, h) sequences against the oracle."""
    B, T, H = 32, 2048, 4
    inp = synth.make_inputs(B, T, H, 256, seed=0, device='cuda', with_dO=True)
    d = cyfa.dims(B, T, H, 256, chunk=64)
    out = gpu_backward(d, inp, want_dA=False)
    pairs = sample_pairs(B, H, 3)
    ref = oracle_backward(oracle_inputs(inp, pairs), pairs_np(inp['dO'], pairs))
    _compare(out, ref, pairs, assert_close_bf16, 'paper shape')


def test_backward_from_fresh_thread():
    """The backward called from a thread whose first CUDA work it is (as in an autograd worker
    thread), reading the forward's saved states: it starts with tensor-map encodes, driver calls
    that need the device's context current in that thread.  The gradients equal those of the
    same call made from the main thread."""
    import threading
    B, T, H, D = 1, 256, 2, 128
    inp = to_device(synth.make_inputs(B, T, H, D, seed=57, with_dO=True))
    d = cyfa.dims(B, T, H, D, chunk=64)
    lam, g, beta, _ = gpu_prepare(d, inp)
    saved = cyfa.saved_buffer(d)
    cyfa.forward(d, inp['q'], inp['k'], inp['v'], lam, g, beta, inp['R'], saved=saved)
    st = torch.cuda.Stream()
    ws = [cyfa.workspace(d, cyfa.CYFA_WS_BWD) for _ in range(2)]

    def outputs():
        return dict(dq=torch.empty_like(inp['q']), dk=torch.empty_like(inp['k']),
                    dv=torch.empty_like(inp['v']), dc=torch.empty_like(lam),
                    dd=torch.empty_like(lam), db=torch.empty_like(lam),
                    dR=torch.empty_like(inp['R']), dA=torch.empty_like(inp['A']))
    outs = [outputs(), outputs()]
    torch.cuda.synchronize()

    def bwd(i):
        o = outs[i]
        cyfa.cyfa_chunk_bwd(d, inp['q'], inp['k'], inp['v'], lam, g, beta, inp['R'],
                            inp['clock_logit'], inp['decay_logit'], inp['A'], inp['dO'], o['dq'],
                            o['dk'], o['dv'], o['dc'], o['dd'], o['db'], o['dR'], o['dA'], ws[i],
                            stream=st, saved=saved)
    errors = []

    def worker():
        try:
            bwd(0)
        except Exception as e:   # reported below, in the test's own thread
            errors.append(e)
    t = threading.Thread(target=worker)
    t.start()
    t.join()
    assert not errors, errors
    bwd(1)
    st.synchronize()
    cyfa.cyfa_check(st)
    for k in outs[0]:
        assert torch.equal(outs[0][k], outs[1][k]), k
