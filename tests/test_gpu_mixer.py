"""The mixer's neighbours (cyfa_mixer_pre / _post and their backward) against oracle/mixer.py,
the autograd wrappers against the C ABI and the oracle, and the mixer module's clock
stop-gradient (Eq. clock_gradient_stabilization)."""
import numpy as np
import pytest
import torch

from oracle import mixer as MX
from paper_2609_36259_gb300 import cyfa, layer, synth

from _harness import (assert_close_bf16, assert_close_fp32, assert_close_rel,
                      assert_close_rounded, oracle_backward, oracle_inputs, pairs_np, rel_l2,
                      to_device)

pytestmark = pytest.mark.gpu

EPS = 1e-6


def _pre_inputs(B, T, H, D, dtype, seed):
    g = torch.Generator().manual_seed(seed)
    x = [torch.randn(B, T, H, D, generator=g).to(dtype).cuda() for _ in range(3)]
    w = [(0.5 * torch.randn(H * D, 4, generator=g)).cuda() for _ in range(3)]
    gains = [(1.0 + 0.1 * torch.randn(D, generator=g)).cuda() for _ in range(2)]
    dy = [torch.randn(B, T, H, D, generator=g).to(dtype).cuda() for _ in range(3)]
    return x, w, gains, dy


def _np(t):
    return t.detach().double().cpu().numpy()


@pytest.mark.parametrize('D,dtype', [(128, torch.bfloat16), (64, torch.float32),
                                     (256, torch.bfloat16), (128, torch.float32)])
def test_mixer_pre_matches_oracle(D, dtype):
    B, T, H = 2, 320, 3     # five 64-token tiles per sequence, several token splits
    x, w, gains, dy = _pre_inputs(B, T, H, D, dtype, seed=51)
    d = cyfa.dims(B, T, H, D, chunk=64, dtype=dtype)
    out = [torch.empty_like(t) for t in x]
    cyfa.cyfa_mixer_pre(d, *x, *w, *gains, EPS, *out)
    dx = [torch.empty_like(t) for t in x]
    dw = [torch.empty_like(t) for t in w]
    dg = [torch.empty_like(t) for t in gains]
    ws = cyfa.workspace(d, cyfa.CYFA_WS_MIXER)
    cyfa.cyfa_mixer_pre_bwd(d, *x, *w, *gains, EPS, *dy, *dx, *dw, *dg, ws)
    cyfa.cyfa_check()
    C = H * D
    xs = [_np(t).reshape(B, T, C) for t in x]
    ws_ = [_np(t) for t in w]
    gs = [_np(t) for t in gains]
    ref = MX.mixer_pre(*xs, *ws_, *gs, EPS, H)
    close = assert_close_rounded if dtype == torch.bfloat16 else assert_close_fp32
    for got, want, nm in zip(out, ref, 'qkv'):
        close(_np(got).reshape(B, T, C), want, 'mixer_pre ' + nm)
    grads = MX.mixer_pre_backward(*xs, *ws_, *gs, EPS, H, *[_np(t).reshape(B, T, C) for t in dy])
    for got, nm in zip(dx, ('dxq', 'dxk', 'dxv')):
        close(_np(got).reshape(B, T, C), grads[nm], nm)
    # parameter gradients are sums over B*T tokens (and heads, for the gains): scale-free bar
    for got, nm in zip(dw + dg, ('dwq', 'dwk', 'dwv', 'dgq', 'dgk')):
        rl = rel_l2(_np(got), grads[nm])
        print('measured %s: rel-L2 %.3e' % (nm, rl))
        assert rl <= (5e-3 if dtype == torch.bfloat16 else 1e-5), (nm, rl)


@pytest.mark.parametrize('D,dtype', [(128, torch.bfloat16), (64, torch.float32),
                                     (256, torch.bfloat16)])
def test_mixer_post_matches_oracle(D, dtype):
    B, T, H = 2, 192, 3
    g = torch.Generator().manual_seed(52)
    o = torch.randn(B, T, H, D, generator=g).to(dtype).cuda()
    z = torch.randn(B, T, H, D, generator=g).to(dtype).cuda()
    gain = (1.0 + 0.1 * torch.randn(D, generator=g)).cuda()
    dy = torch.randn(B, T, H, D, generator=g).to(dtype).cuda()
    d = cyfa.dims(B, T, H, D, chunk=64, dtype=dtype)
    y = torch.empty_like(o)
    cyfa.cyfa_mixer_post(d, o, z, gain, EPS, y)
    d_o, dz, dg = torch.empty_like(o), torch.empty_like(z), torch.empty_like(gain)
    ws = cyfa.workspace(d, cyfa.CYFA_WS_MIXER)
    cyfa.cyfa_mixer_post_bwd(d, o, z, gain, EPS, dy, d_o, dz, dg, ws)
    cyfa.cyfa_check()
    close = assert_close_rounded if dtype == torch.bfloat16 else assert_close_fp32
    close(_np(y), MX.mixer_post(_np(o), _np(z), _np(gain), EPS), 'mixer_post y')
    rdo, rdz, rdg = MX.mixer_post_backward(_np(o), _np(z), _np(gain), EPS, _np(dy))
    close(_np(d_o), rdo, 'do')
    close(_np(dz), rdz, 'dz')
    assert rel_l2(_np(dg), rdg) <= (5e-3 if dtype == torch.bfloat16 else 1e-5)


def test_mixer_full_size():
    """The 1.4B layer's shape (B2 T32768 H16 d128, bf16): pre and post, forward and backward,
    every output against the oracle on two sampled heads; parameter gradients over all heads."""
    B, T, H, D = 2, 32768, 16, 128
    x, w, gains, dy = _pre_inputs(B, T, H, D, torch.bfloat16, seed=53)
    d = cyfa.dims(B, T, H, D, chunk=64)
    out = [torch.empty_like(t) for t in x]
    cyfa.cyfa_mixer_pre(d, *x, *w, *gains, EPS, *out)
    dx = [torch.empty_like(t) for t in x]
    dw = [torch.empty_like(t) for t in w]
    dg = [torch.empty_like(t) for t in gains]
    ws = cyfa.workspace(d, cyfa.CYFA_WS_MIXER)
    cyfa.cyfa_mixer_pre_bwd(d, *x, *w, *gains, EPS, *dy, *dx, *dw, *dg, ws)
    yo = torch.empty_like(x[0])
    cyfa.cyfa_mixer_post(d, x[0], x[1], gains[0], EPS, yo)
    do_, dz, dgo = torch.empty_like(x[0]), torch.empty_like(x[1]), torch.empty_like(gains[0])
    cyfa.cyfa_mixer_post_bwd(d, x[0], x[1], gains[0], EPS, dy[0], do_, dz, dgo, ws)
    cyfa.cyfa_check()
    dg_ref = [np.zeros(D), np.zeros(D)]
    dgo_ref = np.zeros(D)
    for h in range(H):      # one head at a time (fp64 of the whole layer would not fit)
        xs = [_np(t[:, :, h]) for t in x]
        wsl = [_np(t[h * D:(h + 1) * D]) for t in w]
        gs = [_np(t) for t in gains]
        dys = [_np(t[:, :, h]) for t in dy]
        grads = MX.mixer_pre_backward(*xs, *wsl, *gs, EPS, 1, *dys)
        dg_ref[0] += grads['dgq']
        dg_ref[1] += grads['dgk']
        rdo, rdz, rdg = MX.mixer_post_backward(xs[0], xs[1], gs[0], EPS, dys[0])
        dgo_ref += rdg
        for nm, t in zip(('dwq', 'dwk', 'dwv'), dw):
            assert rel_l2(_np(t[h * D:(h + 1) * D]), grads[nm]) <= 5e-3, (h, nm)
        if h in (0, H - 1):
            ref = MX.mixer_pre(*xs, *wsl, *gs, EPS, 1)
            for got, want, nm in zip(out, ref, 'qkv'):
                assert_close_rounded(_np(got[:, :, h]), want, 'full %s head %d' % (nm, h))
            for got, nm in zip(dx, ('dxq', 'dxk', 'dxv')):
                assert_close_rounded(_np(got[:, :, h]), grads[nm], 'full %s head %d' % (nm, h))
            assert_close_rounded(_np(yo[:, :, h]), MX.mixer_post(xs[0], xs[1], gs[0], EPS), 'y')
            assert_close_rounded(_np(do_[:, :, h]), rdo, 'do')
            assert_close_rounded(_np(dz[:, :, h]), rdz, 'dz')
    for got, want, nm in ((dg[0], dg_ref[0], 'dgq'), (dg[1], dg_ref[1], 'dgk'), (dgo, dgo_ref, 'dgo')):
        rl = rel_l2(_np(got), want)
        print('measured full %s: rel-L2 %.3e' % (nm, rl))
        assert rl <= 5e-3, (nm, rl)


@pytest.mark.parametrize('m', [127, 63, 255])
def test_autograd_operator_matches_c_abi_and_oracle(m):
    """CyfaFunction's gradients (through autograd) against the oracle; m = 127 and 63 run the
    tensor-core kernels (with saved states), m = 255 the CUDA-core kernels in 256 storage rows."""
    B, T, H, D = 1, 256, 2, 128
    inp = to_device(synth.make_inputs(B, T, H, D, seed=54, with_dO=True, m=m))
    leaves = {k: inp[k].clone().float().requires_grad_(True) if k in (
        'clock_logit', 'decay_logit', 'beta_logit', 'A', 'R') else inp[k].clone().requires_grad_(True)
        for k in ('q', 'k', 'v', 'clock_logit', 'decay_logit', 'beta_logit', 'A', 'R')}
    o = layer.CyfaFunction.apply(leaves['q'], leaves['k'], leaves['v'], leaves['clock_logit'],
                                 leaves['decay_logit'], leaves['beta_logit'], leaves['A'],
                                 leaves['R'], inp['scale'], 64)
    o.backward(inp['dO'])
    pairs = [(0, h) for h in range(H)]
    oi = oracle_inputs(inp, pairs)
    ref = oracle_backward(oi, pairs_np(inp['dO'], pairs))
    for key, rk in (('q', 'dq'), ('k', 'dk'), ('v', 'dv'), ('clock_logit', 'd_clock'),
                    ('decay_logit', 'd_decay'), ('beta_logit', 'd_beta')):
        assert_close_bf16(pairs_np(leaves[key].grad.float(), pairs), ref[rk], 'autograd ' + key)
    assert leaves['R'].grad.shape == (H, m, m)
    assert_close_rel(_np(leaves['R'].grad), ref['dR'], 'autograd dR')


def test_mixer_module_clock_stop_gradient():
    """The clock path trains W_delta (its gradient is sum_t d_clock_t x_t^T) but sends nothing
    into x: x.grad equals that of the same mixer with the clock logits precomputed as constants."""
    torch.manual_seed(0)
    mix = layer.CyfaMixer(64, 2, 128, chunk=64)
    x = torch.randn(1, 256, 64, device='cuda')
    x1 = x.clone().requires_grad_(True)
    y = mix(x1)
    dy = torch.randn_like(y)
    y.backward(dy)
    gx = x1.grad.clone()
    gw = mix.w_clock.weight.grad.clone()
    assert torch.isfinite(gx).all() and gw.abs().sum() > 0
    # the same forward with the clock logits as constants of the graph
    mix.zero_grad()
    clock_const = mix.w_clock(x).detach()
    orig = mix.w_clock.forward
    mix.w_clock.forward = lambda inp: clock_const
    x2 = x.clone().requires_grad_(True)
    mix(x2).backward(dy)
    mix.w_clock.forward = orig
    assert torch.allclose(x2.grad, gx, rtol=1e-5, atol=1e-7)
    # W_delta's gradient from the operator's d_clock_logit: recompute d_clock with autograd
    mix.zero_grad()
    x3 = x.clone().requires_grad_(True)
    clk = mix.w_clock(x3.detach())
    clk.retain_grad()
    saved = mix.w_clock.forward
    mix.w_clock.forward = lambda inp: clk
    mix(x3).backward(dy)
    mix.w_clock.forward = saved
    want = torch.einsum('bth,btc->hc', clk.grad, x)
    assert torch.allclose(gw, want, rtol=1e-4, atol=1e-5)
