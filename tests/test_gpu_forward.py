"""GPU parity of cyfa_prepare and cyfa_chunk_fwd against the fp64 oracle (through the C ABI)."""
import numpy as np
import pytest
import torch

from oracle import gates as OG
from paper_2609_36259_gb300 import cyfa, synth

from _harness import (assert_close_bf16, assert_close_fp32, gpu_forward, gpu_prepare,
                      oracle_forward, oracle_inputs, pairs_np, sample_pairs, to_device)

pytestmark = pytest.mark.gpu


def _chunk_local_logdecay(f, A, C):
    """App. B: gamma^r within each chunk as a cumulative sum of log alpha (fp64)."""
    la = np.log(OG.forget_gate(f, A[:, None]))
    N, T = la.shape
    return np.cumsum(la.reshape(N, T // C, C), axis=2).reshape(N, T)


@pytest.mark.parametrize('B,T,H,C', [(2, 1088, 3, 64), (1, 2048, 2, 128), (2, 32768, 2, 128)])
def test_prepare_matches_oracle(B, T, H, C):
    inp = to_device(synth.make_inputs(B, T, H, 64, seed=1))
    d = cyfa.dims(B, T, H, 64, chunk=C)
    lam0 = torch.tensor([[0.25 + 3 * b + h for h in range(H)] for b in range(B)],
                        dtype=torch.float64, device='cuda')
    lam, g, beta, lend = gpu_prepare(d, inp, lambda0=lam0, want_lambda_end=True)
    torch.cuda.synchronize()
    pairs = [(b, h) for b in range(B) for h in range(H)]
    c = pairs_np(inp['clock_logit'], pairs)
    f = pairs_np(inp['decay_logit'], pairs)
    bl = pairs_np(inp['beta_logit'], pairs)
    A = inp['A'].double().cpu().numpy()[[h for _, h in pairs]]
    l0 = np.array([lam0[b, h].item() for b, h in pairs])
    lam_ref = OG.cumulative_clock(OG.clock_increment(c), l0[:, None], axis=1)
    got_lam = pairs_np(lam, pairs)
    dist = np.abs(got_lam - np.mod(lam_ref, 127.0))
    dist = np.minimum(dist, 127.0 - dist)            # compare on the circle of period m
    # delta = sigmoid(logit) is formed in fp32 (rounding <= 2^-25 per token, with a small mean
    # bias) and summed in fp64, so the clock may drift by up to ~T * 2^-28 from the fp64 oracle.
    lam_tol = 1e-6 + 4e-9 * T
    assert dist.max() < lam_tol, dist.max()
    np.testing.assert_allclose(pairs_np(g, pairs), _chunk_local_logdecay(f, A, C), rtol=1e-5,
                               atol=2e-5)
    np.testing.assert_allclose(pairs_np(beta, pairs), OG.write_strength(bl), rtol=1e-6, atol=1e-7)
    lend_got = np.array([lend[b, h].item() for b, h in pairs])
    np.testing.assert_allclose(lend_got, lam_ref[:, -1], rtol=0, atol=lam_tol)


def test_fp32_config_parity():
    """fp32 forward, B=1 H=2 T=256 d=64 chunk 64: every output within 1e-4 of the oracle."""
    inp = to_device(synth.make_inputs(1, 256, 2, 64, seed=0, dtype=torch.float32))
    d = cyfa.dims(1, 256, 2, 64, chunk=64, dtype=torch.float32)
    o, Ko, Vo, _ = gpu_forward(d, inp, want_state=True)
    pairs = [(0, 0), (0, 1)]
    oi = oracle_inputs(inp, pairs)
    o_ref, Kb, Vb, _ = oracle_forward(oi)
    assert_close_fp32(pairs_np(o, pairs), o_ref, 'o')
    Kg = Ko[0].double().cpu().numpy()
    Vg = Vo[0].double().cpu().numpy()
    assert_close_fp32(Kg[:, :127], Kb, 'Kbar')
    assert_close_fp32(Vg[:, :127], Vb, 'Vbar')
    assert np.all(Kg[:, 127] == 0) and np.all(Vg[:, 127] == 0)


@pytest.mark.parametrize('cuda_cores', [False, True])
@pytest.mark.parametrize('B,T,H,D,C', [(2, 384, 3, 128, 64), (1, 512, 2, 128, 128),
                                       (3, 256, 1, 64, 128), (1, 64, 1, 128, 64),
                                       (1, 2304, 2, 128, 64), (1, 128, 2, 128, 64),
                                       (2, 1152, 2, 128, 64), (2, 256, 2, 256, 64),
                                       (1, 384, 2, 256, 128)])
def test_bf16_forward_small(B, T, H, D, C, cuda_cores):
    """Tensor-core kernels (bf16, d = 128, T a multiple of 128) and the CUDA-core kernels;
    T = 2304 spans several 1024-token segments plus a partial one, T = 128 is a single chunk
    (its first chunk is its last), T = 1152 ends with a one-chunk segment."""
    inp = to_device(synth.make_inputs(B, T, H, D, seed=2))
    d = cyfa.dims(B, T, H, D, chunk=C, cuda_cores=cuda_cores)
    o, Ko, Vo, _ = gpu_forward(d, inp, want_state=True)
    pairs = [(b, h) for b in range(B) for h in range(H)]
    oi = oracle_inputs(inp, pairs)
    o_ref, Kb, Vb, _ = oracle_forward(oi)
    assert_close_bf16(pairs_np(o.float(), pairs), o_ref, 'o')
    Kg = np.stack([Ko[b, h].double().cpu().numpy() for b, h in pairs])
    assert_close_bf16(Kg[:, :127], Kb, 'Kbar')
    assert np.all(Kg[:, 127] == 0)


def test_fp32_d256_parity():
    """fp32 at d = 256 (the paper's head size), 128-token caller chunks: within 1e-4."""
    inp = to_device(synth.make_inputs(1, 384, 2, 256, seed=12, dtype=torch.float32))
    d = cyfa.dims(1, 384, 2, 256, chunk=128, dtype=torch.float32)
    o, Ko, Vo, _ = gpu_forward(d, inp, want_state=True)
    pairs = [(0, 0), (0, 1)]
    o_ref, Kb, Vb, _ = oracle_forward(oracle_inputs(inp, pairs))
    assert_close_fp32(pairs_np(o, pairs), o_ref, 'o')
    assert_close_fp32(Vo[0].double().cpu().numpy()[:, :127], Vb, 'Vbar')


def test_paper_kernel_shape_forward_sampled():
    """The paper's kernel-latency shape (H = 4, d_k = d_v = 256, T = 2048, B = 32): every output
    of sampled (b, h) sequences against the oracle."""
    B, T, H, D = 32, 2048, 4, 256
    inp = synth.make_inputs(B, T, H, D, seed=0, device='cuda')
    d = cyfa.dims(B, T, H, D, chunk=64)
    o, _, _, _ = gpu_forward(d, inp)
    pairs = sample_pairs(B, H, 3)
    o_ref = oracle_forward(oracle_inputs(inp, pairs))[0]
    assert_close_bf16(pairs_np(o.float(), pairs), o_ref, 'o')


def test_stress_scale_and_identity_readout():
    """A large dot-product scale (sharp slot softmax) and R = I."""
    inp = to_device(synth.make_inputs(1, 256, 2, 128, seed=3, identity_R=True))
    inp['scale'] = 8.0
    d = cyfa.dims(1, 256, 2, 128, chunk=64, scale=8.0)
    o, _, _, _ = gpu_forward(d, inp)
    pairs = [(0, 0), (0, 1)]
    o_ref = oracle_forward(oracle_inputs(inp, pairs))[0]
    assert_close_bf16(pairs_np(o.float(), pairs), o_ref, 'o (s=8, R=I)')


def test_extreme_gates():
    """Saturated logits: clock increments near 0 / 1, forget gates near 0 (hard reset) / 1."""
    inp = to_device(synth.make_inputs(1, 256, 2, 128, seed=4))
    for key in ('clock_logit', 'decay_logit'):
        x = inp[key]
        x[:, ::3] = 12.0
        x[:, 1::3] = -12.0
    d = cyfa.dims(1, 256, 2, 128, chunk=64)
    o, _, _, _ = gpu_forward(d, inp)
    pairs = [(0, 0), (0, 1)]
    o_ref = oracle_forward(oracle_inputs(inp, pairs))[0]
    assert_close_bf16(pairs_np(o.float(), pairs), o_ref, 'o (saturated gates)')


@pytest.mark.parametrize('cuda_cores', [False, True])
@pytest.mark.parametrize('T,T1', [(512, 192), (2560, 1280)])
def test_state_continuation(T, T1, cuda_cores):
    """Forward over [0, T1) exporting (Kbar, Vbar, lambda), then [T1, T) started from them,
    against the oracle: the oracle's own states after T1 (absolute_clock over [0, T1)) are fed
    to absolute_clock over [T1, T) as (lambda0, Kbar0, Vbar0), and the library's exported states
    are compared with the oracle's after T1 and after T."""
    B, H, D = 1, 2, 128
    inp = to_device(synth.make_inputs(B, T, H, D, seed=5))
    seq = ('q', 'k', 'v', 'clock_logit', 'decay_logit', 'beta_logit')
    first = {k: (v[:, :T1].contiguous() if k in seq else v) for k, v in inp.items()}
    second = {k: (v[:, T1:].contiguous() if k in seq else v) for k, v in inp.items()}
    o1, K1, V1, l1 = gpu_forward(cyfa.dims(B, T1, H, D, chunk=64, cuda_cores=cuda_cores), first,
                                 want_state=True)
    o2, K2, V2, l2 = gpu_forward(cyfa.dims(B, T - T1, H, D, chunk=64, cuda_cores=cuda_cores),
                                 second, want_state=True, Kbar0=K1, Vbar0=V1, lambda0=l1)
    pairs = [(0, h) for h in range(H)]
    oi1, oi2 = oracle_inputs(first, pairs), oracle_inputs(second, pairs)
    r1, Kr1, Vr1, lr1 = oracle_forward(oi1)
    r2, Kr2, Vr2, lr2 = oracle_forward(oi2, lambda0=lr1, Kbar0=Kr1, Vbar0=Vr1)
    assert_close_bf16(pairs_np(o1.float(), pairs), r1, 'o [0, T1)')
    assert_close_bf16(pairs_np(o2.float(), pairs), r2, 'o [T1, T) from the exported states')
    for got, want, what in ((K1, Kr1, 'Kbar(T1)'), (V1, Vr1, 'Vbar(T1)'), (K2, Kr2, 'Kbar(T)'),
                            (V2, Vr2, 'Vbar(T)')):
        g = np.stack([got[0, h].double().cpu().numpy() for h in range(H)])
        assert_close_bf16(g[:, :127], want, what)
        assert np.all(g[:, 127] == 0)
    # the running clock continues: lambda_T of the second call against the oracle's
    np.testing.assert_allclose(l2[0].cpu().numpy(), lr2, rtol=0, atol=1e-6 + 4e-9 * T)


@pytest.mark.parametrize('B,T,H,C,cuda_cores', [(8, 4096, 8, 64, False), (8, 4096, 8, 64, True),
                                                 (2, 32768, 16, 64, False),
                                                 (2, 32768, 16, 128, True)])
def test_full_size_forward_sampled(B, T, H, C, cuda_cores):
    """The 400M-shaped (B8 H8 T4096) and 1.4B-shaped (B2 H16 T32768) layers: every output of
    sampled (b, h) sequences against the oracle."""
    inp = synth.make_inputs(B, T, H, 128, seed=0, device='cuda')
    d = cyfa.dims(B, T, H, 128, chunk=C, cuda_cores=cuda_cores)
    o, _, _, _ = gpu_forward(d, inp)
    pairs = sample_pairs(B, H, 3)
    o_ref = oracle_forward(oracle_inputs(inp, pairs))[0]
    assert_close_bf16(pairs_np(o.float(), pairs), o_ref, 'o')


def test_rejects_bad_arguments():
    d = cyfa.dims(1, 96, 1, 128, chunk=64)      # T not a multiple of the chunk
    x = torch.zeros(1, 96, 1, 128, dtype=torch.bfloat16, device='cuda')
    gsc = torch.zeros(1, 96, 1, device='cuda')
    R = torch.eye(127, device='cuda')[None]
    ws = torch.empty(1 << 20, dtype=torch.uint8, device='cuda')
    with pytest.raises(cyfa.CyfaError) as e:
        cyfa.cyfa_chunk_fwd(d, x, x, x, gsc, gsc, gsc, R, None, None, x, None, None, ws)
    assert e.value.code == cyfa.CYFA_ERR_SHAPE
    d = cyfa.dims(1, 128, 1, 128, chunk=64)
    x = torch.zeros(1, 128, 1, 128, dtype=torch.bfloat16, device='cuda')
    gsc = torch.zeros(1, 128, 1, device='cuda')
    with pytest.raises(cyfa.CyfaError) as e:
        cyfa.cyfa_chunk_fwd(d, x, x, x, gsc, gsc, gsc, R, None, None, x, None, None, ws[:16])
    assert e.value.code == cyfa.CYFA_ERR_WORKSPACE
    with pytest.raises(cyfa.CyfaError) as e:
        cyfa.cyfa_chunk_fwd(d, x.view(-1)[1:], x, x, gsc, gsc, gsc, R, None, None, x,
                            None, None, ws)
    assert e.value.code in (cyfa.CYFA_ERR_ALIGN, cyfa.CYFA_ERR_ARG)
