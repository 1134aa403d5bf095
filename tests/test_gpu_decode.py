"""GPU parity of cyfa_step (single-token decode) against the fp64 oracle stepped token by token."""
import numpy as np
import pytest
import torch

from paper_2609_36259_gb300 import cyfa, synth

from _harness import (Guards, assert_close_bf16, gpu_forward, oracle_forward, oracle_inputs,
                      pairs_np, sample_pairs)

pytestmark = pytest.mark.gpu


def _decode(inp, T0, steps, d_prefill, d_step):
    """Prefill tokens [0, T0) with cyfa_chunk_fwd, then cyfa_step for tokens [T0, T0+steps)."""
    seq = ('q', 'k', 'v', 'clock_logit', 'decay_logit', 'beta_logit')
    pre = {k: (v[:, :T0].contiguous() if k in seq else v) for k, v in inp.items()}
    _, K, V, lam = gpu_forward(d_prefill, pre, want_state=True)
    B, _, H, D = inp['q'].shape
    outs = []
    gd = Guards()
    for t in range(T0, T0 + steps):
        o = gd.empty((B, H, D), inp['v'].dtype)
        cyfa.cyfa_step(d_step, inp['q'][:, t].contiguous(), inp['k'][:, t].contiguous(),
                       inp['v'][:, t].contiguous(), inp['clock_logit'][:, t].contiguous(),
                       inp['decay_logit'][:, t].contiguous(), inp['beta_logit'][:, t].contiguous(),
                       inp['A'], inp['R'], K, V, lam, o)
        outs.append(o)
    gd.check('cyfa_step')
    return torch.stack(outs, 1), K, V, lam


@pytest.mark.parametrize('dtype,D', [(torch.bfloat16, 128), (torch.float32, 64),
                                     (torch.bfloat16, 256), (torch.float32, 256)])
def test_decode_small(dtype, D):
    B, H, T0, steps = 2, 3, 128, 24
    inp = synth.make_inputs(B, T0 + steps, H, D, seed=6, dtype=dtype, device='cuda')
    d_pre = cyfa.dims(B, T0, H, D, chunk=64, dtype=dtype)
    d_step = cyfa.dims(B, 1, H, D, chunk=64, dtype=dtype)
    o, K, V, lam = _decode(inp, T0, steps, d_pre, d_step)
    pairs = [(b, h) for b in range(B) for h in range(H)]
    o_ref, Kb, Vb, lam_ref = oracle_forward(oracle_inputs(inp, pairs))
    got = np.stack([o[b, :, h].double().cpu().numpy() for b, h in pairs])
    if dtype == torch.float32:
        assert np.max(np.abs(got - o_ref[:, T0:])) < 1e-4
    else:
        assert_close_bf16(got, o_ref[:, T0:], 'decode o')
    Kg = np.stack([K[b, h].double().cpu().numpy() for b, h in pairs])
    if dtype == torch.float32:
        assert np.max(np.abs(Kg[:, :127] - Kb)) < 1e-4
    else:   # bf16 prefill: the tensor-core kernels round the write vectors to bf16
        assert_close_bf16(Kg[:, :127], Kb, 'Kbar after decode')
    assert np.all(Kg[:, 127] == 0)
    np.testing.assert_allclose([lam[b, h].item() for b, h in pairs], lam_ref, atol=1e-6)


def test_decode_full_size_sampled():
    """B=256 H=16 d=128, fp32 states: 2048-token prefill, then 1024 steps; sampled (b, h)
    sequences checked token by token against the oracle."""
    B, H, D, T0, steps = 256, 16, 128, 2048, 1024
    inp = synth.make_inputs(B, T0 + steps, H, D, seed=0, device='cuda')
    d_pre = cyfa.dims(B, T0, H, D, chunk=64)
    d_step = cyfa.dims(B, 1, H, D, chunk=64)
    o, K, V, lam = _decode(inp, T0, steps, d_pre, d_step)
    pairs = sample_pairs(B, H, 3)
    o_ref, Kb, Vb, _ = oracle_forward(oracle_inputs(inp, pairs))
    got = np.stack([o[b, :, h].double().cpu().numpy() for b, h in pairs])
    assert_close_bf16(got, o_ref[:, T0:], 'decode o')
    Vg = np.stack([V[b, h].double().cpu().numpy() for b, h in pairs])
    assert_close_bf16(Vg[:, :127], Vb, 'Vbar after decode')
