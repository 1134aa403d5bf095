"""The largest accepted number of (b, h) sequences, B * H = 65535 (the per-sequence launches put
B * H on gridDim.y), through prepare, forward, backward and decode, against the oracle on
sampled sequences including the first and the last."""
import numpy as np
import pytest
import torch

from paper_2609_36259_gb300 import cyfa, synth

from _harness import (assert_close_bf16, gpu_forward, oracle_backward, oracle_forward,
                      oracle_inputs, pairs_np, sample_pairs)
from test_gpu_backward import GRADS, gpu_backward
from test_gpu_decode import _decode

pytestmark = pytest.mark.gpu

B_MAX, H = 65535, 1


@pytest.mark.parametrize('cuda_cores', [False, True])
def test_max_sequences_forward_backward(cuda_cores):
    T, D = 128, 128
    inp = synth.make_inputs(B_MAX, T, H, D, seed=21, device='cuda', with_dO=True)
    d = cyfa.dims(B_MAX, T, H, D, chunk=64, cuda_cores=cuda_cores)
    o = gpu_forward(d, inp)[0]
    out = gpu_backward(d, inp, want_dA=False)
    pairs = sample_pairs(B_MAX, H, 4, seed=3)
    assert (B_MAX - 1, H - 1) in pairs
    oi = oracle_inputs(inp, pairs)
    assert_close_bf16(pairs_np(o.float(), pairs), oracle_forward(oi)[0], 'max B*H o')
    ref = oracle_backward(oi, pairs_np(inp['dO'], pairs))
    for gk, rk in GRADS:
        assert_close_bf16(pairs_np(out[gk].float(), pairs), ref[rk], 'max B*H %s' % gk)
    torch.cuda.synchronize()
    del inp, o, out
    torch.cuda.empty_cache()


def test_max_sequences_decode():
    T0, steps, D = 128, 3, 128
    inp = synth.make_inputs(B_MAX, T0 + steps, H, D, seed=22, device='cuda')
    o, K, V, lam = _decode(inp, T0, steps, cyfa.dims(B_MAX, T0, H, D, chunk=64),
                           cyfa.dims(B_MAX, 1, H, D, chunk=64))
    pairs = sample_pairs(B_MAX, H, 4, seed=4)
    o_ref = oracle_forward(oracle_inputs(inp, pairs))[0]
    got = np.stack([o[b, :, h].double().cpu().numpy() for b, h in pairs])
    assert_close_bf16(got, o_ref[:, T0:], 'max B*H decode o')
    torch.cuda.synchronize()
    del inp, o, K, V
    torch.cuda.empty_cache()
