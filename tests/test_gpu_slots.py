"""Slot-count variants (the paper's ablation over m, Table ablations): odd m through the C ABI
against the fp64 oracle, on the tensor-core kernels (bf16, d = 128, 63 <= m <= 127) and on the
CUDA-core kernels.  m <= 127 keeps 128 storage rows, larger m (the ablation's m = 255) 256; the
rows m.. of the storage stay zero."""
import numpy as np
import pytest
import torch

from paper_2609_36259_gb300 import cyfa, synth

from _harness import (assert_close_bf16, assert_close_fp32, assert_close_rel, gpu_forward,
                      oracle_backward, oracle_forward, oracle_inputs, pairs_np, sample_pairs,
                      to_device)
from test_gpu_backward import GRADS, gpu_backward
from test_gpu_decode import _decode

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize('m,dtype,D,cuda_cores', [(5, torch.bfloat16, 128, False),
                                                  (63, torch.bfloat16, 128, False),
                                                  (63, torch.bfloat16, 128, True),
                                                  (1, torch.float32, 64, True),
                                                  (5, torch.float32, 64, True),
                                                  (63, torch.float32, 64, True),
                                                  (255, torch.float32, 64, True),
                                                  (255, torch.bfloat16, 128, False),
                                                  (255, torch.bfloat16, 256, False),
                                                  (131, torch.float32, 128, True)])
def test_slots_forward_backward(m, dtype, D, cuda_cores):
    """m = 5 in bf16 runs on the CUDA-core kernels even unforced (the tensor-core kernels take
    63 <= m <= 127), and so do m = 131 and m = 255 (256 storage rows).  m = 1 runs in fp32 only:
    its single slot sums v over the whole memory (outputs up to ~30 here), where the bf16 rounding
    of the output alone (2^-9 |o|) exceeds the 2e-2 bar."""
    B, T, H = 1, 384, 2
    inp = to_device(synth.make_inputs(B, T, H, D, seed=41, dtype=dtype, with_dO=True, m=m))
    d = cyfa.dims(B, T, H, D, chunk=64, dtype=dtype, m=m, cuda_cores=cuda_cores)
    o, Ko, Vo, _ = gpu_forward(d, inp, want_state=True)
    out = gpu_backward(d, inp, want_dR=True)
    pairs = [(0, h) for h in range(H)]
    oi = oracle_inputs(inp, pairs)
    o_ref, Kb, Vb, _ = oracle_forward(oi)
    ref = oracle_backward(oi, pairs_np(inp['dO'], pairs))
    close = assert_close_bf16 if dtype == torch.bfloat16 else assert_close_fp32
    close(pairs_np(o.float(), pairs), o_ref, 'm=%d o' % m)
    Kg = np.stack([Ko[0, h].double().cpu().numpy() for h in range(H)])
    close(Kg[:, :m], Kb, 'm=%d Kbar' % m)
    assert np.all(Kg[:, m:] == 0)          # the padding rows stay zero
    for gk, rk in GRADS:
        close(pairs_np(out[gk].float(), pairs), ref[rk], 'm=%d %s' % (m, gk))
    dR = out['dR'].double().cpu().numpy()
    assert dR.shape == (H, m, m)
    if dtype == torch.bfloat16:
        assert_close_rel(dR, ref['dR'], 'm=%d dR' % m)
    else:
        assert np.abs(dR - ref['dR']).max() <= 1e-4 * max(1.0, np.abs(ref['dR']).max())


def test_slots_63_full_size_sampled():
    """m = 63 on the 1.4B-shaped layer (B2 H16 T32768 d128, the tensor-core kernels): outputs
    and gradients of sampled (b, h) sequences."""
    B, T, H, m = 2, 32768, 16, 63
    inp = synth.make_inputs(B, T, H, 128, seed=2, device='cuda', with_dO=True, m=m)
    d = cyfa.dims(B, T, H, 128, chunk=64, m=m)
    o = gpu_forward(d, inp)[0]
    out = gpu_backward(d, inp, want_dA=False)
    pairs = sample_pairs(B, H, 2)
    oi = oracle_inputs(inp, pairs)
    assert_close_bf16(pairs_np(o.float(), pairs), oracle_forward(oi)[0], 'm=63 o')
    ref = oracle_backward(oi, pairs_np(inp['dO'], pairs))
    for gk, rk in GRADS:
        assert_close_bf16(pairs_np(out[gk].float(), pairs), ref[rk], 'm=63 %s' % gk)


def test_slots_255_paper_shape_sampled():
    """m = 255 at the shape of the paper's ablation model (400M: H = 4, d = 256, T = 2048; B = 8
    of its 32 here): outputs and gradients of sampled (b, h) sequences (dA and dR, sums over
    every sequence, are checked at the small size above)."""
    B, T, H, D, m = 8, 2048, 4, 256, 255
    inp = synth.make_inputs(B, T, H, D, seed=5, device='cuda', with_dO=True, m=m)
    d = cyfa.dims(B, T, H, D, chunk=64, m=m)
    o = gpu_forward(d, inp)[0]
    out = gpu_backward(d, inp, want_dA=False)
    pairs = sample_pairs(B, H, 3)
    oi = oracle_inputs(inp, pairs)
    assert_close_bf16(pairs_np(o.float(), pairs), oracle_forward(oi)[0], 'm=255 o')
    ref = oracle_backward(oi, pairs_np(inp['dO'], pairs))
    for gk, rk in GRADS:
        assert_close_bf16(pairs_np(out[gk].float(), pairs), ref[rk], 'm=255 %s' % gk)


@pytest.mark.parametrize('m,D', [(5, 128), (63, 128), (255, 128), (255, 256)])
def test_slots_decode(m, D):
    B, H, T0, steps = 2, 3, 128, 16
    inp = synth.make_inputs(B, T0 + steps, H, D, seed=42, device='cuda', m=m)
    o, K, V, lam = _decode(inp, T0, steps, cyfa.dims(B, T0, H, D, chunk=64, m=m),
                           cyfa.dims(B, 1, H, D, chunk=64, m=m))
    pairs = [(b, h) for b in range(B) for h in range(H)]
    o_ref, Kb, _, _ = oracle_forward(oracle_inputs(inp, pairs))
    got = np.stack([o[b, :, h].double().cpu().numpy() for b, h in pairs])
    assert_close_bf16(got, o_ref[:, T0:], 'm=%d decode o' % m)
    Kg = np.stack([K[b, h].double().cpu().numpy() for b, h in pairs])
    assert_close_bf16(Kg[:, :m], Kb, 'm=%d Kbar after decode' % m)
    assert K.shape[2] == cyfa.storage_rows(m)
    assert torch.all(K[:, :, m:] == 0) and torch.all(V[:, :, m:] == 0)   # padding rows stay zero
