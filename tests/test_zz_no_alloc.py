"""cyfa_prepare_noalloc: the prepare call for callers that cannot hand the library device
memory (for example a serving host whose own allocator owns all device memory and forbids
further cudaMalloc calls).  It must give the results of cyfa_prepare, call after call, with its
partial sums in the library's fixed scratch array instead of a workspace.

This file is collected last so that a failure here never hides the other tests."""
import ctypes

import pytest
import torch

from paper_2609_36259_gb300 import cyfa, synth

pytestmark = pytest.mark.gpu


def _both(B, T, H, C, seed):
    inp = synth.make_inputs(B, T, H, 64, seed=seed, device='cuda')
    d = cyfa.dims(B, T, H, 64, chunk=C)
    lam0 = torch.rand(B, H, dtype=torch.float64, device='cuda') * 50
    ref = cyfa.prepare(d, inp['clock_logit'], inp['decay_logit'], inp['beta_logit'], inp['A'],
                       lambda0=lam0, want_lambda_end=True)
    got = [torch.empty_like(ref[0]), torch.empty_like(ref[1]), torch.empty_like(ref[2]),
           torch.empty_like(ref[3])]
    cyfa.cyfa_prepare_noalloc(d, inp['clock_logit'], inp['decay_logit'], inp['beta_logit'],
                              inp['A'], lam0, got[0], got[1], got[2], got[3])
    torch.cuda.synchronize()
    return ref, got


def test_noalloc_prepare_matches_workspace_prepare_twice():
    # two calls in a row, with different shapes, on the same shared scratch array
    for (B, T, H, C, seed) in [(2, 32768, 16, 64, 0), (3, 1088, 5, 64, 1)]:
        ref, got = _both(B, T, H, C, seed)
        for r, g in zip(ref, got):
            assert torch.equal(r, g), (B, T, H)   # same kernels, same order: bit-identical


def test_noalloc_prepare_rejects_shapes_beyond_its_scratch():
    d = cyfa.dims(256, 131072, 16, 64, chunk=64)     # 256*16*128 partial sums > 32768
    with pytest.raises(cyfa.CyfaError) as e:
        cyfa.cyfa_prepare_noalloc(d, *([torch.empty(1, device='cuda')] * 9))
    assert e.value.code == cyfa.CYFA_ERR_WORKSPACE
