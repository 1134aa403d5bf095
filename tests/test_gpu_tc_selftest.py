"""Tensor-core operand layouts (tcgen05 + TMEM + TMA, 128-byte swizzle) against torch matmul."""
import pytest
import torch

from paper_2609_36259_gb300 import cyfa

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize('variant', range(8))
def test_selftest_mma(variant):
    g = torch.Generator(device='cuda').manual_seed(variant)
    X = torch.randn(128, 128, device='cuda', generator=g).to(torch.bfloat16)
    Y = torch.randn(128, 128, device='cuda', generator=g).to(torch.bfloat16)
    D = torch.full((128, 128), float('nan'), device='cuda')
    cyfa.cyfa_selftest_mma(variant, X, Y, D)
    A = X.float().t() if variant & 1 else X.float()
    Bm = Y.float() if variant & 2 else Y.float().t()
    ref = A @ Bm
    torch.testing.assert_close(D, ref, rtol=1e-4, atol=1e-3)
