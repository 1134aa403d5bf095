"""The canary guards of the GPU tests' outputs detect writes past either end (checked on CPU)."""
import pytest
import torch

from _harness import GUARD_BYTES, Guards


def test_guards_pass_in_bounds_and_catch_overruns():
    g = Guards()
    x = g.empty((3, 5), torch.float32, 'cpu')
    x.fill_(1.0)                       # every element, nothing outside
    g.check('in bounds')
    assert x.data_ptr() % 256 == g.bufs[0][0].data_ptr() % 256   # alignment kept
    raw, n = g.bufs[0]
    raw[GUARD_BYTES + n] = 0           # one byte past the end
    with pytest.raises(AssertionError):
        g.check('past the end')
    g2 = Guards()
    y = g2.empty((7,), torch.bfloat16, 'cpu')
    y.zero_()
    g2.bufs[0][0][GUARD_BYTES - 1] = 0  # one byte before the start
    with pytest.raises(AssertionError):
        g2.check('before the start')
