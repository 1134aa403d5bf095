"""Failure detection without a GPU fault: a bounded device-side wait that runs out.

Every wait of the library's kernels on an mbarrier is a bounded poll loop; when it gives up,
the kernel records CYFA_ERR_TIMEOUT in a device error word and returns, and the host reads the
status (cyfa_check, or the self-check's return code).  Here one device thread waits on an
mbarrier that nothing ever completes, with the kernels' own bounded wait given a 20 ms limit
instead of their 2 s.  The test checks the status, the time the wait took, and that the context
is still usable afterwards.
"""
import numpy as np
import pytest
import torch

from paper_2609_36259_gb300 import cyfa, synth
from _harness import assert_close_bf16, oracle_forward, oracle_inputs, pairs_np, to_device


@pytest.mark.gpu
def test_bounded_wait_expires_and_context_survives():
    el = torch.zeros(1, dtype=torch.int64, device='cuda')
    rc = cyfa.cyfa_selftest_timeout(20000, el)
    assert rc == cyfa.CYFA_ERR_TIMEOUT, cyfa.error_string(rc)
    assert 20e6 <= int(el.item()) < 1e9, int(el.item())   # gave up after the limit, not much later
    # the error word of the probe does not leak into the library's own status
    cyfa.cyfa_check()
    # the context still runs kernels: a small tensor-core forward against the oracle
    B, T, H, D = 1, 256, 2, 128
    inp = to_device(synth.make_inputs(B, T, H, D, seed=12))
    d = cyfa.dims(B, T, H, D, chunk=64)
    lam, g, beta, _ = cyfa.prepare(d, inp['clock_logit'], inp['decay_logit'], inp['beta_logit'],
                                   inp['A'])
    o, _, _ = cyfa.forward(d, inp['q'], inp['k'], inp['v'], lam, g, beta, inp['R'])
    cyfa.cyfa_check()
    pairs = [(0, h) for h in range(H)]
    o_ref = oracle_forward(oracle_inputs(inp, pairs))[0]
    assert_close_bf16(pairs_np(o.float(), pairs), o_ref, 'o after the expired wait')


@pytest.mark.gpu
def test_timeout_probe_rejects_bad_limits():
    assert cyfa.cyfa_selftest_timeout(0) == cyfa.CYFA_ERR_ARG
    assert cyfa.cyfa_selftest_timeout(1000001) == cyfa.CYFA_ERR_ARG
