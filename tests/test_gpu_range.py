"""fp16 operand range of the tensor-core kernels: large-magnitude values and near-unit decays.

The tensor-core kernels keep their operands in fp16 (fp32 accumulation).  The operator is
linear in v (o = Vbar^T o'', and o'' does not depend on v) and its gradients are linear in dO,
so scaled inputs are compared with the oracle after dividing by the scale: the stated bars then
apply unchanged.  Each case states the status cyfa_check() must give after the forward and after
the backward: CYFA_OK, and then the results match the oracle at those bars, or CYFA_ERR_RANGE
where an fp16 intermediate overflows (the guard must fire, and must not fire elsewhere).
"""
import numpy as np
import pytest
import torch

from paper_2609_36259_gb300 import cyfa, synth

from _harness import (assert_close_bf16, gpu_prepare, oracle_backward, oracle_forward,
                      oracle_inputs, pairs_np, to_device)

pytestmark = pytest.mark.gpu

B, T, H, D = 1, 2304, 2, 128


def _inputs(v_scale, dO_scale, coherent_v, A_min, seed=21):
    inp = synth.make_inputs(B, T, H, D, seed=seed, with_dO=True)
    v = inp['v'].float()
    if coherent_v:          # every value positive: the DC slot of Vbar adds up coherently
        v = v.abs() + 1.0
    inp['v'] = (v * v_scale).to(torch.bfloat16)
    inp['dO'] = (inp['dO'].float() * dO_scale).to(torch.bfloat16)
    # A_h log-spaced over [A_min, 1]: the slowest head decays by about A_min * 0.7 per token
    inp['A'] = torch.tensor([1.0, A_min], dtype=torch.float32)
    return to_device(inp)


def _status():
    try:
        cyfa.cyfa_check()
        return cyfa.CYFA_OK
    except cyfa.CyfaError as e:
        return e.code


def _run(inp):
    d = cyfa.dims(B, T, H, D, chunk=64)
    lam, g, beta, _ = gpu_prepare(d, inp)
    q, k, v, dO = inp['q'], inp['k'], inp['v'], inp['dO']
    o = cyfa.forward(d, q, k, v, lam, g, beta, inp['R'])[0]
    st_fwd = _status()
    out = dict(dq=torch.empty_like(q), dk=torch.empty_like(k), dv=torch.empty_like(v),
               d_clock=torch.empty_like(lam), d_decay=torch.empty_like(lam),
               d_beta=torch.empty_like(lam))
    ws = cyfa.workspace(d, cyfa.CYFA_WS_BWD, q.device)
    cyfa.cyfa_chunk_bwd(d, q, k, v, lam, g, beta, inp['R'], inp['clock_logit'],
                        inp['decay_logit'], inp['A'], dO, out['dq'], out['dk'], out['dv'],
                        out['d_clock'], out['d_decay'], out['d_beta'], None, None, ws)
    st_bwd = _status()
    return o, st_fwd, out, st_bwd


OK, RANGE = cyfa.CYFA_OK, cyfa.CYFA_ERR_RANGE
# (v scale, dO scale, coherent v, smallest A, expected forward / backward status).  Scaling by a
# power of two is exact, so a case either reproduces the unscaled errors or overflows somewhere.
CASES = [
    (64.0, 1.0, False, 1.0 / 4096, OK, OK),
    (512.0, 1.0, False, 1.0 / 4096, OK, OK),
    (1.0, 64.0, False, 1.0 / 4096, OK, OK),
    (1.0, 512.0, False, 1.0 / 4096, OK, OK),
    (1024.0, 1.0, True, 1.0 / 4096, RANGE, RANGE),   # Vbar's DC row passes 65504
    (64.0, 64.0, False, 1.0 / 4096, OK, RANGE),      # dL/do' = Vbar dO passes 65504
]


@pytest.mark.parametrize('v_scale,dO_scale,coherent,A_min,want_fwd,want_bwd', CASES)
def test_fp16_range(v_scale, dO_scale, coherent, A_min, want_fwd, want_bwd):
    inp = _inputs(v_scale, dO_scale, coherent, A_min)
    o, st_fwd, out, st_bwd = _run(inp)
    assert (st_fwd, st_bwd) == (want_fwd, want_bwd), (st_fwd, st_bwd)
    pairs = [(0, h) for h in range(H)]
    oi = oracle_inputs(inp, pairs)
    if st_fwd == cyfa.CYFA_OK:
        o_ref = oracle_forward(oi)[0]
        assert_close_bf16(pairs_np(o.float(), pairs) / v_scale, o_ref / v_scale, 'o / s_v')
    if st_bwd == cyfa.CYFA_OK:
        ref = oracle_backward(oi, pairs_np(inp['dO'], pairs))
        # dv is linear in dO; dq, dk and the logit gradients in v and dO together
        for key, sc in (('dq', v_scale * dO_scale), ('dk', v_scale * dO_scale),
                        ('dv', dO_scale), ('d_clock', v_scale * dO_scale),
                        ('d_decay', v_scale * dO_scale), ('d_beta', v_scale * dO_scale)):
            assert_close_bf16(pairs_np(out[key].float(), pairs) / sc, ref[key] / sc,
                              '%s / scale' % key)


def test_non_finite_input_is_reported():
    """A NaN in v is not an fp16 overflow, but it reaches o the same way: CYFA_ERR_RANGE."""
    inp = _inputs(1.0, 1.0, False, 1.0 / 256)
    inp['v'][0, 300, 1, 5] = float('nan')
    o, st_fwd, out, st_bwd = _run(inp)
    assert st_fwd == RANGE and st_bwd == RANGE
    # the call after a reported error starts from a clear error word
    inp = _inputs(1.0, 1.0, False, 1.0 / 256)
    _, st_fwd, _, st_bwd = _run(inp)
    assert st_fwd == OK and st_bwd == OK
