"""Host arithmetic of bench.py, on CPU: the flop counting rule of the roofline entry, its split
over the tensor-core launches, and the clock sampler's choice of nvidia-smi samples.

The counting rule charges, per (token, head), key pass 2Cd + 2Cm* + 4dm*, middle readout 4m*^2
and value pass 2Cm* + 2Cd + 4m*d to the forward and twice that to the backward (full C x C
blocks, d = m* = 128).  The expected values below are worked out from those terms by hand.
"""
import datetime
import os
import sys
import time

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import bench  # noqa: E402


def test_counting_rule_totals():
    # C = 64: 16384 + 16384 + 65536 (key) + 65536 (middle) + 16384 + 16384 + 65536 (value)
    assert bench.operator_flops_per_token_head(64) == 262144
    # C = 128: the four C-terms double (4 x 16384 more)
    assert bench.operator_flops_per_token_head(128) == 327680


@pytest.mark.parametrize('C', [16, 32, 64, 128, 256])
def test_counting_rule_is_affine_in_the_chunk(C):
    # C-free part 4dm* + 4m*^2 + 4m*d = 3 x 65536; C-part (2d + 2m* + 2m* + 2d) C = 1024 C
    assert bench.operator_flops_per_token_head(C) == 196608 + 1024 * C


STEP_SAVED = {'tc_seg_state': 1, 'tc_seg_out': 1, 'tc_bwd_chunk1': 1, 'tc_adj_segment': 1,
              'tc_snap_adj': 1, 'tc_bwd_chunk2': 1, 'tc_dm_reduce': 1}


def test_shares_add_up_to_the_rule():
    share, fwd_issued, bwd_issued = bench.tc_algorithmic_shares(STEP_SAVED, 64)
    fwd = share['tc_seg_state'] + share['tc_seg_out']
    bwd = sum(v for k, v in share.items() if k not in ('tc_seg_state', 'tc_seg_out'))
    assert fwd == pytest.approx(262144)
    assert bwd == pytest.approx(2 * 262144)
    # issued 128^3 products per 128-token chunk: forward 2 + 10, backward 13 + 2 + 2 + 12 + 2
    per_product = 2 * 128 ** 3 / 128
    assert fwd_issued == pytest.approx(12 * per_product)
    assert bwd_issued == pytest.approx(31 * per_product)


def test_dominant_kernel_share():
    # bwd_chunk1 issues 13 of the backward's 31 products: 524288 x 13 / 31 flops per token-head,
    # 2.305e11 per launch on the 2^20 token-heads of the B2 T32768 H16 layer
    share, _, _ = bench.tc_algorithmic_shares(STEP_SAVED, 64)
    assert share['tc_bwd_chunk1'] == pytest.approx(524288 * 13 / 31)
    assert share['tc_bwd_chunk1'] * 2 ** 20 == pytest.approx(2.305e11, rel=1e-3)


def test_recomputed_states_widen_the_backward():
    # without saved states the backward also walks the forward's chunk-start snapshots (2
    # products), so the same algorithmic backward is spread over 33 products
    step = dict(STEP_SAVED, tc_snap_fwd=1)
    share, _, _ = bench.tc_algorithmic_shares(step, 64)
    assert share['tc_snap_fwd'] == pytest.approx(524288 * 2 / 33)
    assert share['tc_bwd_chunk1'] == pytest.approx(524288 * 13 / 33)


# ------------------------------------------------------------------------------ clock samples
class _FakeProc:
    def terminate(self):
        pass

    def wait(self, timeout=None):
        pass


def _stamp(t):
    return datetime.datetime.fromtimestamp(t).strftime('%Y/%m/%d %H:%M:%S.%f')[:-3]


def _run_sampler(lines, t_begin, t_end):
    c = bench.ClockSampler(0)
    with open(c.path, 'w') as f:
        f.write('\n'.join(lines) + '\n')
    c.proc = _FakeProc()
    c.fh = open(os.devnull, 'w')
    c.t_begin, c.t_end = t_begin, t_end
    return c.stop()


def _line(t, sm, cap=False, slow=False, stamp=None):
    act = lambda on: 'Active' if on else 'Not Active'  # noqa: E731
    return '%s, 0, %d, 2070, 900.5, 0x0, %s, Not Active, Not Active, %s' % (
        stamp if stamp is not None else _stamp(t), sm, act(slow), act(cap))


def test_clock_samples_inside_the_timed_region_only():
    t = time.time()
    # idle clocks before the region, a slowdown after it: neither may enter the summary
    lines = [_line(t - 0.3, 1200, slow=True), _line(t - 0.1, 1500),
             _line(t + 0.01, 2070), _line(t + 0.06, 2055, cap=True), _line(t + 0.11, 2070),
             _line(t + 0.4, 900, slow=True)]
    clk = _run_sampler(lines, t, t + 0.12)
    assert clk['samples'] == 3
    assert clk['sampled'] == 'timed region'
    assert clk['sm_mhz'] == 2070.0
    assert clk['reasons'] == ['sw_power_cap']


def test_clock_samples_nearest_when_none_inside():
    t = time.time()
    lines = [_line(t - 0.2, 2000), _line(t - 0.1, 2040), _line(t + 0.3, 2070, cap=True)]
    clk = _run_sampler(lines, t, t + 0.005)
    assert clk['samples'] == 2
    assert clk['sampled'] == 'nearest samples around the timed region'
    assert clk['reasons'] == ['sw_power_cap']


def test_clock_samples_without_timestamps_use_all():
    t = time.time()
    lines = [_line(t, 2070, stamp='n/a'), _line(t, 2070, stamp='n/a', slow=True), 'garbage line']
    clk = _run_sampler(lines, t, t + 1)
    assert clk['samples'] == 2
    assert clk['sampled'] == 'all samples'
    assert clk['reasons'] == ['hw_slowdown']
