"""Host logic of bench.py's multi-GPU path, on CPU: two gloo ranks.

With --gpus N every rank runs its own batch; the job's step time is the max over ranks and the
throughput counts the tokens of all ranks.  The reference arm runs on rank 0 only.
"""
import io
import os
import socket
import sys
from contextlib import redirect_stdout

import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import bench  # noqa: E402


def _free_port():
    with socket.socket() as s:
        s.bind(('127.0.0.1', 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR='127.0.0.1', MASTER_PORT=str(port))
    dist.init_process_group('gloo', rank=rank, world_size=world)
    try:
        my_ms = [2.0, 5.0][rank]
        ms = bench.job_step_ms(my_ms, dist, torch.device('cpu'))
        out[rank] = (ms, bench.job_tokens_per_s(65536, world, ms))
    finally:
        dist.destroy_process_group()


def test_job_step_time_is_the_max_over_two_gloo_ranks():
    world = 2
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_rank_main, args=(world, _free_port(), out), nprocs=world, join=True)
        res = dict(out)
    for rank in range(world):
        ms, tps = res[rank]
        assert ms == 5.0                                  # the slower rank sets the step time
        assert abs(tps - 2 * 65536 / 5e-3) < 1e-6 * tps   # tokens of both ranks


def test_single_rank_keeps_its_own_time():
    assert bench.job_step_ms(3.5) == 3.5
    assert bench.job_tokens_per_s(1000, 1, 2.0) == 500000.0


def test_reference_arm_runs_on_rank_zero_only(monkeypatch):
    monkeypatch.setenv('RANK', '1')
    monkeypatch.setenv('WORLD_SIZE', '2')

    class A:
        steps, warmup, ref_tokens, chunk = 1, 0, 64, 64

    buf = io.StringIO()
    with redirect_stdout(buf):
        bench.run_reference(A())
    assert buf.getvalue() == ''
