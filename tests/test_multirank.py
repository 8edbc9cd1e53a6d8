"""Replica bookkeeping across ranks (gloo, world size 2, CPU): the barrier, the
max-over-ranks of the timed duration and the whole-job rate bench.py reports."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from paper_2604_26412_gb300 import replicas


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        replicas.barrier()
        local_ms = 100.0 + 50.0 * rank          # rank 1 is the slow one
        worst = replicas.max_over_ranks(local_ms)
        rate = replicas.whole_job_rate(128, steps=10, world=world, max_ms=worst)
        out[rank] = (worst, rate)
    finally:
        dist.destroy_process_group()


def test_two_ranks_agree_on_slowest_time_and_rate():
    port = _free_port()
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_worker, args=(2, port, out), nprocs=2, join=True)
        res = dict(out)
    assert res[0] == res[1]
    worst, rate = res[0]
    assert worst == 150.0
    assert rate == pytest.approx(128 * 2 * 10 / 0.150)


def test_single_process_needs_no_process_group():
    assert replicas.max_over_ranks(3.5) == 3.5
    assert replicas.whole_job_rate(10, steps=4, world=1, max_ms=2.0) == pytest.approx(20000.0)
