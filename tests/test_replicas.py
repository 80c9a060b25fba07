"""The multi-GPU bookkeeping of the benchmark (replicas: one process per GPU, no data-path
collective) on the CPU with two gloo ranks: the job time is the slowest rank's, the throughput
counts every rank's tokens, and a rank that dies is noticed by the other's next collective
instead of hanging it."""
import datetime
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from paper_2606_00395_gb300 import replicas


def _port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _init(rank, world, port, timeout_s=30):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world,
                            timeout=datetime.timedelta(seconds=timeout_s))


def _job(rank, world, port, out):
    _init(rank, world, port)
    assert replicas.rank_env() == (rank, world, rank)
    local = 10.0 + 5.0 * rank  # rank 1 is the slow one
    job = replicas.job_time_ms(local, dist)
    out[rank] = (job, replicas.job_throughput(4096 * 100, world, job))
    dist.barrier()
    dist.destroy_process_group()


def _dies(rank, world, port, out):
    _init(rank, world, port, timeout_s=10)
    dist.barrier()
    if rank == 1:
        os._exit(0)  # leaves between steps, with no collective in flight
    try:
        replicas.job_time_ms(1.0, dist)
        out[rank] = "no error"
    except Exception as e:  # noqa: BLE001 - any error is the expected detection
        out[rank] = "error: " + type(e).__name__


def _run(fn, world=2):
    ctx = mp.get_context("spawn")
    with ctx.Manager() as m:
        out = m.dict()
        port = _port()
        procs = [ctx.Process(target=fn, args=(r, world, port, out)) for r in range(world)]
        for p in procs:
            p.start()
        for p in procs:
            p.join(60)
            assert not p.is_alive(), "a rank hung"
        return dict(out)


def test_job_time_is_the_slowest_rank_and_throughput_counts_every_rank():
    out = _run(_job)
    assert out[0] == out[1]
    job, tput = out[0]
    assert job == 15.0
    assert tput == pytest.approx(2 * 4096 * 100 / 0.015)


def test_single_process_needs_no_group():
    assert replicas.job_time_ms(3.5) == 3.5
    assert replicas.job_throughput(10, 1, 1000.0) == 10.0
    with pytest.raises(ValueError):
        replicas.job_throughput(10, 1, 0.0)


def test_a_rank_that_leaves_is_detected_by_the_next_collective():
    out = _run(_dies)
    assert out[0].startswith("error"), out
