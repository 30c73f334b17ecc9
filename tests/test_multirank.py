"""The multi-rank host logic of bench.py on world size 2 with the gloo backend
(CPU): the barrier, the max-over-ranks timing reduction, the whole-job rate,
and the reference arm printing on rank 0 only."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        dist.barrier()
        # each rank times its own replica; the slower rank decides the job's time
        local_seconds = 2.0 if rank == 1 else 1.0
        slowest = bench.max_over_ranks(local_seconds, "cpu")
        rate = bench.whole_job_rate(128, world, slowest)
        q.put((rank, slowest, rate))
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_and_rate_on_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    got = sorted(q.get(timeout=10) for _ in range(2))
    for rank, slowest, rate in got:
        assert slowest == 2.0                 # max over ranks, seen by every rank
        assert rate == pytest.approx(128.0)   # 2 ranks x 128 windows / 2 s


def test_single_rank_reduction_is_identity():
    assert bench.max_over_ranks(3.5) == 3.5
    assert bench.whole_job_rate(10, 1, 2.0) == 5.0


def test_reference_arm_prints_nothing_on_other_ranks(monkeypatch, capsys):
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    monkeypatch.setattr("sys.argv", ["bench.py", "--impl", "reference", "--gpus", "2", "--workload", "tiny"])
    bench.main()
    assert capsys.readouterr().out == ""
