"""The multi-GPU path of bench.py on the CPU: replicas of the draft step, one process per rank,
no collective on the data path.  Two gloo ranks check the host logic the GPU run uses: the
job's time is its slowest rank's (a MAX all-reduce), the value counts every rank's blocks, and
the reference arm runs on rank 0 alone."""
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


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", init_method="env://", rank=rank, world_size=world)
    try:
        r, w, local = bench.dist_env()
        # each rank timed its own steps; rank r took (1 + r) seconds
        t = bench.max_over_ranks(1.0 + r, w, torch.device("cpu"))
        dist.barrier()
        out.put((r, w, local, t, bench.job_throughput(w, 1, 100, t)))
    finally:
        dist.destroy_process_group()


def test_two_rank_replicas_take_the_slowest_rank():
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    got = sorted(q.get(timeout=120) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [g[0] for g in got] == [0, 1]
    assert all(g[1] == world and g[2] == g[0] for g in got)
    # both ranks see the slowest rank's 2.0 s; 2 ranks x 100 steps x 1 block / 2.0 s
    assert all(g[3] == 2.0 for g in got)
    assert all(g[4] == pytest.approx(100.0) for g in got)


def test_single_rank_needs_no_process_group():
    assert bench.max_over_ranks(3.5, 1, torch.device("cpu")) == 3.5
    assert bench.job_throughput(1, 32, 10, 2.0) == pytest.approx(160.0)


def test_reference_arm_runs_on_rank_zero_only(monkeypatch):
    """Under torchrun every rank but 0 leaves at once, before any work (and prints nothing)."""
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    monkeypatch.setenv("LOCAL_RANK", "1")

    class Args:
        config = "qwen3-8b"
        steps = 1
        warmup = 3
    assert bench.run_reference(Args()) == 0
