"""Host logic of bench.py's multi-GPU mode (replicas only: the path shards by
sequence with no exchange), checked on CPU with world_size-2 gloo process
groups: the job's time is the slowest rank's, throughput is whole-job, and the
reference arm runs on rank 0 alone."""
import os
import socket
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    import torch
    import torch.distributed as dist

    sys.path.insert(0, ROOT)
    import bench

    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank,
                            world_size=world)
    try:
        local_ms = [12.5, 20.0][rank]
        out[rank] = bench.max_over_ranks(local_ms, torch.device("cpu"), world)
    finally:
        dist.destroy_process_group()


def test_max_over_two_gloo_ranks():
    world = 2
    port = _free_port()
    ctx = mp.get_context("spawn")
    with ctx.Manager() as m:
        out = m.dict()
        mp.start_processes(_worker, args=(world, port, out), nprocs=world, join=True,
                           start_method="spawn")
        assert out[0] == out[1] == 20.0


def test_single_rank_needs_no_process_group():
    import bench

    assert bench.max_over_ranks(3.5, None, 1) == 3.5


def test_replica_throughput_is_whole_job():
    import bench

    # 2 ranks x 100 steps, the slowest in 50 ms -> 4000 steps/s for the job
    assert bench.replica_throughput(100, 2, 50.0) == pytest.approx(4000.0)
    assert bench.replica_throughput(100, 1, 50.0) == pytest.approx(2000.0)


def test_reference_arm_runs_on_rank_zero_only(monkeypatch, capsys):
    import bench

    monkeypatch.setenv("WORLD_SIZE", "2")
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("LOCAL_RANK", "1")

    class Args:
        workload = "decode_small"
        steps = 1
        warmup = 1

    assert bench.run_reference(Args()) is None
    assert capsys.readouterr().out == ""
