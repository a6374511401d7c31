"""The benchmark's multi-rank path on CPU: world size 2 over gloo (one process per rank, as
torchrun launches them).  Each rank runs its own replica and times it; the job time is the
slowest rank's and the value counts every rank's bytes (weak scaling, no data-path
collective).  The reference arm runs on rank 0 only."""
import os
import socket
import sys

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        local_ms = [120.0, 150.0][rank]  # rank 1 is the slow replica
        dist.barrier()
        m = bench.max_over_ranks(local_ms, world, "cpu")
        out[rank] = (m, bench.weak_scaling_gbs(1_000_000_000, 10, world, m))
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_agree_on_job_time_and_value():
    world, port = 2, _free_port()
    out = mp.Manager().dict()
    mp.spawn(_rank_main, args=(world, port, out), nprocs=world, join=True)
    assert out[0] == out[1]
    m, gbs = out[0]
    assert m == 150.0
    # 2 ranks x 10 steps x 1 GB in 150 ms
    assert gbs == pytest.approx(2 * 10 * 1.0 / 0.150)


def test_single_rank_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(3.5, 1, "cpu") == 3.5
    assert bench.weak_scaling_gbs(2_000_000_000, 5, 1, 1000.0) == pytest.approx(10.0)


def test_reference_arm_skips_non_zero_ranks(monkeypatch, capsys):
    sys.path.insert(0, ROOT)
    import bench
    monkeypatch.setenv("RANK", "1")
    ns = type("A", (), dict(steps=1, warmup=0, gpus=2))()
    assert bench.run_reference(ns) is None
    assert capsys.readouterr().out == ""
