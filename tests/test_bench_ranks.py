"""Host logic of the N > 1 benchmark path on CPU: two gloo ranks, each a
replica with its own seeded inputs, combine their step times by a maximum
and report the whole-job rate (no data-path collective exists)."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as tmp

import bench
from paper_2609_06663_gb300.workloads import make_inputs, small_workload


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ms = [3.0, 5.0][rank]
        slowest = bench.max_over_ranks(ms, world, "cpu")
        w = small_workload(200, h_kv=2, dtype="bf16")
        K, _, _ = make_inputs(bench.rank_workload(w, rank))
        # the replicas really differ: gather a fingerprint of each rank's keys
        fp = torch.tensor([float(K.float().sum())], dtype=torch.float64)
        fps = [torch.zeros(1, dtype=torch.float64) for _ in range(world)]
        dist.all_gather(fps, fp)
        out[rank] = (slowest, bench.job_rate(world, 1000, slowest), [float(f) for f in fps])
    finally:
        dist.destroy_process_group()


def test_two_rank_replicas_combine_by_max():
    world = 2
    out = tmp.Manager().dict()
    tmp.spawn(_rank_main, args=(world, _free_port(), out), nprocs=world, join=True)
    for r in range(world):
        slowest, rate, fps = out[r]
        assert slowest == 5.0
        assert rate == pytest.approx(world * 1000 / 5e-3)
        assert fps[0] != fps[1]


def test_single_rank_is_identity():
    assert bench.max_over_ranks(2.5, 1, "cpu") == 2.5
    assert bench.job_rate(1, 100, 1.0) == pytest.approx(1e5)
