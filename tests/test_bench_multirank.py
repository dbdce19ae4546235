"""The multi-GPU path of bench.py on CPU: two gloo ranks (no GPU).

Each rank runs its own replica (weak scaling, no data exchange); the job's
time is the slowest rank's and the throughput counts every rank's steps."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        from paper_2608_02625_gb300 import workloads
        base = workloads.get("c3_batch32_512")
        w = bench.replica_workload(base, rank)
        local_ms = 10.0 + 5.0 * rank          # rank 1 is the slow one
        slowest = bench.max_over_ranks(local_ms, world, torch.device("cpu"))
        dist.barrier()
        out[rank] = (w.seed, w.B, w.L, slowest, bench.job_steps_per_s(slowest, world))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks():
    world, port = 2, _free_port()
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_rank_main, args=(world, port, out), nprocs=world, join=True)
        res = dict(out)
    (s0, b0, l0, t0, v0), (s1, b1, l1, t1, v1) = res[0], res[1]
    assert s0 != s1                       # each replica refines its own batch
    assert (b0, l0) == (b1, l1) == (32, 512)  # of the same shape
    assert t0 == t1 == 15.0               # max over ranks
    assert v0 == pytest.approx(2 * 1000.0 / 15.0)


def test_single_rank_is_local():
    import bench
    assert bench.max_over_ranks(12.5, 1, torch.device("cpu")) == 12.5
    assert bench.job_steps_per_s(4.0, 1) == 250.0
