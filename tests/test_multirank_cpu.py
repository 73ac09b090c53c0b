"""The benchmark's multi-rank path on CPU: two gloo ranks, each an
independent replica; the job's time is the slowest rank's and the job's
throughput counts every rank's tokens."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    from paper_2609_35440_gb300 import workloads
    ms = [12.5, 17.25][rank]                     # each rank's own timed region
    slowest = bench.max_over_ranks(ms)
    value = bench.job_throughput(32768, 10, world, slowest)
    seed = bench.replica_workload(workloads.W1P3B, rank).seed
    dist.barrier()
    out[rank] = (slowest, value, seed)
    dist.destroy_process_group()


def test_two_gloo_ranks_take_the_slowest_time_and_all_tokens():
    world = 2
    port = _free_port()
    mgr = mp.Manager()
    out = mgr.dict()
    mp.spawn(_worker, args=(world, port, out), nprocs=world, join=True)
    (s0, v0, seed0), (s1, v1, seed1) = out[0], out[1]
    assert s0 == s1 == 17.25
    assert v0 == v1 == pytest.approx(2 * 32768 * 10 / 17.25e-3)
    assert seed0 != seed1                        # independent replicas, distinct inputs


def test_single_process_is_identity():
    import bench
    assert bench.max_over_ranks(3.5) == 3.5
    assert bench.job_throughput(100, 4, 1, 2.0) == pytest.approx(200000.0)
