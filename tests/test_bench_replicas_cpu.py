"""The benchmark's multi-rank path on CPU: two gloo ranks, each timing its own
replica, aggregate to the whole-job throughput of the slowest rank."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, out):
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    # rank r pretends its timed region took 100 * (r + 1) ms and 2 * (r + 1) ms per e2e step
    tok, e2e, job_ms = bench.aggregate_replicas(100.0 * (rank + 1), 0.002 * (rank + 1), batch=1, steps=50)
    out[rank] = (tok, e2e, job_ms)
    dist.barrier()
    dist.destroy_process_group()


@pytest.mark.parametrize("world", [2])
def test_aggregate_replicas_takes_the_slowest_rank(world):
    port = _free_port()
    manager = mp.Manager()
    out = manager.dict()
    mp.spawn(_worker, args=(world, port, out), nprocs=world, join=True)
    for r in range(world):
        tok, e2e, job_ms = out[r]
        assert job_ms == 100.0 * world                        # max over ranks
        assert tok == pytest.approx(world * 1 * 50 / (job_ms / 1e3))
        assert e2e == pytest.approx(world / (0.002 * world))


def test_aggregate_single_process():
    import bench
    tok, e2e, job_ms = bench.aggregate_replicas(200.0, 0.004, batch=2, steps=100)
    assert job_ms == 200.0 and tok == pytest.approx(2 * 100 / 0.2) and e2e == pytest.approx(2 / 0.004)
