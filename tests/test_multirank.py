"""Host logic of the multi-GPU bench path, on CPU with gloo (world size 2).

The update path does not shard (episodes are independent), so N GPUs run N
replicas with no data-path collective; the only cross-rank step is the
timing reduction: the slowest rank decides, and the value sums the replicas.
"""
import os
import socket

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    got = bench.max_over_ranks([10.0 + rank, 5.0 - rank], dist, "cpu")
    q.put((rank, got))
    dist.barrier()
    dist.destroy_process_group()


def test_max_over_ranks_gloo():
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    results = dict(q.get(timeout=120) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for r in range(world):
        assert results[r] == [11.0, 5.0]


def test_replica_throughput():
    import bench
    # 2 replicas x 10 updates x 2048 tokens in 20 ms
    assert bench.replica_throughput(2048, 10, 2, 20.0) == pytest.approx(2048 * 10 * 2 / 0.02)
    assert bench.replica_throughput(2048, 10, 1, 20.0) == pytest.approx(2048 * 10 / 0.02)
