"""Host logic of the multi-GPU bench path, on CPU with two gloo ranks.

Each rank runs an independent replica of the layer; the bench reports the
tokens of all ranks divided by the slowest rank's time, after a barrier."""
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


def _worker(rank, world, port, q):
    os.environ.update({"MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port), "RANK": str(rank),
                       "WORLD_SIZE": str(world), "LOCAL_RANK": str(rank)})
    import torch.distributed as dist
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    bench.dist_barrier(world)
    tokens, secs = bench.aggregate(world, 64 * 10, 0.5 + rank)   # rank 1 is slower
    q.put((rank, tokens, secs))
    dist.destroy_process_group()


def test_two_rank_aggregation_takes_total_tokens_and_max_time():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    res = sorted(q.get(timeout=10) for _ in range(2))
    for rank, tokens, secs in res:
        assert tokens == 2 * 64 * 10
        assert secs == pytest.approx(1.5)
