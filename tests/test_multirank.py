"""The N > 1 path of bench.py on CPU: two gloo ranks run replicas on
different sequences and agree on the job time (max over ranks)."""

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
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import torch.distributed as dist
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    local_ms = 10.0 + 5.0 * rank  # rank 1 is the slow one
    ms, us = bench.aggregate(local_ms, steps=5, batch=2, world=world)
    dist.barrier()
    q.put((rank, ms, us, bench.replica_seed(7, rank), bench._dist()))
    dist.destroy_process_group()


def test_two_rank_aggregation_and_replica_seeds():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    (r0, ms0, us0, s0, d0), (r1, ms1, us1, s1, d1) = out
    assert ms0 == ms1 == pytest.approx(15.0 / 5)       # max over ranks
    assert us0 == us1 == pytest.approx(3.0 * 1e3 / (2 * 2))
    assert s0 != s1                                     # independent sequences
    assert d0 == (0, 2, 0) and d1 == (1, 2, 1)
