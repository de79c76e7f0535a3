"""The multi-GPU (replica) bookkeeping of bench.py, run as world-size-2 gloo
ranks on the CPU: barrier, max over ranks of the elapsed time, sum of the
launch counts, whole-job throughput.  No GPU and no data-path collective."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, results):
    import torch.distributed as dist
    os.environ.update({"MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port), "RANK": str(rank),
                       "WORLD_SIZE": str(world), "LOCAL_RANK": str(rank)})
    dist.init_process_group("gloo", rank=rank, world_size=world)
    from paper_2609_30057_gb300 import replicas
    r, w, lr = replicas.rank_world()
    replicas.barrier(dist)
    elapsed = 1.0 + 0.5 * rank                     # rank 1 is the slow replica
    slowest = replicas.max_over_ranks(dist, elapsed)
    launches = replicas.sum_over_ranks(dist, 100 + rank)
    value = replicas.aggregate_throughput(20, w, slowest)
    results[rank] = (r, w, lr, slowest, launches, value)
    dist.destroy_process_group()


def test_two_replicas_aggregate_over_gloo():
    world = 2
    port = _free_port()
    with mp.get_context("spawn").Manager() as m:   # no fork of a threaded process
        results = m.dict()
        mp.spawn(_rank_main, args=(world, port, results), nprocs=world, join=True)
        res = dict(results)
    for rank in range(world):
        r, w, lr, slowest, launches, value = res[rank]
        assert (r, w, lr) == (rank, world, rank)
        assert slowest == 1.5                       # every rank sees the slowest time
        assert launches == 201
        assert value == pytest.approx(20 * 2 / 1.5)


def test_single_process_defaults(monkeypatch):
    from paper_2609_30057_gb300 import replicas
    for k in ("RANK", "WORLD_SIZE", "LOCAL_RANK"):
        monkeypatch.delenv(k, raising=False)
    assert replicas.rank_world() == (0, 1, 0)
    assert replicas.max_over_ranks(None, 2.5) == 2.5
    assert replicas.aggregate_throughput(10, 1, 2.0) == 5.0
    with pytest.raises(ValueError):
        replicas.aggregate_throughput(10, 1, 0.0)
