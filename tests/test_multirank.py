"""The multi-rank (replica) logic of bench.py on CPU: two gloo ranks.

The hot path shards by request: every rank serves its own requests and only
the timing is reduced (maximum over ranks); no data-path collective exists.
"""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    r, local, w = bench.rank_env()
    ms = bench.max_over_ranks(10.0 + 5.0 * rank, w)     # rank 1 is the slower one
    first = bench.rank_first_sample(r, 1)
    seeds = [int(t) for t in torch.tensor([first])]
    gathered = [torch.zeros(1, dtype=torch.int64) for _ in range(w)]
    dist.all_gather(gathered, torch.tensor(seeds))
    out[rank] = (r, local, w, ms, [int(g) for g in gathered],
                 bench.job_throughput(w, 4, 1, 10, ms))
    dist.destroy_process_group()


def test_two_gloo_ranks_shard_requests_and_take_the_slowest_time():
    world = 2
    port = _free_port()
    with mp.Manager() as mgr:
        out = mgr.dict()
        mp.spawn(_worker, args=(world, port, out), nprocs=world, join=True)
        res = dict(out)
    for rank in range(world):
        r, local, w, ms, firsts, value = res[rank]
        assert (r, local, w) == (rank, rank, world)
        assert ms == 15.0                       # maximum over ranks
        assert sorted(firsts) == [0, 1]          # disjoint requests per rank
        assert value == pytest.approx(2 * 4 * 10 / 0.015)


def test_single_process_defaults(monkeypatch):
    import bench
    for k in ("RANK", "WORLD_SIZE", "LOCAL_RANK"):
        monkeypatch.delenv(k, raising=False)
    assert bench.rank_env() == (0, 0, 1)
    assert bench.max_over_ranks(7.5, 1) == 7.5
