"""Host side of the multi-GPU path, on CPU: two gloo ranks on 127.0.0.1.

Each rank runs its own queries (weak scaling); the only cross-rank traffic
is the barrier and the max / sum of per-rank numbers that bench.py reports.
"""
import os
import socket

import pytest
import torch.multiprocessing as mp

from paper_2510_20064_gb300 import dist as hdist


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    r, w, lr = hdist.rank_info()
    assert (r, w, lr) == (rank, world, rank)
    hdist.init("gloo", w)
    hdist.barrier(w)
    t_max = hdist.max_over_ranks(1.5 + rank, w)
    total = hdist.sum_over_ranks(10 * (rank + 1), w)
    start, count = hdist.shard(13, r, w)
    hdist.barrier(w)
    hdist.finalize(w)
    out.put((rank, t_max, total, start, count, hdist.rank_seed(2000, r)))


def test_two_gloo_ranks():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    procs = [ctx.Process(target=_worker, args=(r, world, port, out)) for r in range(world)]
    for p in procs:
        p.start()
    res = sorted(out.get(timeout=120) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [r[1] for r in res] == [2.5, 2.5]          # slowest rank's time
    assert [r[2] for r in res] == [30.0, 30.0]
    assert [(r[3], r[4]) for r in res] == [(0, 7), (7, 6)]
    assert res[0][5] != res[1][5]                      # disjoint input streams


@pytest.mark.parametrize("B,world", [(1, 1), (8, 2), (13, 4), (128, 8), (3, 8)])
def test_shard_covers_every_query_once(B, world):
    seen = []
    for r in range(world):
        start, count = hdist.shard(B, r, world)
        seen.extend(range(start, start + count))
    assert seen == list(range(B))


def test_shard_rejects_bad_rank():
    with pytest.raises(ValueError):
        hdist.shard(8, 2, 2)
