"""Sharding one batch over ranks: local top-k per shard, one k-sized
all-gather, merge by (score desc, index asc) -- equals the oracle's top-k of
the whole batch.  World size 2 (and 3, uneven shards) with gloo on CPU; the
library's device merge (mlt_merge_topk) is checked on the GPU in
test_gpu_dist.py, so here the oracle's order stands in for it."""
import multiprocessing as mp
import socket

import numpy as np
import pytest

import oracle as O
from paper_2411_10764_gb300 import dist as D
from paper_2411_10764_gb300 import workloads as W
import dist_ranks


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def test_shard_bounds_cover_the_batch():
    for n in [0, 1, 7, 1000, 65537]:
        for world in [1, 2, 3, 8]:
            b = [D.shard_bounds(n, r, world) for r in range(world)]
            assert b[0][0] == 0 and b[-1][1] == n
            assert all(b[i][1] == b[i + 1][0] for i in range(world - 1))


def test_oracle_merge_breaks_ties_across_ranks_by_global_index():
    scores = np.array([2.0, 1.0, -0.0, 2.0, 0.0, 5.0], np.float32)
    idx = np.array([10, 11, 12, 3, 4, -1])
    assert dist_ranks.oracle_merge(scores, idx, 6).tolist() == [3, 10, 11, 4, 12, -1]


@pytest.mark.parametrize("world,cid,n", [(2, 2, 5000), (3, 1, 4001)])
def test_gloo_ranks_merge_to_the_global_topk(world, cid, n):
    ctx = mp.get_context("spawn")
    with ctx.Manager() as mgr:
        results = mgr.dict()
        port = _free_port()
        procs = [ctx.Process(target=dist_ranks.merge_rank, args=(r, world, port, cid, n, 5, results))
                 for r in range(world)]
        for p in procs:
            p.start()
        for p in procs:
            p.join(timeout=180)
            assert p.exitcode == 0
        got = [results[r] for r in range(world)]
    w = W.make_workload(cid, seed=5, n=n)
    _, pf, valid, _ = O.screen_rows(w.feats, w.v, w.p, w.thr)
    want, _ = O.topk(pf, valid, w.k)
    for r in range(world):
        assert got[r] == want.tolist()
