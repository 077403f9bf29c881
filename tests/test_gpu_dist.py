"""One batch screened as shards by two processes sharing cuda:0, top-k
exchanged over gloo: equals the oracle's top-k of the whole batch, and each
shard's P scores equal the oracle's bit for bit."""
import multiprocessing as mp
import socket

import numpy as np
import pytest

import oracle as O
from paper_2411_10764_gb300 import dist as D
from paper_2411_10764_gb300 import workloads as W
import dist_ranks

pytestmark = pytest.mark.gpu


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def test_two_gpu_processes_shard_and_merge():
    world, cid, n = 2, 2, 20001
    ctx = mp.get_context("spawn")
    with ctx.Manager() as mgr:
        results = mgr.dict()
        port = _free_port()
        procs = [ctx.Process(target=dist_ranks.gpu_shard_rank, args=(r, world, port, cid, n, 9, results))
                 for r in range(world)]
        for p in procs:
            p.start()
        for p in procs:
            p.join(timeout=300)
            assert p.exitcode == 0
        got = {r: results[r] for r in range(world)}
    w = W.make_workload(cid, seed=9, n=n)
    _, pf, valid, _ = O.screen_rows(w.feats, w.v, w.p, w.thr)
    want, _ = O.topk(pf, valid, w.k)
    for r in range(world):
        top, perf_bits = got[r]
        assert top == want.tolist()
        a, b = D.shard_bounds(n, r, world)
        assert np.array_equal(np.array(perf_bits, np.uint32), pf[a:b].view(np.uint32))
