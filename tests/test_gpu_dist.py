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


def _merge_case(rng, m, k, pad_frac=0.2, tie_frac=0.3):
    scores = rng.normal(size=m).astype(np.float32)
    ties = rng.random(m) < tie_frac
    scores[ties] = np.float32(0.5)  # many equal scores: order by global index
    scores[rng.random(m) < 0.05] = np.float32(-0.0)
    scores[rng.random(m) < 0.05] = np.float32(0.0)
    idx = rng.choice(1 << 40, size=m, replace=False).astype(np.int64)  # distinct, past 2^32
    idx[rng.random(m) < pad_frac] = -1
    return scores, idx


@pytest.mark.parametrize("m,k", [(0, 5), (1, 1), (7, 20), (2048, 1024), (8 * 1024, 1024), (16 * 2048, 2048),
                                 (5000, 16384), (262144, 64)])
def test_device_merge_matches_the_oracle_order(m, k):
    """mlt_merge_topk: the k best of m (score, global index) pairs by (score
    desc, index asc), -0 equal to +0, empty slots skipped, -1 padded."""
    import torch

    from paper_2411_10764_gb300 import mlt
    from dist_ranks import oracle_merge

    rng = np.random.default_rng(m + k)
    scores, idx = _merge_case(rng, m, k)
    got = mlt.merge_topk(torch.from_numpy(scores).cuda(), torch.from_numpy(idx).cuda(), k)
    mlt.sync_status()
    assert np.array_equal(got.cpu().numpy(), oracle_merge(scores, idx, k))
