"""Rank bodies of the multi-process tests (spawned with gloo on CPU)."""
import os

import numpy as np


def oracle_merge(scores, indices, k):
    """The oracle's order over (score, global index) pairs: pairs sorted by
    index, then the oracle's top-k (score descending, position ascending),
    so positions order like global indices.  Negative indices are empty."""
    import oracle as O

    scores = np.asarray(scores, np.float32).reshape(-1)
    indices = np.asarray(indices, np.int64).reshape(-1)
    keep = indices >= 0
    order = np.argsort(indices[keep], kind="stable")
    s, i = scores[keep][order], indices[keep][order]
    tk, _ = O.topk(s, np.ones(s.size, bool), k)
    return np.where(tk >= 0, i[np.maximum(tk, 0)] if i.size else -1, -1)


def merge_rank(rank, world, port, cid, n, seed, results):
    import torch.distributed as dist

    import oracle as O
    from paper_2411_10764_gb300 import dist as D
    from paper_2411_10764_gb300 import workloads as W

    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        w = W.make_workload(cid, seed=seed, n=n)
        a, b = D.shard_bounds(w.n, rank, world)
        # this rank's shard, screened by the oracle (no GPU here); the
        # exchange and merge under test are the same ones the GPU path uses
        _, pf, valid, _ = O.screen_rows(w.feats[a:b], w.v, w.p, w.thr)
        loc, _ = O.topk(pf, valid, w.k)
        glob = np.where(loc >= 0, loc + a, -1)
        scores = np.where(loc >= 0, pf[np.maximum(loc, 0)] if pf.size else -np.inf, -np.inf)
        # no GPU here: the oracle stands in for the library's merge
        top = D.gather_topk(glob, scores, w.k, merge=oracle_merge)
        results[rank] = top.tolist()
    finally:
        dist.destroy_process_group()


def gpu_shard_rank(rank, world, port, cid, n, seed, results):
    """Each rank screens its shard with the CUDA library on cuda:0 and the
    ranks exchange their top-k over gloo (host memory; no device waits)."""
    import torch
    import torch.distributed as dist

    from paper_2411_10764_gb300 import dist as D
    from paper_2411_10764_gb300 import mlt
    from paper_2411_10764_gb300 import workloads as W

    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        torch.cuda.set_device(0)
        w = W.make_workload(cid, seed=seed, n=n)
        mlt.load_workload_models(w)
        a, b = D.shard_bounds(w.n, rank, world)
        x = torch.from_numpy(np.ascontiguousarray(w.feats[a:b])).cuda()
        _, pf, top = D.screen_shard(x, w.thr, w.k, a)
        mlt.sync_status()
        results[rank] = (top.tolist(), pf.cpu().numpy().view(np.uint32).tolist())
    finally:
        dist.destroy_process_group()
