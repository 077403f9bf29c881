"""Rank bodies of the multi-process tests (spawned with gloo on CPU)."""
import os

import numpy as np


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
        top = D.gather_topk(glob, scores, w.k)
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
