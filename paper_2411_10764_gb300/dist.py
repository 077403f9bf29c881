"""Screening one candidate batch across several GPUs (one process per GPU).

Candidates are independent, so a batch shards by contiguous index ranges:
rank r screens [r*n/G, (r+1)*n/G) with the library on its own GPU, keeps its
local top-k, and one exchange of k (score, index) pairs per rank gives every
rank the global top-k.  The merge uses the same total order as the library
(score descending, then global index ascending), so the result equals
screening the whole batch on one device.  ML^2Tuner Sec. 2: the explorer keeps
the candidates P ranks best; nothing else crosses ranks.
"""
from __future__ import annotations

import numpy as np

from . import mlt


def shard_bounds(n: int, rank: int, world: int) -> tuple[int, int]:
    """Contiguous index range of rank `rank` out of `world`."""
    return n * rank // world, n * (rank + 1) // world


def gather_topk(local_indices, local_scores, k: int, group=None, merge=None):
    """Exchange every rank's local top-k and return the global top-k (on all
    ranks) as a numpy int64 array.  Works with any torch.distributed backend;
    the exchanged tensors live on the backend's device (CPU for gloo, the
    current GPU for nccl).  The merge runs in the library on the current GPU
    (mlt_merge_topk: score descending, then global index ascending, -1
    padded); `merge(scores, indices, k)` replaces it where no GPU is present
    (the CPU multi-process tests)."""
    import torch
    import torch.distributed as dist

    backend = dist.get_backend(group)
    device = torch.device("cuda", torch.cuda.current_device()) if backend == "nccl" else torch.device("cpu")
    idx = torch.full((int(k),), -1, dtype=torch.int64, device=device)
    sc = torch.full((int(k),), float("-inf"), dtype=torch.float32, device=device)
    li = torch.as_tensor(np.asarray(local_indices, dtype=np.int64).reshape(-1)[:k])
    ls = torch.as_tensor(np.asarray(local_scores, dtype=np.float32).reshape(-1)[:k])
    idx[: li.numel()] = li.to(device)
    sc[: ls.numel()] = ls.to(device)
    world = dist.get_world_size(group)
    all_idx = [torch.empty_like(idx) for _ in range(world)]
    all_sc = [torch.empty_like(sc) for _ in range(world)]
    dist.all_gather(all_idx, idx, group=group)
    dist.all_gather(all_sc, sc, group=group)
    cat_sc, cat_idx = torch.cat(all_sc), torch.cat(all_idx)
    if merge is not None:
        return np.asarray(merge(cat_sc.cpu().numpy(), cat_idx.cpu().numpy(), int(k)), dtype=np.int64)
    gpu = torch.device("cuda", torch.cuda.current_device())
    top = mlt.merge_topk(cat_sc.to(gpu), cat_idx.to(gpu), int(k))
    return top.cpu().numpy()


def screen_shard(feats_shard, thr: float, k: int, index_base: int, group=None, stream=None):
    """Screen this rank's shard (a CUDA [n_r][F] tensor holding candidates
    index_base .. index_base+n_r-1) and return (pvalid, perf, global top-k)."""
    import torch

    pv, pf, tk = mlt.screen(feats_shard, thr, k, stream=stream)
    if pf.numel() == 0:
        scores = torch.full(tk.shape, float("-inf"), dtype=torch.float32, device=tk.device)
    else:
        local = tk.clamp_min(0)
        scores = torch.where(tk >= 0, pf[local], torch.full_like(pf[local], float("-inf")))
    glob = torch.where(tk >= 0, tk + int(index_base), tk)
    top = gather_topk(glob.cpu().numpy(), scores.cpu().numpy(), k, group=group)
    return pv, pf, top
