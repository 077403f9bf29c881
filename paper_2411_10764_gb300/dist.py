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


def merge_topk(scores, indices, k: int) -> np.ndarray:
    """Global top-k from the concatenated per-rank lists.

    `indices` are global candidate indices (-1 marks an empty slot) and
    `scores` their P scores.  Returns k indices, -1 padded."""
    scores = np.asarray(scores, dtype=np.float32).reshape(-1)
    indices = np.asarray(indices, dtype=np.int64).reshape(-1)
    keep = indices >= 0
    s, i = scores[keep], indices[keep]
    order = np.lexsort((i, -s.astype(np.float64)))
    out = np.full(int(k), -1, dtype=np.int64)
    m = min(int(k), order.size)
    out[:m] = i[order[:m]]
    return out


def gather_topk(local_indices, local_scores, k: int, group=None) -> np.ndarray:
    """Exchange every rank's local top-k and return the global top-k (on all
    ranks).  Works with any torch.distributed backend; tensors live on the
    backend's device (CPU for gloo, the current GPU for nccl)."""
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
    return merge_topk(torch.cat(all_sc).cpu().numpy(), torch.cat(all_idx).cpu().numpy(), k)


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
