"""Multi-GPU sharding of the candidate pool (host logic).

Candidates are independent, so a pool is split into contiguous index ranges,
one per rank, with the per-round state replicated.  The only exchange is the
final one: each rank's top-q (value, global index) pairs are gathered and
merged in the selection order of Section 4.7 (value descending, then index
ascending), which gives exactly the single-pool top-q.
"""
from __future__ import annotations

import numpy as np


def shard_range(n: int, rank: int, world: int) -> tuple[int, int]:
    """Contiguous [begin, end) of rank's share of n candidates."""
    per = -(-n // world)
    b = min(n, rank * per)
    return b, min(n, b + per)


def merge_topq(vals: np.ndarray, idxs: np.ndarray, counts: np.ndarray, q: int):
    """Merge per-rank top-q lists.

    vals, idxs: [world][q] (entries beyond counts[r] are ignored);
    returns (idx int64[k], val float32[k]) with k = min(q, sum(counts)).
    """
    vals = np.asarray(vals, np.float32)
    idxs = np.asarray(idxs, np.int64)
    pairs = []
    for r in range(vals.shape[0]):
        for j in range(int(counts[r])):
            pairs.append((float(vals[r, j]), int(idxs[r, j])))
    pairs.sort(key=lambda p: (-p[0], p[1]))
    pairs = pairs[:q]
    return (np.array([p[1] for p in pairs], np.int64),
            np.array([p[0] for p in pairs], np.float32))


def gather_topq(idx, val, count, q: int, group=None):
    """All-gather the ranks' top-q lists (torch.distributed) and merge them.

    idx/val/count are this rank's results (tensors on the process group's
    device type); returns the merged (idx, val) as numpy arrays.
    """
    import torch
    import torch.distributed as dist
    world = dist.get_world_size(group)
    vals = [torch.empty_like(val) for _ in range(world)]
    idxs = [torch.empty_like(idx) for _ in range(world)]
    cnts = [torch.empty_like(count) for _ in range(world)]
    dist.all_gather(vals, val, group=group)
    dist.all_gather(idxs, idx, group=group)
    dist.all_gather(cnts, count, group=group)
    V = torch.stack(vals).cpu().numpy()
    I = torch.stack(idxs).cpu().numpy()
    C = torch.stack(cnts).cpu().numpy().reshape(-1)
    return merge_topq(V, I, C, q)
