"""Multi-GPU sharding of the candidate pool (host logic).

Candidates are independent, so a pool is split into contiguous index ranges,
one per rank, with the per-round state replicated.  The only exchange is the
final one: each rank's top-q (value, global index) pairs are gathered and
merged in the selection order of Section 4.7 (value descending, then index
ascending), which gives exactly the single-pool top-q.  For MACE (Sections
4.5 and 4.7) each rank's Pareto front of (UCB, PI, EI) is gathered instead:
a candidate is on the pool's front iff it is on its rank's front and no
other rank's front member dominates it, and the random k-subset is drawn
with the same keys (SplitMix64 of the global index) as on one GPU, so the
picks equal the single-pool picks.
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


_SM_GAMMA = np.uint64(0x9E3779B97F4A7C15)


def splitmix64_keys(seed: int, idx: np.ndarray) -> np.ndarray:
    """Output idx (0-based) of the SplitMix64 generator seeded with seed, for
    every entry of idx: the draw keys of the Pareto selection."""
    i = np.asarray(idx, np.int64).astype(np.uint64)
    with np.errstate(over="ignore"):
        z = np.uint64(seed & 0xFFFFFFFFFFFFFFFF) + (i + np.uint64(1)) * _SM_GAMMA
        z = (z ^ (z >> np.uint64(30))) * np.uint64(0xBF58476D1CE4E5B9)
        z = (z ^ (z >> np.uint64(27))) * np.uint64(0x94D049BB133111EB)
        return z ^ (z >> np.uint64(31))


def merge_mace_fronts(triples: np.ndarray, idxs: np.ndarray, counts: np.ndarray, k: int, seed: int):
    """Merge per-rank Pareto fronts of (UCB, PI, EI).

    triples: [world][cap][3] float32 (each front member's values), idxs:
    [world][cap] global indices, counts: members per rank.  Returns (picks
    int64[min(k, F)] in draw order, the pool's front int64[F] ascending)."""
    T = np.concatenate([np.asarray(triples[r][:int(counts[r])], np.float32) for r in range(len(counts))])
    I = np.concatenate([np.asarray(idxs[r][:int(counts[r])], np.int64) for r in range(len(counts))])
    if len(I) == 0:
        return np.zeros(0, np.int64), np.zeros(0, np.int64)
    ge = np.all(T[:, None, :] >= T[None, :, :], axis=2)   # ge[j, i]: T_j >= T_i everywhere
    gt = np.any(T[:, None, :] > T[None, :, :], axis=2)
    dominated = np.any(ge & gt, axis=0)
    front = I[~dominated]
    keys = splitmix64_keys(seed, front)
    order = np.lexsort((front, keys))  # key ascending, then index ascending
    return front[order][:k], np.sort(front)


def gather_mace_front(acq3, front_idx, front_count: int, base: int, k: int, seed: int, group=None):
    """All-gather the ranks' fronts (torch.distributed) and merge them.

    acq3: this rank's [3][lda] (UCB, PI, EI) tensor; front_idx: its front's
    local indices (front_count of them, as scoot_select_pareto writes them);
    base: the global index of its first candidate.  Returns (picks, front)
    as numpy arrays of global indices."""
    import torch
    import torch.distributed as dist
    world = dist.get_world_size(group)
    cnt = torch.tensor([int(front_count)], dtype=torch.int64, device=acq3.device)
    cnts = [torch.empty_like(cnt) for _ in range(world)]
    dist.all_gather(cnts, cnt, group=group)
    C = torch.stack(cnts).cpu().numpy().reshape(-1)
    cap = max(1, int(C.max()))
    loc = front_idx[:int(front_count)].to(torch.int64)
    tri = torch.full((cap, 3), -float("inf"), dtype=torch.float32, device=acq3.device)
    gid = torch.full((cap,), -1, dtype=torch.int64, device=acq3.device)
    if int(front_count):
        tri[:int(front_count)] = acq3[:, loc].t().to(torch.float32)
        gid[:int(front_count)] = loc + int(base)
    tris = [torch.empty_like(tri) for _ in range(world)]
    gids = [torch.empty_like(gid) for _ in range(world)]
    dist.all_gather(tris, tri, group=group)
    dist.all_gather(gids, gid, group=group)
    return merge_mace_fronts(torch.stack(tris).cpu().numpy(), torch.stack(gids).cpu().numpy(), C, k, seed)
