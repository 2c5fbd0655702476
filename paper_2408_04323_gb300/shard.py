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

The sequential fantasised picks exchange once per pick: every rank's best
candidate of the pass (its record: selection key with the global index and
the candidate's configuration words) is all-gathered, and every rank commits
the record with the largest key, computing the pick's rank-1 terms from the
configuration it carries; no rank needs another rank's pool.
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


# ------------------------------------------------------------------ sequential fantasised picks

FANT_REC = 9  # 64-bit words of a record (include/scoot.h, SCOOT_FANT_REC)


def selection_key(value: float, global_index: int) -> int:
    """The 64-bit selection key of Section 4.7's order (the device's make_key):
    order-preserving bits of the fp32 value (-0 as +0) in the high word,
    0xFFFFFFFF - index in the low word; 0 for NaN and -inf (never selected)."""
    v = np.float32(value)
    if np.isnan(v) or v == -np.inf:
        return 0
    b = int(np.array([v], np.float32).view(np.uint32)[0])
    if b == 0x80000000:
        b = 0
    b = (~b & 0xFFFFFFFF) if b & 0x80000000 else (b | 0x80000000)
    return (b << 32) | (0xFFFFFFFF - int(global_index))


def encode_fantasy_record(value: float, global_index: int, words) -> np.ndarray:
    """A shard's record as the device writes it (int64 view of the uint64
    words): the key, then the configuration words two per element."""
    rec = np.zeros(FANT_REC, np.uint64)
    key = selection_key(value, global_index)
    rec[0] = np.uint64(key)
    if key:
        w = np.zeros(2 * (FANT_REC - 1), np.uint32)
        w[:len(words)] = np.asarray(words, np.uint32)
        rec[1:] = w.view(np.uint64)
    return rec.view(np.int64)


def decode_fantasy_record(rec, d: int):
    """(value, global index, words) of a record, or None for key 0."""
    r = np.asarray(rec).view(np.uint64)
    key = int(r[0])
    if key == 0:
        return None
    b = key >> 32
    b = (b & 0x7FFFFFFF) if b & 0x80000000 else (~b & 0xFFFFFFFF)
    value = float(np.array([b], np.uint32).view(np.float32)[0])
    return value, 0xFFFFFFFF - (key & 0xFFFFFFFF), r[1:].view(np.uint32)[:d].copy()


def best_record(recs) -> int:
    """Row of the record with the largest (unsigned) key, -1 if every key is 0."""
    keys = np.asarray(recs).view(np.uint64)[:, 0]
    k = int(np.argmax(keys))
    return k if keys[k] != 0 else -1


def gather_fantasy_records(rec, group=None):
    """All ranks' records ([world][FANT_REC], same device as rec)."""
    import torch
    import torch.distributed as dist
    world = dist.get_world_size(group)
    parts = [torch.empty_like(rec.reshape(-1)) for _ in range(world)]
    dist.all_gather(parts, rec.reshape(-1).contiguous(), group=group)
    return torch.stack(parts)


def sharded_fantasy_picks(S, ctx, layout, state, fant_state, box_cap, cand, n, eps, q, work, idx, val, count,
                          index_offset, mask=None, var_out=None, group=None, stream=None):
    """q sequential fantasised picks over a pool sharded across the ranks of
    `group`: this rank holds candidates index_offset .. index_offset + n - 1.
    One all-gather of the ranks' records per pick; idx, val, count (device)
    end up identical on every rank and equal to the single-pool picks."""
    import torch
    S.scoot_fantasy_begin(ctx, layout, state, fant_state, box_cap, cand, n, eps, q, work, idx, val, count, mask=mask,
                          index_offset=index_offset, stream=stream)
    rec = torch.zeros(FANT_REC, dtype=torch.int64, device=idx.device)
    for j in range(q):
        S.scoot_fantasy_local_best(ctx, j, rec, stream)
        S.scoot_fantasy_commit(ctx, j, gather_fantasy_records(rec, group), stream)
    S.scoot_fantasy_end(ctx, var_out, stream)
