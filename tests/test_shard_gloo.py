"""Pool sharding across ranks (world size 2 and 3, gloo on CPU): each rank
selects the top-q of its contiguous shard, the lists are all-gathered and
merged; the result must equal the single-pool top-q bit for bit."""
import os
import socket

import numpy as np
import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402

from conftest import ROOT  # noqa: E402


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, seed, n, q):
    import sys
    sys.path.insert(0, ROOT)
    import oracle as O
    from paper_2408_04323_gb300.shard import gather_topq, shard_range
    from workloads import Stream

    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        st = Stream(seed, "shard")
        acq = np.round(st.normal(n) * 3).astype(np.float32) / 3  # ties across shard borders
        acq[st.uniform(n) < 0.1] = -np.inf
        mask = st.uniform(n) < 0.8
        b, e = shard_range(n, rank, world)
        li, lv, lc = O.select_topq(acq[b:e], mask[b:e], q)
        idx = np.full(q, -1, np.int64)
        val = np.full(q, -np.inf, np.float32)
        idx[:lc] = li + b
        val[:lc] = acq[b:e][li]
        mi, mv = gather_topq(torch.from_numpy(idx), torch.from_numpy(val),
                             torch.tensor([lc], dtype=torch.int32), q)
        want, _, c = O.select_topq(acq, mask, q)
        assert mi.tolist() == want.tolist(), (rank, mi, want)
        assert np.array_equal(mv, acq[want])
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world,n,q", [(2, 1001, 4), (2, 7, 16), (3, 5000, 1), (2, 40000, 64)])
def test_sharded_topq_equals_single_pool(world, n, q):
    mp.spawn(_worker, args=(world, _free_port(), 17 + n + q, n, q), nprocs=world, join=True)


def test_shard_ranges_cover_the_pool():
    from paper_2408_04323_gb300.shard import shard_range
    for n in (0, 1, 5, 1000, 1001):
        for world in (1, 2, 3, 8):
            got = [shard_range(n, r, world) for r in range(world)]
            assert got[0][0] == 0 and got[-1][1] == n
            assert all(got[i][1] == got[i + 1][0] for i in range(world - 1))


def _mace_worker(rank, world, port, seed, n, k):
    import sys
    sys.path.insert(0, ROOT)
    import oracle as O
    from paper_2408_04323_gb300.shard import gather_mace_front, shard_range
    from workloads import Stream

    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        st = Stream(seed, "mace-shard")
        acq3 = np.floor(st.uniform(3 * n).reshape(3, n) * 6).astype(np.float32)  # ties and duplicates
        acq3[0, st.uniform(n) < 0.05] = -np.inf
        mask = st.uniform(n) < 0.9
        b, e = shard_range(n, rank, world)
        _, lfront, _ = O.mace_select(acq3[:, b:e], mask[b:e], k, seed)  # this rank's front (local indices)
        picks, front = gather_mace_front(torch.from_numpy(np.ascontiguousarray(acq3[:, b:e])),
                                         torch.from_numpy(lfront), len(lfront), b, k, seed)
        want_picks, want_front, _ = O.mace_select(acq3, mask, k, seed)
        assert front.tolist() == want_front.tolist(), (rank, front, want_front)
        assert picks.tolist() == want_picks.tolist(), (rank, picks, want_picks)
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world,n,k", [(2, 1001, 4), (3, 300, 64), (2, 5, 3), (3, 20000, 1)])
def test_sharded_mace_equals_single_pool(world, n, k):
    """Each rank's front of (UCB, PI, EI) over its shard is gathered and
    merged: the pool's front and the k random picks equal the single-pool
    selection (the oracle's mace_select), with ties, duplicates, -inf and
    masked candidates, and shards whose front is empty."""
    mp.spawn(_mace_worker, args=(world, _free_port(), 23 + n + k, n, k), nprocs=world, join=True)


def test_splitmix64_keys_match_the_oracle():
    import oracle as O
    from paper_2408_04323_gb300.shard import splitmix64_keys
    idx = np.array([0, 1, 2, 17, 1 << 20, (1 << 40) + 3])
    for seed in (0, 1, 0xDEADBEEFCAFEF00D):
        got = splitmix64_keys(seed, idx)
        assert [int(g) for g in got] == [O.splitmix64(seed, int(i)) for i in idx]


def _fantasy_worker(rank, world, port, name, seed, n, q):
    """One rank of the sharded sequential picks: the oracle scores this rank's
    shard at every step (GP refit on the observations and the fantasies so
    far, the fantasised front, picked candidates of the shard excluded); the
    ranks' records are all-gathered; every rank commits the best record and
    takes the pick's configuration from it alone."""
    import sys
    sys.path.insert(0, ROOT)
    import oracle as O
    from paper_2408_04323_gb300.shard import (best_record, decode_fantasy_record, encode_fantasy_record,
                                              gather_fantasy_records, selection_key, shard_range)
    from workloads import make_instance

    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        inst = make_instance(name, seed, n_cand=n)
        w = inst.workload
        words = inst.cand[:, :n]
        known = O.prune_mask(inst.space, inst.clauses, words, n)
        votes = O.rf_votes(inst.nodes, inst.tree_offset, inst.space, words, n)
        feas = known & O.pof_feasible(votes, inst.n_trees, w.leaf_scale, w.delta_num, w.delta_den)
        b, e = shard_range(n, rank, world)
        xw, yf = inst.x_obs, inst.y_obs.astype(np.float64)
        mine, picks = set(), []
        for j in range(q):
            gps = [O.GP(inst.space, xw, yf[m], inst.lengthscale[m], inst.signal_var[m], inst.noise_var[m])
                   for m in range(inst.n_obj)]
            rec = np.zeros(9, np.int64)
            if e > b:
                mv = [gp.posterior(np.ascontiguousarray(words[:, b:e])) for gp in gps]
                mu = np.stack([x for x, _ in mv], 1)
                var = np.stack([v for _, v in mv], 1)
                a = O.ehvi_mc(mu, var, inst.eps, O.pareto_front(yf.T, inst.ref), inst.ref)
                ok = feas[b:e].copy()
                ok[list(mine)] = False
                a = np.where(ok, a, -np.inf)
                if np.any(np.isfinite(a)):
                    a32 = a.astype(np.float32)  # the device's keys order fp32 values
                    k = int(np.flatnonzero(a32 == a32.max())[0])
                    rec = encode_fantasy_record(a32[k], b + k, words[:, b + k])
                    assert int(rec.view(np.uint64)[0]) == selection_key(a32[k], b + k)
            recs = gather_fantasy_records(torch.from_numpy(rec)).numpy()
            win = best_record(recs)
            if win < 0:
                break
            value, g, wds = decode_fantasy_record(recs[win], inst.d)
            assert np.array_equal(wds, words[:, g])  # the configuration travels in the record
            picks.append(int(g))
            if b <= g < e:
                mine.add(int(g) - b)
            # kriging believer from the record alone: the refit GP's mean at the pick
            mu_p = np.array([gp.posterior(wds[:, None].astype(np.uint32))[0][0] for gp in gps])
            xw = np.concatenate([xw, wds[:, None].astype(np.uint32)], axis=1)
            yf = np.concatenate([yf, mu_p[:, None]], axis=1)
        want = O.fantasy_picks(inst, q, feas)["picks"]
        assert picks == want, (rank, picks, want)
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world,name,n,q", [(2, "tiny", 301, 5), (3, "tiny", 240, 4), (3, "d8-ehvi2", 150, 3)])
def test_sharded_fantasy_picks_equal_single_pool(world, name, n, q):
    """The per-pick exchange of the sequential fantasised picks (one record
    per rank, the largest key wins, the configuration travels in the record)
    reproduces the single-pool pick sequence of the oracle."""
    from workloads import seeds
    mp.spawn(_fantasy_worker, args=(world, _free_port(), name, seeds(name)[1], n, q), nprocs=world, join=True)


def test_fantasy_record_round_trip():
    from paper_2408_04323_gb300.shard import (best_record, decode_fantasy_record, encode_fantasy_record,
                                              selection_key)
    words = np.array([7, 0xFFFFFFFF, 3, 12345, 0, 9, 1, 2, 3, 4, 5], np.uint32)
    rec = encode_fantasy_record(0.25, 4_000_000_000, words)
    v, g, w = decode_fantasy_record(rec, len(words))
    assert v == 0.25 and g == 4_000_000_000 and np.array_equal(w, words)
    # the order of keys is value descending, then index ascending; -0 == +0
    assert selection_key(1.0, 5) > selection_key(0.5, 1) > selection_key(-3.0, 0)
    assert selection_key(0.5, 1) > selection_key(0.5, 2)
    assert selection_key(-0.0, 3) == selection_key(0.0, 3)
    assert selection_key(float("nan"), 1) == 0 and selection_key(float("-inf"), 1) == 0
    recs = np.stack([encode_fantasy_record(0.5, 9, words), encode_fantasy_record(0.5, 2, words),
                     np.zeros(9, np.int64)])
    assert best_record(recs) == 1
    assert best_record(np.zeros((3, 9), np.int64)) == -1
    assert decode_fantasy_record(np.zeros(9, np.int64), 4) is None
