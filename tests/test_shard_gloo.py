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
