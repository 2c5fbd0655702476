"""CART training of the feasibility forest (Algorithm 1's TRAIN, Section 4.6)
through the C ABI, against the oracle's breadth-first CART.

Bar: trees are integer/structural results (split feature, child index, leaf
flag, integer votes) and float32 thresholds that are copies of sample
values, so every node record must be identical, bit for bit.  The oracle
trains one tree in pure Python, so full-size forests are checked on a
sample of their trees (each tree is an independent block on the GPU); the
trained forest is also packed and evaluated by the forest kernel.
"""
import numpy as np
import pytest

import oracle as O
from workloads import CATEGORICAL, CONTINUOUS, INT_UNIFORM, PARAM_DTYPE, Stream, make_instance, seeds

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def S():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2408_04323_gb300 as pkg
    pkg.build()
    from paper_2408_04323_gb300 import scoot
    return scoot


@pytest.fixture(scope="module")
def ctx(S):
    c = S.Context(0)
    yield c
    c.close()


def _space(kinds):
    sp = np.zeros(len(kinds), PARAM_DTYPE)
    for i, k in enumerate(kinds):
        sp[i]["kind"] = k
        sp[i]["n_choices"] = 4 if k == CATEGORICAL else 0
        sp[i]["lo"], sp[i]["hi"] = (0, 1) if k == CONTINUOUS else (0, 1000)
    return sp


def _train_gpu(S, ctx, space, words, labels, boot, max_depth, leaf_scale, node_cap=None):
    T, m = boot.shape
    n = len(labels)
    ld = max(4, -(-n // 4) * 4)
    obs = np.zeros((len(space), ld), np.uint32)
    obs[:, :n] = words[:, :n]
    cap = 2 * m - 1 if node_cap is None else node_cap
    nodes = torch.full((max(T, 1), cap), -1, dtype=torch.int64, device="cuda")
    cnt = torch.full((max(T, 1),), -1, dtype=torch.int32, device="cuda")
    S.scoot_rf_train(ctx, space, torch.from_numpy(obs.view(np.int32)).cuda(), n,
                     torch.from_numpy(labels.astype(np.uint8)).cuda(),
                     torch.from_numpy(boot.astype(np.int32)).cuda(), max_depth, leaf_scale, nodes, cnt)
    torch.cuda.synchronize()
    return nodes.cpu().numpy()[:T], cnt.cpu().numpy()[:T]


def _check_trees(S, nodes, cnt, feats, labels, boot, max_depth, leaf_scale, trees):
    """Compares trees `trees` with the oracle's; returns the oracle's trees."""
    recs = nodes.view(S.NODE_DTYPE)
    out = []
    for t in trees:
        want, _ = O.train_forest(feats, labels, boot[t:t + 1], max_depth, leaf_scale)
        out.append(want)
        got = recs[t, :int(cnt[t])]
        assert int(cnt[t]) == len(want), f"tree {t}: {int(cnt[t])} nodes, oracle {len(want)}"
        for f in ("val", "left", "feat", "flags"):
            a, b = got[f], want[f]
            if f == "val":
                a, b = a.view(np.uint32), b.view(np.uint32)
            assert np.array_equal(a, b), f"tree {t} field {f}: first difference at node {np.argmax(a != b)}"
    return out


def _expect_status(S, ctx, status):
    with pytest.raises(S.ScootError) as e:
        ctx.check()
    assert e.value.status == status


def _feats(space, words, n):
    return O.decode(space, words, n).astype(np.float32)


@pytest.mark.parametrize("n,m,d,card,p,max_depth,leaf_scale,T", [
    (1, 1, 1, 5, 0.5, 6, 255, 3),
    (2, 2, 3, 2, 0.5, 6, 255, 8),
    (7, 11, 2, 3, 0.5, 255, 1, 8),
    (33, 33, 16, 4, 0.4, 255, 255, 6),
    (64, 64, 5, 1000, 0.7, 0, 255, 4),
    (64, 64, 5, 1000, 0.7, 1, 1000, 4),
    (100, 100, 8, 6, 0.3, 10, 255, 12),
    (200, 150, 12, 50, 0.5, 14, 255, 5),
    (50, 50, 4, 3, 1.0, 8, 255, 3),
    (50, 50, 4, 3, 0.0, 8, 255, 3),
])
def test_rf_train_matches_oracle(S, ctx, n, m, d, card, p, max_depth, leaf_scale, T):
    """Random mixed spaces; low-cardinality features force ties in values and
    in split costs."""
    st = Stream(n * 1000 + d * 10 + max_depth, "rf-train")
    kinds = [(INT_UNIFORM, CATEGORICAL, CONTINUOUS)[j % 3] for j in range(d)]
    space = _space(kinds)
    words = np.zeros((d, n), np.uint32)
    for j, k in enumerate(kinds):
        v = st.integers(0, card - 1, n)
        if k == CONTINUOUS:
            words[j] = (v.astype(np.float32) / np.float32(card) - np.float32(0.25)).view(np.uint32)
        else:
            words[j] = (v - (card // 2 if k == INT_UNIFORM else 0)).astype(np.int32).view(np.uint32)
    labels = (st.uniform(n) < p).astype(np.uint8)
    boot = st.integers(0, n - 1, T * m).reshape(T, m)
    nodes, cnt = _train_gpu(S, ctx, space, words, labels, boot, max_depth, leaf_scale)
    ctx.check()
    _check_trees(S, nodes, cnt, _feats(space, words, n), labels, boot, max_depth, leaf_scale, range(T))
    print(f"[parity] rf_train n={n} m={m} d={d}: {T} trees, {int(cnt.sum())} nodes identical")


def test_rf_train_maximum_size(S, ctx):
    """n = m = 1024 observations (the limit), two features of few values."""
    n = m = 1024
    st = Stream(7, "rf-train-max")
    space = _space([INT_UNIFORM, CATEGORICAL])
    words = np.stack([st.integers(0, 9, n), st.integers(0, 3, n)]).astype(np.uint32)
    labels = (st.uniform(n) < 0.5).astype(np.uint8)
    boot = st.integers(0, n - 1, 2 * m).reshape(2, m)
    nodes, cnt = _train_gpu(S, ctx, space, words, labels, boot, 255, 255)
    _check_trees(S, nodes, cnt, _feats(space, words, n), labels, boot, 255, 255, range(2))


@pytest.mark.parametrize("name,sample", [("d8-ehvi2", 6), ("d12-fantasy", 3)])
def test_rf_train_workload(S, ctx, name, sample):
    """The workload's observations, crash labels and forest shape (trees,
    depth limit, bootstrap of n draws): all trees trained, a sample compared
    with the oracle, and the forest packed and evaluated on the pool agrees
    with the oracle's votes from the oracle's trees."""
    inst = make_instance(name, seeds(name)[0], n_cand=4096)
    w = inst.workload
    n = w.n_obs
    labels = (inst.label_obs > 0.5).astype(np.uint8)
    st = Stream(seeds(name)[0], "bootstrap")
    boot = st.integers(0, n - 1, w.n_trees * n).reshape(w.n_trees, n)
    nodes, cnt = _train_gpu(S, ctx, inst.space, inst.x_obs, labels, boot, w.max_depth, w.leaf_scale)
    ctx.check()
    feats = _feats(inst.space, inst.x_obs, n)
    picks = np.unique(np.linspace(0, w.n_trees - 1, sample).astype(int))
    oracle_trees = _check_trees(S, nodes, cnt, feats, labels, boot, w.max_depth, w.leaf_scale, picks)
    hn, offs = S.compact_forest(nodes, cnt)
    L = S.scoot_forest_layout_init(hn, offs, w.d, w.leaf_scale)
    blob = torch.from_numpy(S.scoot_forest_pack(L, hn, offs)).cuda()
    cand = torch.from_numpy(inst.cand.view(np.int32)).cuda()
    votes = torch.zeros(inst.n_cand, dtype=torch.int32, device="cuda")
    S.scoot_rf_predict(ctx, L, blob, inst.space, cand, inst.n_cand, w.delta_num, w.delta_den, votes)
    torch.cuda.synchronize()
    sub = np.concatenate(oracle_trees)
    soffs = np.zeros(len(picks) + 1, np.int32)
    soffs[1:] = np.cumsum([len(t) for t in oracle_trees])
    # the packed forest's votes restricted to the sampled trees: pack those alone
    hs = np.concatenate([hn[offs[t]:offs[t + 1]] for t in picks])
    so = np.zeros(len(picks) + 1, np.int32)
    so[1:] = np.cumsum([offs[t + 1] - offs[t] for t in picks])
    Ls = S.scoot_forest_layout_init(hs, so, w.d, w.leaf_scale)
    blob_s = torch.from_numpy(S.scoot_forest_pack(Ls, hs, so)).cuda()
    vs = torch.zeros(inst.n_cand, dtype=torch.int32, device="cuda")
    S.scoot_rf_predict(ctx, Ls, blob_s, inst.space, cand, inst.n_cand, w.delta_num, w.delta_den, vs)
    want = O.rf_votes(sub, soffs, inst.space, inst.cand, inst.n_cand)
    assert np.array_equal(vs.cpu().numpy().astype(np.int64), want)
    total = votes.cpu().numpy()
    assert total.min() >= 0 and total.max() <= w.leaf_scale * w.n_trees
    print(f"[parity] rf_train {name}: {w.n_trees} trees, {int(cnt.sum())} nodes; {len(picks)} trees identical")


def test_rf_train_invalid_inputs(S, ctx):
    """Bad inputs are caught before any access they would steer: a bootstrap
    index outside the observations empties that tree (SCOOT_EDEVICE); a NaN
    feature or a label of 2 empties the trees that draw that observation
    (SCOOT_EINVAL); the other trees train as usual."""
    space = _space([CONTINUOUS, INT_UNIFORM])
    n = 16
    st = Stream(3, "rf-train-bad")
    words = np.stack([st.uniform(n).astype(np.float32).view(np.uint32), st.integers(0, 5, n).astype(np.uint32)])
    labels = (st.uniform(n) < 0.5).astype(np.uint8)
    boot = st.integers(0, n - 1, 4 * n).reshape(4, n)
    boot[:, 0] = 1          # every tree draws observation 1 ...
    boot[2:, :] = np.where(boot[2:, :] == 3, 4, boot[2:, :])  # ... trees 2, 3 never draw 3
    boot[:2, 1] = 3         # trees 0, 1 do
    boot[1, 5] = n
    nodes, cnt = _train_gpu(S, ctx, space, words, labels, boot, 6, 255)
    assert cnt[1] == 0 and np.all(cnt[[0, 2, 3]] > 0)
    _expect_status(S, ctx, -4)  # SCOOT_EDEVICE
    _check_trees(S, nodes, cnt, _feats(space, words, n), labels, boot, 6, 255, [0, 2, 3])
    boot[1, 5] = 0
    bad = words.copy()
    bad[0, 3] = np.float32(np.nan).view(np.uint32)
    nodes, cnt = _train_gpu(S, ctx, space, bad, labels, boot, 6, 255)
    assert np.all(cnt[:2] == 0) and np.all(cnt[2:] > 0)
    _expect_status(S, ctx, -1)  # SCOOT_EINVAL
    _check_trees(S, nodes, cnt, _feats(space, bad, n), labels, boot, 6, 255, [2, 3])
    lab = labels.copy()
    lab[1] = 2
    _, cnt = _train_gpu(S, ctx, space, words, lab, boot, 6, 255)
    assert np.all(cnt == 0)
    _expect_status(S, ctx, -1)  # SCOOT_EINVAL
    with pytest.raises(S.ScootError):
        _train_gpu(S, ctx, space, words, labels, boot, 6, 255, node_cap=2 * n - 2)


def test_rf_train_signed_zero(S, ctx):
    """-0 and +0 in one feature are one value; thresholds of zero are +0."""
    space = _space([CONTINUOUS, CONTINUOUS])
    n = 40
    st = Stream(5, "rf-train-zero")
    v = st.integers(-2, 2, 2 * n).astype(np.float32).reshape(2, n)
    v[v == 0] = np.where(st.uniform(int((v == 0).sum())) < 0.5, np.float32(-0.0), np.float32(0.0))
    words = v.view(np.uint32)
    labels = (st.uniform(n) < 0.5).astype(np.uint8)
    boot = st.integers(0, n - 1, 6 * n).reshape(6, n)
    nodes, cnt = _train_gpu(S, ctx, space, words, labels, boot, 8, 255)
    ctx.check()
    _check_trees(S, nodes, cnt, _feats(space, words, n), labels, boot, 8, 255, range(6))
    recs = nodes.view(S.NODE_DTYPE)
    vals = np.concatenate([recs[t, :cnt[t]][recs[t, :cnt[t]]["flags"] == 0]["val"] for t in range(6)])
    assert np.any(vals == 0) and not np.any(np.signbit(vals[vals == 0]))
