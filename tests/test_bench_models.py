"""The algorithmic work counts behind bench.py's roofline figures, checked
against independent counts (CPU only).

- The forest-training count (sorted-list entries touched by the split
  search and the partitions) equals a count made by re-growing each tree's
  node sample sets from the oracle's CART and applying the rule: a node
  that searches scans its m' samples in each of the d lists, a split node
  moves them.
- The MLE flop count is the documented polynomial.
- The scoring work model's per-stage figures follow the formulas stated
  for each kernel (bytes of the columns a stage reads, flops of the
  posterior and acquisition).
"""
import sys

import numpy as np
import pytest

import oracle as O
from conftest import ROOT
from workloads import make_instance, seeds

sys.path.insert(0, ROOT)
import bench  # noqa: E402


def _node_sample_sets(tree, feats, boot):
    """Sample indices reaching each node, by walking the bootstrap down."""
    sets = {0: list(boot)}
    for k, (val, left, f, leaf) in enumerate(tree):
        if leaf:
            continue
        samp = sets[k]
        sets[left] = [i for i in samp if feats[i, f] <= val]
        sets[left + 1] = [i for i in samp if feats[i, f] > val]
    return sets


@pytest.mark.parametrize("name,trees", [("d8-ehvi2", 4), ("tiny", 6)])
def test_rf_list_entries_counts_the_search_and_the_partitions(name, trees):
    from paper_2408_04323_gb300 import scoot as S
    inst, labels, boot = bench.rf_train_inputs(name)
    w = inst.workload
    n, d = w.n_obs, inst.d
    feats = O.decode(inst.space, inst.x_obs, n).astype(np.float32)
    nodes = np.zeros((trees, 2 * n - 1), np.int64)
    cnt = np.zeros(trees, np.int32)
    want = 0
    for t in range(trees):
        tree = O.train_cart(feats, labels, boot[t], w.max_depth, w.leaf_scale)
        recs, _ = O.train_forest(feats, labels, boot[t:t + 1], w.max_depth, w.leaf_scale)
        nodes[t].view(S.NODE_DTYPE)[:len(recs)] = recs
        cnt[t] = len(recs)
        sets = _node_sample_sets(tree, feats, boot[t])
        # depth of each node by breadth-first numbering: children follow their parent
        depth = {0: 0}
        for k, (_, left, _, leaf) in enumerate(tree):
            if not leaf:
                depth[left] = depth[left + 1] = depth[k] + 1
        for k, (_, _, _, leaf) in enumerate(tree):
            m = len(sets[k])
            p = int(sum(labels[i] for i in sets[k]))
            if depth[k] < w.max_depth and 0 < p < m:
                want += d * m
            if not leaf:
                want += d * m
    got = bench.rf_list_entries(S, nodes, cnt, feats, labels, boot[:trees], w.max_depth)
    assert got == want


def test_mle_flops_polynomial():
    for n, d in [(1, 1), (64, 8), (200, 10)]:
        want = 2 * (n ** 3 / 3 + n ** 3 / 6 + n * n) + n * (n + 1) / 2 * (6 * d + 60)
        assert bench.mle_flops(n, d) == pytest.approx(want)


@pytest.mark.parametrize("name", ["d8-ehvi2", "d10-ei", "d10-ehvi3"])
def test_scoring_work_model(name):
    inst = make_instance(name, seeds(name)[0], n_cand=16)
    w = inst.workload
    d, n, M = inst.d, inst.n_obs, inst.n_obj
    cols = set()
    for c in inst.clauses:
        cols.update(int(c["guard_param"][g]) for g in range(int(c["n_guard"])))
        cols.update(int(c["term_param"][t]) for t in range(int(c["n_term"])))
    B = 12
    wm = bench.work_model(inst, B)
    assert wm["prune"] == ("hbm", 4 * len(cols) + 1)  # referenced columns + the mask byte
    assert wm["rf"] == ("hbm", 4 * d + 6)             # every column, mask in/out, votes
    m_eff = M if w.acq == "ehvi" else 1
    post = m_eff * (n * (3 * d + 12) + 2 * n + n * (n + 1) + 2 * n)
    acq = 30 if w.acq == "ei" else w.n_mc * B * 4 * M
    assert wm["score"] == ("alu", post + acq)
    assert wm["topq"] == ("hbm", 5)
    mace = bench.work_model(inst, B, "mace")["score"][1]
    assert mace == n * (3 * d + 12) + 2 * n + n * (n + 1) + 2 * n + 47


@pytest.mark.parametrize("name", ["d8-ehvi2", "d10-ei", "d12-fantasy"])
def test_tensor_flops_count_the_issued_part_products(name):
    """bf16 flops per candidate of the tensor-core posterior: every (row i,
    column c) pair the MMAs touch (rows from the first row of c's 32-column
    k-block on, the rest of the triangle skipped), six part products of two
    flops each, per objective; enumerated pair by pair here."""
    inst = make_instance(name, seeds(name)[0], n_cand=16)
    n_pad = 64 * ((inst.n_obs + 63) // 64)
    pairs = sum(1 for i in range(n_pad) for c in range(n_pad) if i >= 32 * (c // 32))
    assert bench.posterior_tensor_flops(inst) == inst.n_obj * 6 * 2 * pairs
    assert bench.posterior_tensor_flops(inst, 1) == 6 * 2 * pairs
    # at least the triangle, at most the square
    assert n_pad * (n_pad + 1) // 2 <= pairs <= n_pad * n_pad
