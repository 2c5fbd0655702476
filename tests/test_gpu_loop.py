"""Algorithm 1's loop on the library's calls (paper_2408_04323_gb300/loop.py):
Sobol initial design, then rounds of forest training, hyperparameter MLE,
scoring of a Sobol pool and the threshold controller, against a synthetic
engine with a hidden crash region.

An integration test: each step is parity-tested on its own elsewhere.
Here the suggestions must satisfy the known constraints (checked by the
oracle's pruning), come in batches of q, and the threshold must follow the
oracle's controller over the same outcomes.
"""
import numpy as np
import pytest

import oracle as O
from workloads import make_instance, seeds

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


def engine(space, words):
    """Two conflicting maximised objectives of the configurations' feature
    coordinates, and a crash wherever the first coordinate exceeds 0.8."""
    u, _ = O.gp_features(space, O.decode(space, words))
    y0 = -((u - 0.3) ** 2).sum(axis=1)
    y1 = -((u - 0.6) ** 2).sum(axis=1)
    ok = u[:, 0] <= 0.8
    return np.stack([y0, y1]), ok


@pytest.mark.parametrize("acq", ["ehvi", "ei"])
def test_tuning_loop_runs_algorithm_1(S, acq):
    from paper_2408_04323_gb300.loop import TuningLoop
    inst = make_instance("d8-ehvi2", seeds("d8-ehvi2")[0], n_cand=16)
    ctx = S.Context(0)
    try:
        M = 2 if acq == "ehvi" else 1
        loop = TuningLoop(ctx, inst.space, inst.clauses, n_obj=M, q=4, acq=acq, n_trees=32, max_depth=8,
                          pool=1 << 14, mle_starts=4, mle_steps=30, seed=3)
        x0 = loop.initial_design(10)
        assert x0.shape == (inst.d, 10)
        assert np.all(O.prune_mask(inst.space, inst.clauses, x0, 10))
        y, ok = engine(inst.space, x0)
        delta, count = 0.5, 0
        loop.observe(x0, y[:M], ok)
        delta, count = O.delta_update(delta, count, int(ok.sum()), bool((~ok).any()))
        assert loop.delta == pytest.approx(delta) and loop.delta_count == count
        best0 = np.nanmax(np.where(loop.ok, loop.y[0], np.nan))
        for _ in range(3):
            x = loop.suggest()
            assert x.shape == (inst.d, 4)
            assert np.all(O.prune_mask(inst.space, inst.clauses, x, x.shape[1]))
            assert loop.theta is not None and np.all(np.isfinite(loop.theta))
            y, ok = engine(inst.space, x)
            loop.observe(x, y[:M], ok)
            delta, count = O.delta_update(delta, count, int(ok.sum()), bool((~ok).any()))
            assert loop.delta == pytest.approx(delta) and loop.delta_count == count
        assert loop.x.shape[1] == 22
        best = np.nanmax(np.where(loop.ok, loop.y[0], np.nan))
        assert best >= best0
        print(f"[loop] {acq}: best first objective {best0:.4f} -> {best:.4f}, Delta {loop.delta:.2f}, "
              f"crashes {int((~loop.ok).sum())} of {loop.ok.size}")
    finally:
        ctx.close()
