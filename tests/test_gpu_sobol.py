"""Sobol configurations (Algorithm 1's initial design, Section 4.6's
shortfall fill) and the selection of the first feasible ones, through the C
ABI, against the oracle.

Bar: the words are integer/bit results and must be identical.  The one
transcendental step (exp for integer log-uniform parameters, rounded half to
even) could in principle land on opposite sides of a rounding boundary on
the two sides; the test allows a difference only where the oracle's fp64
value is within 1e-9 of such a boundary, and reports how many there were.
"""
import math

import numpy as np
import pytest

import oracle as O
from workloads import (CATEGORICAL, CONTINUOUS, INT_LOG, INT_UNIFORM, PARAM_DTYPE, Stream, make_instance,
                       seeds)

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


def np_(t):
    torch.cuda.synchronize()
    return t.cpu().numpy()


def _space(*params):
    sp = np.zeros(len(params), PARAM_DTYPE)
    for i, (kind, nc, lo, hi) in enumerate(params):
        sp[i]["kind"], sp[i]["n_choices"], sp[i]["lo"], sp[i]["hi"] = kind, nc, lo, hi
    return sp


def _boundary(space, j, u):
    """Oracle fp64 values of an integer log-uniform parameter sit within 1e-9 of .5."""
    p = space[j]
    lo, hi = float(p["lo"]), float(p["hi"])
    x = np.exp(math.log(lo) + u * (math.log(hi) - math.log(lo)))
    return np.abs(x - np.floor(x) - 0.5) < 1e-9


@pytest.mark.parametrize("skip,n", [(0, 1), (0, 4096), (12345, 3001), ((1 << 31) - 1000, 2000)])
def test_sobol_configs_match_oracle(S, ctx, skip, n):
    sp = _space((INT_LOG, 0, 1, 8192), (INT_LOG, 0, 16, 65536), (INT_UNIFORM, 0, -5, 1000), (CATEGORICAL, 3, 0, 0),
                (CONTINUOUS, 0, 0.5, 0.95), (INT_UNIFORM, 0, 0, 1), (CATEGORICAL, 7, 0, 0), (INT_LOG, 0, 2, 3),
                (CONTINUOUS, 0, -3.0, 2.0), (INT_UNIFORM, 0, 1, 4096), (CATEGORICAL, 2, 0, 0), (INT_LOG, 0, 1, 2),
                (CONTINUOUS, 0, 0.0, 1.0), (INT_UNIFORM, 0, 7, 7), (CATEGORICAL, 5, 0, 0), (INT_LOG, 0, 100, 200))
    ld = (n + 3) // 4 * 4 + 4
    out = torch.full((len(sp), ld), -1, dtype=torch.int32, device="cuda")
    S.scoot_sobol_configs(ctx, sp, skip, n, out)
    g = np_(out).view(np.uint32)
    assert np.all(g[:, n:] == 0xFFFFFFFF)
    want = O.sobol_configs(sp, n, skip)
    X = O.sobol_integers(len(sp), n, skip)
    diff = g[:, :n] != want
    allowed = np.zeros_like(diff)
    for j in range(len(sp)):
        if int(sp[j]["kind"]) == INT_LOG:
            allowed[j] = _boundary(sp, j, X[:, j].astype(np.float64) / 4294967296.0)
    print(f"[parity] sobol skip={skip} n={n}: {int(diff.sum())} differing words, {int(allowed.sum())} at rounding boundaries")
    assert not np.any(diff & ~allowed)


@pytest.mark.parametrize("n,need,p", [(0, 4, 0.5), (1, 1, 1.0), (5000, 64, 0.01), (100003, 17, 0.3), (777, 64, 0.0),
                                      (2048, 3, 1.0)])
def test_first_feasible(S, ctx, n, need, p):
    st = Stream(n + need, "first")
    mask = (st.uniform(max(n, 1))[:n] < p).astype(np.uint8)
    idx = torch.full((need,), 9, dtype=torch.int64, device="cuda")
    cnt = torch.full((1,), 9, dtype=torch.int32, device="cuda")
    m = torch.from_numpy(mask).cuda() if n else torch.zeros(1, dtype=torch.uint8, device="cuda")
    S.scoot_first_feasible(ctx, m, n, need, idx, cnt)
    want = np.nonzero(mask)[0][:need]
    c = int(np_(cnt)[0])
    got = np_(idx)
    assert c == len(want) and got[:c].tolist() == want.tolist() and np.all(got[c:] == -1)


def test_shortfall_fill_round(S, ctx):
    """A round with fewer feasible candidates than q: the fill is the first
    Sobol points that satisfy the known constraints, in order, and the next
    fill continues the sequence."""
    from paper_2408_04323_gb300.pipeline import RoundInputs, ScoringRound
    name = "d10-ei"
    inst = make_instance(name, seeds(name)[0], n_cand=40)
    w = inst.workload
    q = 64
    inp = RoundInputs(inst.space, inst.clauses, inst.nodes, inst.tree_offset, w.leaf_scale, w.delta_num,
                      w.delta_den, inst.x_obs, inst.y_obs, inst.lengthscale, inst.signal_var, inst.noise_var,
                      inst.ref, inst.eps, w.acq, q)
    rnd = ScoringRound(ctx, inp, inst.n_cand)
    rnd.run(torch.from_numpy(inst.cand.view(np.int32)).cuda(), inst.n_cand)
    count = int(np_(rnd.top_count)[0])
    assert count < q
    fill = rnd.fill_shortfall(batch=1024)
    need = q - count
    pool = O.sobol_configs(inst.space, 1024)
    ok = np.nonzero(O.prune_mask(inst.space, inst.clauses, pool, 1024))[0][:need]
    assert fill.shape == (inst.d, need) and np.array_equal(fill, pool[:, ok])
    assert rnd.sobol_skip == int(ok[-1]) + 1
    fill2 = rnd.fill_shortfall(batch=1024)
    pool2 = O.sobol_configs(inst.space, 1024, int(ok[-1]) + 1)
    ok2 = np.nonzero(O.prune_mask(inst.space, inst.clauses, pool2, 1024))[0][:need]
    assert np.array_equal(fill2, pool2[:, ok2])
