"""MACE for one objective (Sections 4.5 and 4.7) through the C ABI: UCB, PI
and EI on the same posterior, the exact Pareto front of the three, and the
SplitMix64-keyed random k-subset of it.

Bars: the front and the picks are bit-exact against the oracle's selection
applied to the GPU's own fp32 triples (the decision is taken in the
kernel's precision on both sides); the acquisition values are within
1e-6 + 1e-4 |oracle| plus, for PI and UCB on given moments, the first-order
effect of the fp32 rounding of mu - y+ + xi, sigma and z (PI's slope in mu
is phi(z) / sigma, unbounded as sigma -> 0, so the stated bound alone does
not hold there for any fp32 evaluation); values computed from the GPU's own
posterior add the propagated posterior tolerance as in the EI test.
"""
import math

import numpy as np
import pytest

import oracle as O
from workloads import Stream, make_instance, seeds

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from parity_tol import ATOL, RTOL, posterior_tols, propagated_tol  # noqa: E402

U32 = 2.0 ** -24  # unit roundoff of fp32
CAP = 65536


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


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def np_(t):
    torch.cuda.synchronize()
    return t.cpu().numpy()


def rounding_tol(mu, var, yb, xi, kappa):
    """First-order effect of fp32 rounding inside the kernel on (UCB, PI, EI)."""
    sd = np.sqrt(np.maximum(var, 0.0))
    a = mu - yb + xi
    da = 2 * U32 * (np.abs(mu) + abs(yb) + xi)
    z = np.where(sd > 0, a / np.where(sd > 0, sd, 1.0), 0.0)
    phi = np.exp(-0.5 * z * z) / math.sqrt(2 * math.pi)
    t_pi = np.where(sd > 0, 2 * phi * (da / np.where(sd > 0, sd, 1.0) + 3 * U32 * np.abs(z)), 0.0)
    t_ucb = 4 * U32 * (np.abs(mu) + abs(kappa) * sd)
    t_ei = 2 * da
    return np.stack([t_ucb, t_pi, t_ei])


def check_rows(name, g, want, extra):
    tol = ATOL + RTOL * np.abs(want) + extra
    r = np.abs(g - want) / tol
    for row, label in enumerate(("UCB", "PI", "EI")):
        print(f"[parity] {name} {label}: n={g.shape[1]} max|err|/tol={r[row].max():.3f}")
    assert r.max() <= 1.0


# ------------------------------------------------------------------ acquisitions

@pytest.mark.parametrize("kappa", [19.9, 2.5])
def test_mace_kernel_on_generated_moments(S, ctx, kappa):
    st = Stream(31, "mace-moments")
    n = 40000 + 13
    mu = (st.normal(n) * 1.5).astype(np.float32)
    var = (st.uniform(n) ** 3).astype(np.float32)
    var[:100] = 0.0
    var[100:200] = 1e-30
    var[200:210] = -1e-3  # clamped to 0
    mask = (st.uniform(n) < 0.9).astype(np.uint8)
    lda = n + 5
    acq = torch.full((3, lda), 9.0, device="cuda")
    yb, xi = 0.7, 1e-4
    S.scoot_acq_mace(ctx, dev(mu), dev(var), n, yb, xi, kappa, acq, dev(mask))
    g = np_(acq)
    assert np.all(g[:, n:] == 9.0)
    assert np.all(g[:, :n][:, mask == 0] == -np.inf)
    m64, v64 = mu.astype(np.float64), var.astype(np.float64)
    want = O.mace_acquisitions(m64, v64, yb, xi, kappa)
    live = mask == 1
    check_rows(f"acq_mace kappa={kappa}", g[:, :n][:, live], want[:, live],
               rounding_tol(m64, v64, yb, xi, kappa)[:, live])
    step = live & (var <= 0)
    assert np.array_equal(g[1, :n][step], (m64[step] - yb + xi > 0).astype(np.float32))


def _gp(S, inst):
    L = S.scoot_gp_layout_init(inst.space, inst.n_obs, inst.n_obj, 0)
    blob, _ = S.scoot_gp_prepare(inst.space, inst.x_obs, inst.y_obs, inst.lengthscale,
                                 inst.signal_var, inst.noise_var, L)
    return L, dev(blob)


@pytest.mark.parametrize("tc", [1, 0], ids=["tensor", "simt"])
def test_score_mace_parity(S, ctx, tc):
    """Fused posterior + (UCB, PI, EI) against the oracle's fp64 posterior,
    with either product of L^{-1} k (tensor cores or fp32 SIMT)."""
    name = "d10-ei"
    n = 8192 + 77
    inst = make_instance(name, seeds(name)[1], n_cand=n)
    L, state = _gp(S, inst)
    cand = dev(inst.cand.view(np.int32))
    mask = torch.empty(n, dtype=torch.uint8, device="cuda")
    S.scoot_prune(ctx, inst.space, inst.clauses, cand, n, mask)
    kappa, xi = 6.31, 1e-4
    acq = torch.full((3, n), 5.0, device="cuda")
    S.scoot_ctx_set_tensor_cores(ctx, tc)
    try:
        S.scoot_score_mace(ctx, L, state, cand, n, xi, kappa, acq, mask)
        g = np_(acq)
    finally:
        S.scoot_ctx_set_tensor_cores(ctx, 1)
    known = O.prune_mask(inst.space, inst.clauses, inst.cand, n)
    assert np.all(g[:, ~known] == -np.inf) and np.all(np.isfinite(g[:, known]))
    idx = np.nonzero(known)[0]
    gps = [O.GP(inst.space, inst.x_obs, inst.y_obs[0], inst.lengthscale[0], inst.signal_var[0],
                inst.noise_var[0], 0)]
    mu, var, e_mu, e_var = posterior_tols(gps, np.ascontiguousarray(inst.cand[:, idx]))
    yb = float(inst.y_obs[0].max())
    rows = []
    for r in range(3):
        f = lambda a, b, r=r: O.mace_acquisitions(a[:, 0], b[:, 0], yb, xi, kappa)[r]
        want, tol = propagated_tol(f, mu, var, e_mu, e_var)
        tol = tol + rounding_tol(mu[:, 0], var[:, 0], yb, xi, kappa)[r]
        ratio = np.abs(g[r, idx] - want) / tol
        print(f"[parity] score_mace {name} tc={tc} row {r}: n={len(idx)} max|err|/tol={ratio.max():.3f}")
        rows.append(ratio.max())
    assert max(rows) <= 1.0
    # the fused kernel agrees with posterior + acq_mace (the posterior with the same product)
    mean = torch.empty((1, n), device="cuda")
    vv = torch.empty((1, n), device="cuda")
    S.scoot_ctx_set_tensor_cores(ctx, tc)
    try:
        S.scoot_gp_posterior(ctx, L, state, cand, n, mean, vv, mask)
    finally:
        S.scoot_ctx_set_tensor_cores(ctx, 1)
    acq2 = torch.empty((3, n), device="cuda")
    S.scoot_acq_mace(ctx, mean[0], vv[0], n, yb, xi, kappa, acq2, mask)
    g2 = np_(acq2)
    assert np.allclose(g2[:, idx], g[:, idx], rtol=1e-5, atol=1e-6)


# ------------------------------------------------------------------ Pareto front and random k-subset

def _triples(n, levels, seed, bad=True):
    st = Stream(seed, "pareto")
    A = np.floor(st.uniform(3 * n).reshape(3, n) * levels).astype(np.float32)
    if bad and n > 10:
        A[0, st.uniform(n) < 0.01] = np.nan
        A[2, st.uniform(n) < 0.01] = -np.inf
    mask = (st.uniform(n) < 0.8).astype(np.uint8)
    return A, mask


def _select(S, ctx, A, n, k, seed, mask=None, front_cap=None):
    idx = torch.full((k,), -7, dtype=torch.int64, device="cuda")
    cnt = torch.full((2,), -7, dtype=torch.int32, device="cuda")
    fr = None if front_cap is None else torch.full((max(front_cap, 1),), -7, dtype=torch.int64, device="cuda")
    S.scoot_select_pareto(ctx, dev(A), n, k, seed, idx, cnt, None if mask is None else dev(mask), fr)
    return np_(idx), np_(cnt), None if fr is None else np_(fr)


@pytest.mark.parametrize("n,levels,k", [(1, 3, 1), (17, 3, 4), (1023, 6, 64), (1024, 40, 4), (1025, 6, 8),
                                        (5000, 1000, 16), (3001, 2, 5)])
def test_pareto_select_bit_exact(S, ctx, n, levels, k):
    A, mask = _triples(n, levels, n * 7 + levels)
    for m in (None, mask):
        for seed in (3, 0xDEADBEEFCAFEF00D):
            gi, gc, gf = _select(S, ctx, A, n, k, seed, m, front_cap=n)
            picks, front, c = O.mace_select(A.astype(np.float64), m, k, seed)
            assert gc.tolist() == [c, len(front)]
            assert gi[:c].tolist() == picks.tolist() and np.all(gi[c:] == -1)
            assert sorted(gf[:len(front)].tolist()) == front.tolist() and np.all(gf[len(front):] == -7)


def _eligible(A, mask):
    ok = ~np.any(np.isnan(A) | (A == -np.inf), axis=0)
    return ok if mask is None else ok & (mask != 0)


def _check_front_properties(A, mask, front):
    """Exact at any size: the front members are eligible and no eligible
    candidate dominates one of them, and every other eligible candidate is
    dominated by a front member; together these fix the maxima set."""
    A = A.astype(np.float64)
    ok = _eligible(A, mask)
    assert np.all(ok[front])
    E = A[:, ok]
    F = A[:, front]
    for j in range(F.shape[1]):
        f = F[:, j:j + 1]
        assert not np.any(np.all(E >= f, axis=0) & np.any(E > f, axis=0))
    rest = np.setdiff1d(np.nonzero(ok)[0], front)
    for s in range(0, len(rest), 1 << 14):
        R = A[:, rest[s:s + (1 << 14)]]
        dom = np.zeros(R.shape[1], bool)
        for j in range(F.shape[1]):
            f = F[:, j:j + 1]
            dom |= np.all(f >= R, axis=0) & np.any(f > R, axis=0)
        assert dom.all()


def test_pareto_select_large_pool_properties(S, ctx):
    n = 300007
    A, mask = _triples(n, 200, 77)
    gi, gc, gf = _select(S, ctx, A, n, 16, 5, mask, front_cap=4096)
    F = int(gc[1])
    assert 0 < F <= 4096
    front = np.sort(gf[:F])
    assert len(np.unique(front)) == F
    _check_front_properties(A, mask, front)
    keys = sorted((O.splitmix64(5, int(i)), int(i)) for i in front)
    assert gi[:gc[0]].tolist() == [i for _, i in keys[:16]]


def test_pareto_degenerate_cases(S, ctx):
    A, mask = _triples(500, 5, 1, bad=False)
    # nothing eligible
    gi, gc, _ = _select(S, ctx, A, 500, 4, 1, np.zeros(500, np.uint8))
    assert gc.tolist() == [0, 0] and np.all(gi == -1)
    gi, gc, _ = _select(S, ctx, A, 0, 4, 1)
    assert gc.tolist() == [0, 0] and np.all(gi == -1)
    # all equal: everything is on the front; k larger than the front
    E = np.ones((3, 40), np.float32)
    gi, gc, gf = _select(S, ctx, E, 40, 64, 9, front_cap=40)
    assert gc.tolist() == [40, 40] and sorted(gi[:40].tolist()) == list(range(40)) and np.all(gi[40:] == -1)
    # one candidate dominates all others
    D = A.copy()
    D[:, 123] = 10.0
    gi, gc, _ = _select(S, ctx, D, 500, 3, 2)
    assert gc.tolist() == [1, 1] and gi.tolist() == [123, -1, -1]
    # a front larger than front_cap: the first front_cap entries only
    gi, gc, gf = _select(S, ctx, E, 40, 2, 9, front_cap=7)
    assert gc.tolist() == [2, 40] and len(set(gf.tolist())) == 7 and set(gf.tolist()) <= set(range(40))


def test_pareto_rejects_bad_arguments(S, ctx):
    A, _ = _triples(100, 5, 2, bad=False)
    for k in (0, 65):
        with pytest.raises(S.ScootError) as e:
            _select(S, ctx, A, 100, k, 1)
        assert e.value.status == -6
    idx = torch.empty(4, dtype=torch.int64, device="cuda")
    cnt = torch.empty(2, dtype=torch.int32, device="cuda")
    with pytest.raises(S.ScootError) as e:
        S.scoot_select_pareto(ctx, dev(A[:, :50]), 100, 4, 1, idx, cnt)  # lda = 50 < n
    assert e.value.status == -1


def test_pareto_capacity(S, ctx):
    """A front of exactly SCOOT_PARETO_CAP candidates is found whole; one
    more surviving candidate is reported (count {-1, -1}, EUNSUPPORTED from
    the context check), and the context stays usable."""
    for n, over in ((CAP, False), (CAP + 4464, True)):
        t = np.arange(n, dtype=np.float32)
        A = np.stack([t, -t, np.zeros(n, np.float32)])  # mutually non-dominated
        gi, gc, gf = _select(S, ctx, A, n, 4, 11, front_cap=n)
        if not over:
            assert gc.tolist() == [4, n]
            assert np.array_equal(np.sort(gf), np.arange(n))
            keys = sorted((O.splitmix64(11, i), i) for i in range(n))
            assert gi.tolist() == [i for _, i in keys[:4]]
            ctx.check()
        else:
            assert gc.tolist() == [-1, -1] and np.all(gi == -1)
            with pytest.raises(S.ScootError) as e:
                ctx.check()
            assert e.value.status == -6
    A, mask = _triples(1000, 5, 3)
    gi, gc, _ = _select(S, ctx, A, 1000, 4, 1, mask)
    picks, front, c = O.mace_select(A.astype(np.float64), mask, 4, 1)
    assert gc.tolist() == [c, len(front)] and gi[:c].tolist() == picks.tolist()
    ctx.check()


# ------------------------------------------------------------------ one MACE round at full size

def test_mace_round_full_pool(S, ctx):
    """d10-ei at its full pool: prune, forest, fused MACE scores and the
    random front subset; the front is checked exactly against the GPU's own
    triples at full size, the scores on a sample against the oracle."""
    from paper_2408_04323_gb300.pipeline import RoundInputs, ScoringRound
    name = "d10-ei"
    inst = make_instance(name, seeds(name)[0])
    w = inst.workload
    n = inst.n_cand
    inp = RoundInputs(inst.space, inst.clauses, inst.nodes, inst.tree_offset, w.leaf_scale, w.delta_num,
                      w.delta_den, inst.x_obs, inst.y_obs, inst.lengthscale, inst.signal_var,
                      inst.noise_var, inst.ref, inst.eps, "mace", 4, seed=12345)
    rnd = ScoringRound(ctx, inp, n)
    idx, _, count = rnd.run(dev(inst.cand.view(np.int32)), n)
    ctx.check()
    acq = np_(rnd.acq3)
    mask = np_(rnd.mask)
    cnt = np_(count)
    F = int(cnt[1])
    assert 0 < F <= rnd.front_cap
    front = np.sort(np_(rnd.front)[:F])
    _check_front_properties(acq[:, :n], mask, front)
    keys = sorted((O.splitmix64(rnd.seed, int(i)), int(i)) for i in front)
    k = int(cnt[0])
    assert k == min(4, F)
    assert np_(idx)[:k].tolist() == [i for _, i in keys[:k]]
    feas = O.pof_feasible(O.rf_votes(inst.nodes, inst.tree_offset, inst.space, inst.cand, n), inst.n_trees,
                          w.leaf_scale, w.delta_num, w.delta_den)
    known = O.prune_mask(inst.space, inst.clauses, inst.cand, n)
    assert np.array_equal(mask.astype(bool), known & feas)
    sample = np.union1d(np.nonzero(mask)[0][::997], front)
    gps = [O.GP(inst.space, inst.x_obs, inst.y_obs[0], inst.lengthscale[0], inst.signal_var[0],
                inst.noise_var[0], 0)]
    mu, var, e_mu, e_var = posterior_tols(gps, np.ascontiguousarray(inst.cand[:, sample]))
    yb = float(inst.y_obs[0].max())
    for r in range(3):
        f = lambda a, b, r=r: O.mace_acquisitions(a[:, 0], b[:, 0], yb, inp.xi, rnd.kappa)[r]
        want, tol = propagated_tol(f, mu, var, e_mu, e_var)
        tol = tol + rounding_tol(mu[:, 0], var[:, 0], yb, inp.xi, rnd.kappa)[r]
        assert (np.abs(acq[r, sample] - want) / tol).max() <= 1.0
