"""Parity of the CUDA path with the fp64 oracle, through the C ABI.

Bars: bit-exact for masks, vote counts and selected indices; for floating
point |gpu - oracle| <= 1e-6 + 1e-4 |oracle| for the posterior variance and
for EI / EHVI evaluated on given moments.  Two derived terms, both computed
by the oracle:
 * the posterior mean adds 2^-22 * sum_j |k_j alpha_j|, the rounding scale of
   an fp32 evaluation of mu = k . alpha (it matters only where mu crosses
   zero, where the relative part of the bound vanishes);
 * an acquisition computed from the GPU's own posterior adds the first-order
   change of the oracle's acquisition when mu and sigma^2 move by their own
   tolerances (central differences), i.e. the posterior error it inherits.
"""
import math

import numpy as np
import pytest

import oracle as O
from workloads import Stream, make_instance, seeds

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from parity_tol import ATOL, MU_COND, RTOL, posterior_tols, propagated_tol  # noqa: E402


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


def cand_dev(inst):
    return dev(inst.cand.view(np.int32))


def np_(t):
    torch.cuda.synchronize()
    return t.cpu().numpy()


def report(name, g, o, extra=0.0):
    g = np.asarray(g, np.float64)
    o = np.asarray(o, np.float64)
    tol = ATOL + RTOL * np.abs(o) + extra
    ratio = np.abs(g - o) / tol
    worst = float(ratio.max()) if ratio.size else 0.0
    print(f"[parity] {name}: n={g.size} max|err|/tol={worst:.3f} max|err|={np.abs(g - o).max() if g.size else 0:.3e}")
    return ratio


def report_tol(name, g, o, tol):
    g = np.asarray(g, np.float64)
    ratio = np.abs(g - o) / tol
    plain = np.abs(g - o) / (ATOL + RTOL * np.abs(o))
    print(f"[parity] {name}: n={g.size} max|err|/tol={ratio.max():.3f} max|err|={np.abs(g - o).max():.3e} "
          f"beyond the stated tolerance alone: {int((plain > 1).sum())}")
    return ratio


def sample_idx(n, k, seed):
    if n <= k:
        return np.arange(n)
    st = Stream(seed, "sample")
    return np.unique(st.integers(0, n - 1, k))


POOL = {"tiny": 4096, "d8-ehvi2": 1 << 18, "d10-ei": 1 << 20, "d10-ehvi3": 1 << 20, "d12-fantasy": 1 << 22}
NAMES = list(POOL)


# ------------------------------------------------------------------ prune, Eq. (2)

@pytest.mark.parametrize("name", NAMES)
def test_prune_bit_exact_full_pool(S, ctx, name):
    inst = make_instance(name, seeds(name)[0])
    n = inst.n_cand
    mask = torch.full((n,), 7, dtype=torch.uint8, device="cuda")
    cnt = torch.zeros(1, dtype=torch.int64, device="cuda")
    S.scoot_prune(ctx, inst.space, inst.clauses, cand_dev(inst), n, mask, cnt)
    got = np_(mask)
    want = O.prune_mask(inst.space, inst.clauses, inst.cand, n)
    assert np.array_equal(got, want.astype(np.uint8))
    assert int(np_(cnt)[0]) == int(want.sum())
    ctx.check()


def test_prune_edge_cases(S, ctx):
    inst = make_instance("d10-ei", seeds("d10-ei")[1], n_cand=1037)
    want = O.prune_mask(inst.space, inst.clauses, inst.cand, 1037).astype(np.uint8)
    cand = cand_dev(inst)
    for n in (0, 1, 2, 3, 5, 1037):
        buf = torch.full((1040,), 9, dtype=torch.uint8, device="cuda")
        mask = buf[1:1 + max(n, 1)]  # deliberately not 4-byte aligned
        cnt = torch.full((1,), 123, dtype=torch.int64, device="cuda")
        S.scoot_prune(ctx, inst.space, inst.clauses, cand, n, mask, cnt)
        got = np_(buf)
        assert np.array_equal(got[1:1 + n], want[:n]) and got[0] == 9 and np.all(got[1 + n:] == 9)
        assert int(np_(cnt)[0]) == int(want[:n].sum())
    # no clauses: everything feasible
    mask = torch.zeros(1037, dtype=torch.uint8, device="cuda")
    S.scoot_prune(ctx, inst.space, inst.clauses[:0], cand, 1037, mask)
    assert np_(mask).all()


@pytest.mark.parametrize("big", [False, True])
def test_prune_many_clauses_and_wide_sums(S, ctx, big):
    """Sixteen random guarded clauses over most of the twelve parameters
    (distinct-column slots), with 2^40-sized coefficients when big (the
    int128 path) or small ones (the int64 path)."""
    from workloads import CLAUSE_DTYPE
    inst = make_instance("d12-fantasy", seeds("d12-fantasy")[2], n_cand=20011)
    st = Stream(88 + big, "clauses")
    ints = [c for c in range(inst.d) if int(inst.space[c]["kind"]) != 3]
    cats = [c for c in ints if int(inst.space[c]["kind"]) == 2]
    cl = np.zeros(16, CLAUSE_DTYPE)
    vals = inst.cand.view(np.int32)
    for k in range(16):
        nt = 1 + k % 4
        terms = [ints[int(x)] for x in st.integers(0, len(ints) - 1, nt)]
        scale = (1 << 40) if big else 1000
        coef = [int(x) for x in (st.integers(0, 2 * scale, nt) - scale)]
        cl[k]["n_term"] = nt
        for t in range(nt):
            cl[k]["term_param"][t] = terms[t]
            cl[k]["coef"][t] = coef[t]
        # rhs at the 5% quantile of the sum over a sample: each clause fails
        # for about 5% of the pool, all sixteen together for about half
        smp = sum(c * vals[p, :2000].astype(object) for c, p in zip(coef, terms))
        cl[k]["rhs"] = int(sorted(smp)[100])
        if cats and k % 3 == 0:
            g = cats[k % len(cats)]
            cl[k]["n_guard"] = 1
            cl[k]["guard_param"][0] = g
            cl[k]["guard_value"][0] = int(vals[g, 0])
    n = inst.n_cand
    mask = torch.empty(n, dtype=torch.uint8, device="cuda")
    cnt = torch.zeros(1, dtype=torch.int64, device="cuda")
    S.scoot_prune(ctx, inst.space, cl, cand_dev(inst), n, mask, cnt)
    want = O.prune_mask(inst.space, cl, inst.cand, n)
    assert np.array_equal(np_(mask).astype(bool), want)
    assert int(np_(cnt)[0]) == int(want.sum()) and 0 < want.sum() < n


def test_prune_rejects_bad_arguments(S, ctx):
    inst = make_instance("tiny", 1001, n_cand=64)
    cand = cand_dev(inst)
    mask = torch.zeros(64, dtype=torch.uint8, device="cuda")
    with pytest.raises(S.ScootError) as e:  # ld not a multiple of 4
        S.scoot_prune(ctx, inst.space, inst.clauses, cand[:, :63].contiguous(), 63, mask)
    assert e.value.status == -1
    bad = inst.clauses.copy()
    bad[0]["term_param"][0] = 3  # a continuous parameter in a clause
    with pytest.raises(S.ScootError):
        S.scoot_prune(ctx, inst.space, bad, cand, 64, mask)
    big = torch.zeros((inst.d, 68), dtype=torch.int32, device="cuda")
    with pytest.raises(S.ScootError):  # ld < n
        S.scoot_prune(ctx, inst.space, inst.clauses, big[:, :64].contiguous(), 65, mask)


# ------------------------------------------------------------------ forest, Eq. (3)

def forest_dev(S, inst):
    L = S.scoot_forest_layout_init(inst.nodes, inst.tree_offset, inst.d, inst.workload.leaf_scale)
    return L, dev(S.scoot_forest_pack(L, inst.nodes, inst.tree_offset))


@pytest.mark.parametrize("name", NAMES)
def test_rf_votes_bit_exact(S, ctx, name):
    n = POOL[name] if name != "d12-fantasy" else 1 << 18
    inst = make_instance(name, seeds(name)[0], n_cand=n)
    w = inst.workload
    L, forest = forest_dev(S, inst)
    cand = cand_dev(inst)
    mask = torch.empty(n, dtype=torch.uint8, device="cuda")
    S.scoot_prune(ctx, inst.space, inst.clauses, cand, n, mask)
    votes = torch.full((n,), -1, dtype=torch.int32, device="cuda")
    cnt = torch.zeros(1, dtype=torch.int64, device="cuda")
    S.scoot_rf_predict(ctx, L, forest, inst.space, cand, n, w.delta_num, w.delta_den, votes, mask, cnt)
    ctx.check()
    known = O.prune_mask(inst.space, inst.clauses, inst.cand, n)
    want_votes = O.rf_votes(inst.nodes, inst.tree_offset, inst.space, inst.cand, n)
    got_votes = np_(votes).astype(np.int64)
    assert np.array_equal(got_votes[known], want_votes[known])
    assert np.all(got_votes[~known] == 0)
    feas = known & O.pof_feasible(want_votes, inst.n_trees, w.leaf_scale, w.delta_num, w.delta_den)
    assert np.array_equal(np_(mask).astype(bool), feas)
    assert int(np_(cnt)[0]) == int(feas.sum())
    # without a mask every candidate is walked
    S.scoot_rf_predict(ctx, L, forest, inst.space, cand, n, w.delta_num, w.delta_den, votes, None)
    assert np.array_equal(np_(votes).astype(np.int64), want_votes)


def test_rf_multi_chunk_forest(S, ctx):
    """A forest too large for one shared-memory chunk gives the same votes."""
    inst = make_instance("d12-fantasy", seeds("d12-fantasy")[1], n_cand=20000)
    reps = 4
    nodes = np.concatenate([inst.nodes] * reps)
    offs = np.zeros(inst.n_trees * reps + 1, np.int32)
    offs[1:] = np.cumsum(np.tile(np.diff(inst.tree_offset), reps))
    L = S.scoot_forest_layout_init(nodes, offs, inst.d, 255)
    assert L.n_chunks >= 2
    forest = dev(S.scoot_forest_pack(L, nodes, offs))
    votes = torch.empty(inst.n_cand, dtype=torch.int32, device="cuda")
    S.scoot_rf_predict(ctx, L, forest, inst.space, cand_dev(inst), inst.n_cand, 10, 20, votes, None)
    want = O.rf_votes(nodes, offs, inst.space, inst.cand, inst.n_cand)
    assert np.array_equal(np_(votes).astype(np.int64), want)


# ------------------------------------------------------------------ GP posterior (Section 4.3)

def gp_state(S, inst, kernel=0):
    L = S.scoot_gp_layout_init(inst.space, inst.n_obs, inst.n_obj, kernel)
    blob, _ = S.scoot_gp_prepare(inst.space, inst.x_obs, inst.y_obs, inst.lengthscale,
                                 inst.signal_var, inst.noise_var, L)
    return L, dev(blob)


def oracle_gps(inst, kernel=0):
    return [O.GP(inst.space, inst.x_obs, inst.y_obs[m], inst.lengthscale[m], inst.signal_var[m],
                 inst.noise_var[m], kernel) for m in range(inst.n_obj)]


@pytest.mark.parametrize("tc", [1, 0], ids=["tensor", "simt"])
@pytest.mark.parametrize("name,kernel", [("tiny", 0), ("d8-ehvi2", 0), ("d10-ei", 0), ("d10-ehvi3", 0),
                                         ("d12-fantasy", 0), ("d8-ehvi2", 1)])
def test_posterior_parity(S, ctx, name, kernel, tc):
    """Both products of L^{-1} k: the tensor-core one (three bf16 parts, six
    part products) and the fp32 SIMT one."""
    n = 4096 + 37  # several tiles (32 and 128 candidates) and a ragged tail
    inst = make_instance(name, seeds(name)[1], n_cand=n)
    L, state = gp_state(S, inst, kernel)
    M = inst.n_obj
    ldo = n + 3
    mean = torch.full((M, ldo), 77.0, device="cuda")
    var = torch.full((M, ldo), 77.0, device="cuda")
    S.scoot_ctx_set_tensor_cores(ctx, tc)
    try:
        S.scoot_gp_posterior(ctx, L, state, cand_dev(inst), n, mean, var)
        gm, gv = np_(mean), np_(var)
    finally:
        S.scoot_ctx_set_tensor_cores(ctx, 1)
    name = f"{name} {'tensor' if tc else 'simt'}"
    assert np.all(gm[:, n:] == 77.0) and np.all(gv[:, n:] == 77.0)
    for m, gp in enumerate(oracle_gps(inst, kernel)):
        mu, v = gp.posterior(inst.cand, n)
        cond = gp.mean_condition(inst.cand, n)
        r_mu = report(f"{name} k{kernel} mu[{m}]", gm[m, :n], mu, MU_COND * cond)
        r_mu_plain = report(f"{name} k{kernel} mu[{m}] (stated tol only)", gm[m, :n], mu)
        r_v = report(f"{name} k{kernel} var[{m}]", gv[m, :n], v)
        beyond = int((r_mu_plain > 1).sum())
        print(f"[mu-exceed] {name} kernel={kernel} objective={m}: {beyond} of {n} means beyond the stated "
              f"1e-6 + 1e-4|mu| alone, worst {r_mu_plain.max():.2f}x it; all within the derived bar "
              f"(worst {r_mu.max():.2f}x)")
        assert r_mu.max() <= 1.0
        # the derived term is rarely needed: at most 2% of means, none beyond 8x the stated bar
        assert beyond <= 0.02 * n and r_mu_plain.max() <= 8.0
        assert r_v.max() <= 1.0
        assert np.all(gv[m, :n] >= 0) and np.all(gv[m, :n] <= inst.signal_var[m] * (1 + 1e-6))


def test_posterior_mask_skips(S, ctx):
    inst = make_instance("d8-ehvi2", seeds("d8-ehvi2")[2], n_cand=999)
    L, state = gp_state(S, inst)
    maskh = (Stream(5, "m").uniform(999) < 0.5).astype(np.uint8)
    mean = torch.full((2, 999), 5.0, device="cuda")
    var = torch.full((2, 999), 5.0, device="cuda")
    S.scoot_gp_posterior(ctx, L, state, cand_dev(inst), 999, mean, var, dev(maskh))
    gm = np_(mean)
    assert np.all(gm[:, maskh == 0] == 5.0) and np.all(gm[:, maskh == 1] != 5.0)


# ------------------------------------------------------------------ acquisition

def test_ei_kernel_on_generated_moments(S, ctx):
    """Eq. (6) on seeded (mu, sigma^2) arrays, including sigma = 0 and far tails."""
    st = Stream(21, "ei")
    n = 50000
    mu = (st.normal(n) * 1.5).astype(np.float32)
    var = (st.uniform(n) ** 3).astype(np.float32)
    var[:100] = 0.0
    var[100:200] = 1e-30
    mask = (st.uniform(n) < 0.9).astype(np.uint8)
    acq = torch.empty(n, device="cuda")
    S.scoot_acq_ei(ctx, dev(mu), dev(var), n, 0.7, 1e-4, acq, dev(mask))
    g = np_(acq)
    want = O.expected_improvement(mu.astype(np.float64), var.astype(np.float64), 0.7, 1e-4)
    assert np.all(g[mask == 0] == -np.inf)
    assert report("ei kernel", g[mask == 1], want[mask == 1]).max() <= 1.0


@pytest.mark.parametrize("M,nf", [(2, 1), (2, 9), (3, 14), (4, 6)])
def test_ehvi_kernel_on_generated_moments(S, ctx, M, nf):
    """Eq. (7) on seeded moments and a seeded front (boxes from the library, cells from the oracle)."""
    st = Stream(30 + M * 10 + nf, "ehvi")
    Y = (st.uniform(M * nf).reshape(M, nf) * 2.0).astype(np.float32)
    ref = np.zeros(M, np.float32)
    lo, hi, fs = S.scoot_boxes_build(Y, ref)
    n, Sm = 3001, 48
    mu = (st.uniform(n * M).reshape(M, n) * 2.4 - 0.2).astype(np.float32)
    var = (st.uniform(n * M).reshape(M, n) * 0.3).astype(np.float32)
    var[:, :50] = 0.0
    eps = st.normal(Sm * M).reshape(Sm, M).astype(np.float32)
    acq = torch.empty(n, device="cuda")
    S.scoot_acq_ehvi(ctx, dev(mu), dev(var), n, dev(lo), dev(hi), dev(eps), acq)
    g = np_(acq)
    front = O.pareto_front(Y.T, ref)
    want = O.ehvi_mc(mu.T.astype(np.float64), var.T.astype(np.float64), eps, front, ref)
    assert report(f"ehvi kernel M={M} P={fs}", g, want).max() <= 1.0


def ehvi_inputs(S, inst):
    lo, hi, fs = S.scoot_boxes_build(inst.y_obs, inst.ref)
    return dev(lo), dev(hi), dev(inst.eps), fs


@pytest.mark.parametrize("name,k", [("tiny", 4096), ("d8-ehvi2", 1024), ("d10-ehvi3", 96), ("d12-fantasy", 384)])
def test_score_ehvi_parity(S, ctx, name, k):
    inst = make_instance(name, seeds(name)[0])
    n = inst.n_cand
    L, state = gp_state(S, inst)
    lo, hi, eps, fs = ehvi_inputs(S, inst)
    cand = cand_dev(inst)
    mask = torch.empty(n, dtype=torch.uint8, device="cuda")
    S.scoot_prune(ctx, inst.space, inst.clauses, cand, n, mask)
    acq = torch.empty(n, device="cuda")
    S.scoot_score_ehvi(ctx, L, state, cand, n, lo, hi, eps, acq, mask)
    g = np_(acq)
    known = O.prune_mask(inst.space, inst.clauses, inst.cand, n)
    assert np.array_equal(np.isfinite(g), known)
    idx = sample_idx(n, k, 7)
    idx = idx[known[idx]]
    gps = oracle_gps(inst)
    sub = np.ascontiguousarray(inst.cand[:, idx])
    mu, var, e_mu, e_var = posterior_tols(gps, sub)
    front = O.pareto_front(inst.y_obs.T, inst.ref)
    f = lambda a, b: O.ehvi_mc(a, b, inst.eps, front, inst.ref)
    want, tol = propagated_tol(f, mu, var, e_mu, e_var)
    assert report_tol(f"score_ehvi {name} (P={fs})", g[idx], want, tol).max() <= 1.0
    # the two-kernel path gives the same numbers as the fused kernel
    if n <= 1 << 18:
        M = inst.n_obj
        mean = torch.empty((M, n), device="cuda")
        var_d = torch.empty((M, n), device="cuda")
        S.scoot_ctx_set_tensor_cores(ctx, 0)  # the fused kernel's fp32 SIMT product
        try:
            S.scoot_gp_posterior(ctx, L, state, cand, n, mean, var_d, mask)
        finally:
            S.scoot_ctx_set_tensor_cores(ctx, 1)
        acq2 = torch.empty(n, device="cuda")
        S.scoot_acq_ehvi(ctx, mean, var_d, n, lo, hi, eps, acq2, mask)
        g2 = np_(acq2)
        # same arithmetic, only the order of the sample sum differs
        assert np.array_equal(np.isfinite(g2), np.isfinite(g))
        fin = np.isfinite(g)
        assert np.all(np.abs(g2[fin] - g[fin]) <= 1e-6 + 1e-5 * np.abs(g[fin]))


@pytest.mark.parametrize("name", ["d8-ehvi2", "d10-ehvi3"])
def test_score_ehvi_bounded_boxes(S, ctx, name):
    """Boxes bounded on the last objective take the kernel's general path
    (the saturated form needs boxes open there): every library box is cut at
    a finite height on that axis into two boxes covering the same region, so
    the EHVI is unchanged."""
    inst = make_instance(name, seeds(name)[2], n_cand=8192 + 19)
    n = inst.n_cand
    L, state = gp_state(S, inst)
    lo, hi, fs = S.scoot_boxes_build(inst.y_obs, inst.ref)
    cut = lo[:, -1] + 0.37
    lo2 = np.concatenate([lo, lo]).copy()
    hi2 = np.concatenate([hi, hi]).copy()
    hi2[:len(lo), -1] = cut
    lo2[len(lo):, -1] = cut
    cand = cand_dev(inst)
    mask = torch.empty(n, dtype=torch.uint8, device="cuda")
    S.scoot_prune(ctx, inst.space, inst.clauses, cand, n, mask)
    out = []
    for a, b in ((lo, hi), (lo2, hi2)):
        acq = torch.empty(n, device="cuda")
        S.scoot_score_ehvi(ctx, L, state, cand, n, dev(a), dev(b), dev(inst.eps), acq, mask)
        out.append(np_(acq))
    fin = np.isfinite(out[0])
    assert np.array_equal(fin, np.isfinite(out[1]))
    assert np.all(np.abs(out[1][fin] - out[0][fin]) <= 1e-6 + 1e-5 * np.abs(out[0][fin]))
    live = np.nonzero(fin)[0]
    idx = live[np.linspace(0, len(live) - 1, 48 if inst.n_obj > 2 else 181).astype(int)]
    mu, var, e_mu, e_var = posterior_tols(oracle_gps(inst), np.ascontiguousarray(inst.cand[:, idx]))
    front = O.pareto_front(inst.y_obs.T, inst.ref)
    want, tol = propagated_tol(lambda a, b: O.ehvi_mc(a, b, inst.eps, front, inst.ref), mu, var, e_mu, e_var)
    assert report_tol(f"score_ehvi bounded boxes {name} (B={2 * len(lo)})", out[1][idx], want, tol).max() <= 1.0


def test_score_ehvi_four_objectives_at_large_scale(S, ctx):
    """The fused 4-objective EHVI on objectives of magnitude ~1e3 (the
    library's last box is open on all three leading axes): the kernel must
    not fold the open widths into one product that overflows fp32, and must
    match the oracle's Monte-Carlo EHVI (Eq. 7) within the propagated bar."""
    inst = make_instance("tiny", seeds("tiny")[1], n_cand=4096 + 37)
    n = inst.n_cand
    y = inst.y_obs.astype(np.float64)
    Y = (np.stack([y[0], y[1], -0.5 * y[0] + 0.2 * y[1], 0.3 * y[0] - 0.6 * y[1]]) * 1000.0 + 500.0)
    Y = Y.astype(np.float32)
    M = 4
    ell = np.ascontiguousarray(inst.lengthscale[[0, 1, 0, 1]])
    sv = np.full(M, 1e6, np.float32)
    nv = np.full(M, 1e6 * float(inst.noise_var[0]), np.float32)
    ref = Y.min(axis=1)
    eps = Stream(4242, "eps4").normal(64 * M).reshape(64, M).astype(np.float32)
    L = S.scoot_gp_layout_init(inst.space, inst.n_obs, M)
    blob, _ = S.scoot_gp_prepare(inst.space, inst.x_obs, Y, ell, sv, nv, L)
    lo, hi, fs = S.scoot_boxes_build(Y, ref)
    assert np.all(np.isinf(hi[:, -1])) and np.any(np.all(np.isinf(hi[:, :-1]), axis=1))
    cand = cand_dev(inst)
    mask = torch.empty(n, dtype=torch.uint8, device="cuda")
    S.scoot_prune(ctx, inst.space, inst.clauses, cand, n, mask)
    acq = torch.empty(n, device="cuda")
    S.scoot_score_ehvi(ctx, L, dev(blob), cand, n, dev(lo), dev(hi), dev(eps), acq, mask)
    g = np_(acq)
    known = O.prune_mask(inst.space, inst.clauses, inst.cand, n)
    assert np.array_equal(np.isfinite(g), known)
    assert not np.any(np.isnan(g))
    idx = sample_idx(n, 512, 11)
    idx = idx[known[idx]]
    gps = [O.GP(inst.space, inst.x_obs, Y[m], ell[m], sv[m], nv[m]) for m in range(M)]
    mu, var, e_mu, e_var = posterior_tols(gps, np.ascontiguousarray(inst.cand[:, idx]))
    front = O.pareto_front(Y.T.astype(np.float64), ref.astype(np.float64))
    f = lambda a, b: O.ehvi_mc(a, b, eps, front, ref.astype(np.float64))
    want, tol = propagated_tol(f, mu, var, e_mu, e_var)
    assert np.any(want > 1e6)  # volumes at the scale of the objectives
    assert report_tol(f"score_ehvi M=4 at scale 1e3 (P={fs}, B={len(lo)})", g[idx], want, tol).max() <= 1.0


@pytest.mark.parametrize("tc", [1, 0], ids=["tensor", "simt"])
def test_score_ei_parity(S, ctx, tc):
    """Posterior + EI in one launch, at the full d10-ei pool, with either
    product of L^{-1} k (the tensor-core kernel's EI epilogue, the fused SIMT
    kernel)."""
    name = "d10-ei"
    inst = make_instance(name, seeds(name)[0])
    n = inst.n_cand
    L, state = gp_state(S, inst)
    cand = cand_dev(inst)
    mask = torch.empty(n, dtype=torch.uint8, device="cuda")
    S.scoot_prune(ctx, inst.space, inst.clauses, cand, n, mask)
    acq = torch.full((n,), 5.0, device="cuda")
    S.scoot_ctx_set_tensor_cores(ctx, tc)
    try:
        S.scoot_score_ei(ctx, L, state, cand, n, 1e-4, acq, mask)
        g = np_(acq)
    finally:
        S.scoot_ctx_set_tensor_cores(ctx, 1)
    known = O.prune_mask(inst.space, inst.clauses, inst.cand, n)
    assert np.array_equal(np.isfinite(g), known)
    top = np.argsort(-np.where(known, g, -np.inf))[:64]
    idx = np.union1d(sample_idx(n, 8192, 9), top)
    idx = idx[known[idx]]
    mu, var, e_mu, e_var = posterior_tols(oracle_gps(inst), np.ascontiguousarray(inst.cand[:, idx]))
    yb = float(inst.y_obs[0].max())
    f = lambda a, b: O.expected_improvement(a[:, 0], b[:, 0], yb, 1e-4)
    want, tol = propagated_tol(f, mu, var, e_mu, e_var)
    assert report_tol(f"score_ei d10-ei {'tensor' if tc else 'simt'}", g[idx], want, tol).max() <= 1.0


# ------------------------------------------------------------------ top-q (Section 4.7)

@pytest.mark.parametrize("n,q", [(1, 1), (7, 4), (1000, 1), (5000, 16), (100003, 17), (1 << 20, 64), (300, 64)])
def test_topq_bit_exact_on_generated_arrays(S, ctx, n, q):
    st = Stream(n * 131 + q, "topq")
    acq = np.round(st.normal(n) * 4.0).astype(np.float32) / 4  # many exact ties
    acq[st.uniform(n) < 0.05] = -np.inf
    acq[st.uniform(n) < 0.02] = np.nan
    mask = (st.uniform(n) < 0.7).astype(np.uint8)
    idx = torch.empty(q, dtype=torch.int64, device="cuda")
    val = torch.empty(q, device="cuda")
    cnt = torch.empty(1, dtype=torch.int32, device="cuda")
    for m in (None, mask):
        S.scoot_select_topq(ctx, dev(acq), n, q, idx, val, cnt, None if m is None else dev(m))
        want, wval, c = O.select_topq(acq.astype(np.float64), m, q)
        gi, gv, gc = np_(idx), np_(val), int(np_(cnt)[0])
        assert gc == c
        assert gi[:c].tolist() == want.tolist()
        assert np.array_equal(gv[:c], acq[want])
        assert np.all(gi[c:] == -1) and np.all(gv[c:] == -np.inf)


def test_topq_signed_zeros_are_one_value(S, ctx):
    """-0 and +0 compare equal in the selection rule (Section 4.7 order), so
    among interleaved -0/+0 values the lowest indices win, whatever the sign
    bit; the static entry point agrees."""
    n, q = 4099, 16
    cases = []
    for neg in (0, 1):  # -0 at the even indices, then at the odd ones
        a = np.zeros(n, np.float32)
        a[neg::2] = -0.0
        a[5] = -1.0
        a[n - 1] = -np.inf
        cases.append(a)
    assert np.signbit(cases[0][0]) and not np.signbit(cases[1][0])
    for a in cases:
        idx = torch.empty(q, dtype=torch.int64, device="cuda")
        val = torch.empty(q, device="cuda")
        cnt = torch.empty(1, dtype=torch.int32, device="cuda")
        S.scoot_select_topq(ctx, dev(a), n, q, idx, val, cnt)
        want, _, c = O.select_topq(a.astype(np.float64), None, q)
        assert int(np_(cnt)[0]) == c == q
        assert np_(idx).tolist() == want.tolist() == [0, 1, 2, 3, 4] + list(range(6, 17))
        assert np.all(np_(val) == 0.0)
        S.scoot_select_topq_static(dev(a), n, q, idx, val, cnt)
        assert np_(idx).tolist() == want.tolist()


def test_topq_degenerate(S, ctx):
    idx = torch.empty(4, dtype=torch.int64, device="cuda")
    val = torch.empty(4, device="cuda")
    cnt = torch.empty(1, dtype=torch.int32, device="cuda")
    acq = torch.full((100,), -math.inf, device="cuda")
    S.scoot_select_topq(ctx, acq, 100, 4, idx, val, cnt)
    assert int(np_(cnt)[0]) == 0 and np.all(np_(idx) == -1)
    S.scoot_select_topq(ctx, acq, 0, 4, idx, val, cnt)
    assert int(np_(cnt)[0]) == 0
    acq = torch.zeros(100, device="cuda")  # all tied: lowest indices win
    S.scoot_select_topq(ctx, acq, 100, 4, idx, val, cnt)
    assert np_(idx).tolist() == [0, 1, 2, 3]
    with pytest.raises(S.ScootError):
        S.scoot_select_topq(ctx, acq, 100, 65, idx, val, cnt)


# ------------------------------------------------------------------ whole round

@pytest.mark.parametrize("name", ["tiny", "d8-ehvi2", "d10-ei", "d10-ehvi3"])
def test_round_selects_valid_top_q(S, ctx, name):
    """Gate B: the picks of a full round are a valid top-q of the oracle's own
    acquisition values, up to swaps within the tolerance."""
    from paper_2408_04323_gb300.pipeline import RoundInputs, ScoringRound
    inst = make_instance(name, seeds(name)[0])
    w = inst.workload
    inp = RoundInputs(inst.space, inst.clauses, inst.nodes, inst.tree_offset, w.leaf_scale, w.delta_num,
                      w.delta_den, inst.x_obs, inst.y_obs, inst.lengthscale, inst.signal_var,
                      inst.noise_var, inst.ref, inst.eps, w.acq, w.q)
    rnd = ScoringRound(ctx, inp, inst.n_cand)
    idx, val, cnt = rnd.run(cand_dev(inst), inst.n_cand)
    ctx.check()
    gi, gv, c = np_(idx), np_(val), int(np_(cnt)[0])
    known = O.prune_mask(inst.space, inst.clauses, inst.cand, inst.n_cand)
    votes = O.rf_votes(inst.nodes, inst.tree_offset, inst.space, inst.cand, inst.n_cand)
    feas = known & O.pof_feasible(votes, inst.n_trees, w.leaf_scale, w.delta_num, w.delta_den)
    assert np.array_equal(np_(rnd.mask).astype(bool), feas)
    assert c == min(w.q, int(feas.sum()))
    g = np_(rnd.acq)
    # oracle acquisition on the GPU's best candidates and the next ones by the GPU's ranking
    order = np.argsort(-np.where(feas, g, -np.inf), kind="stable")[:max(4 * w.q, 32)]
    mu, var, e_mu, e_var = posterior_tols(oracle_gps(inst), np.ascontiguousarray(inst.cand[:, order]))
    if w.acq == "ei":
        yb = float(inst.y_obs[0].max())
        f = lambda a, b: O.expected_improvement(a[:, 0], b[:, 0], yb, 1e-4)
    else:
        front = O.pareto_front(inst.y_obs.T, inst.ref)
        f = lambda a, b: O.ehvi_mc(a, b, inst.eps, front, inst.ref)
    oacq, tol = propagated_tol(f, mu, var, e_mu, e_var)
    pos = [int(np.nonzero(order == i)[0][0]) for i in gi[:c]]
    assert report_tol(f"round {name} picked acq", gv[:c], oacq[pos], tol[pos]).max() <= 1.0
    # every pick is within tolerance of the oracle's c-th best value among these candidates
    kth = np.sort(oacq)[::-1][c - 1]
    assert np.all(oacq[pos] >= kth - tol[pos] - tol[np.argsort(oacq)[::-1][c - 1]])
    # and no candidate of a seeded sample of the feasible pool (which the GPU
    # may have under-scored) beats the weakest pick by more than the two
    # values' tolerances: the oracle's own top of the sample is below the picks
    live = np.nonzero(feas)[0]
    k = {"d10-ehvi3": 96}.get(name, 2048)
    samp = live[sample_idx(len(live), k, 31)]
    samp = samp[~np.isin(samp, gi[:c])]  # the picks themselves may rank above the weakest pick
    mu_s, var_s, e_mu_s, e_var_s = posterior_tols(oracle_gps(inst), np.ascontiguousarray(inst.cand[:, samp]))
    oacq_s, tol_s = propagated_tol(f, mu_s, var_s, e_mu_s, e_var_s)
    weakest = int(np.argmin(oacq[pos]))
    beat = (oacq_s - oacq[pos][weakest]) / (tol_s + tol[pos][weakest])
    print(f"[gate-b] {name}: {len(samp)} sampled feasible candidates, oracle's best of them "
          f"{oacq_s.max():.6g} vs the weakest pick {oacq[pos][weakest]:.6g}; max excess/tol {beat.max():.3f}")
    assert beat.max() <= 1.0


def test_out_of_range_category_is_reported_not_read(S, ctx):
    """A category index outside 0..n_choices-1 is clamped inside the kernel
    (no read outside the state) and reported as SCOOT_EDEVICE by the next
    context check; the check clears the flag."""
    inst = make_instance("d8-ehvi2", seeds("d8-ehvi2")[2], n_cand=256)
    cat_cols = [c for c in range(inst.d) if inst.space[c]["kind"] == 2]
    words = inst.cand.copy()
    words[cat_cols[0], 5] = np.uint32(7)
    L, state = gp_state(S, inst)
    mean = torch.empty((2, 256), device="cuda")
    var = torch.empty((2, 256), device="cuda")
    S.scoot_gp_posterior(ctx, L, state, dev(words.view(np.int32)), 256, mean, var)
    with pytest.raises(S.ScootError) as e:
        ctx.check()
    assert e.value.status == -4
    ctx.check()  # cleared
    assert np.all(np.isfinite(np_(mean)))
