"""Pins of the fp64 oracle against closed forms, invariants, brute force and
library routines (no GPU).  Each group names the equation or passage of the
paper it checks."""
import itertools
import math
import os

import numpy as np
import pytest
from scipy import integrate, special

import oracle as O
from workloads import (CATEGORICAL, CLAUSE_DTYPE, CONTINUOUS, INT_LOG, INT_UNIFORM, NODE_DTYPE,
                       PARAM_DTYPE, Stream, make_instance, seeds, WORKLOADS)


def _space(*params):
    a = np.zeros(len(params), PARAM_DTYPE)
    for i, p in enumerate(params):
        a[i] = p
    return a


def _clause(guards=(), terms=(), rhs=0):
    c = np.zeros(1, CLAUSE_DTYPE)
    c[0]["n_guard"] = len(guards)
    for g, (p, v) in enumerate(guards):
        c[0]["guard_param"][g] = p
        c[0]["guard_value"][g] = v
    c[0]["n_term"] = len(terms)
    for t, (p, k) in enumerate(terms):
        c[0]["term_param"][t] = p
        c[0]["coef"][t] = k
    c[0]["rhs"] = rhs
    return c


def _words_int(cols):
    return np.stack([np.asarray(c, np.int32).view(np.uint32) for c in cols])


# ------------------------------------------------------------------ Eq. (2)

@pytest.mark.parametrize("K", [1, 2, 7, 33])
def test_prune_closed_form_counts(K):
    """#{(a, b) in [1..K]^2 : a >= b} = K(K+1)/2; #{a + b >= K + 1} = K(K+1)/2."""
    a, b = np.meshgrid(np.arange(1, K + 1), np.arange(1, K + 1), indexing="ij")
    words = _words_int([a.ravel(), b.ravel()])
    sp = _space((INT_UNIFORM, 0, 1, K), (INT_UNIFORM, 0, 1, K))
    n = K * K
    m = O.prune_mask(sp, _clause(terms=((0, 1), (1, -1)), rhs=0), words, n)
    assert m.sum() == K * (K + 1) // 2
    m = O.prune_mask(sp, _clause(terms=((0, 1), (1, 1)), rhs=K + 1), words, n)
    assert m.sum() == K * (K + 1) // 2
    # strict a > b via rhs 1: K(K-1)/2
    m = O.prune_mask(sp, _clause(terms=((0, 1), (1, -1)), rhs=1), words, n)
    assert m.sum() == K * (K - 1) // 2


def test_prune_guards_and_degenerate_clauses():
    K = 6
    a, b, c = np.meshgrid(np.arange(1, K + 1), np.arange(1, K + 1), np.arange(3), indexing="ij")
    words = _words_int([a.ravel(), b.ravel(), c.ravel()])
    sp = _space((INT_UNIFORM, 0, 1, K), (INT_UNIFORM, 0, 1, K), (CATEGORICAL, 3, 0, 0))
    n = words.shape[1]
    # guard c == 1 => a >= b : the two other categories pass untouched
    m = O.prune_mask(sp, _clause(guards=((2, 1),), terms=((0, 1), (1, -1))), words, n)
    assert m.sum() == 2 * K * K + K * (K + 1) // 2
    # a guard no candidate meets (category 5 of 3) leaves everything feasible
    m = O.prune_mask(sp, _clause(guards=((2, 5),), terms=((0, 1),), rhs=10 ** 9), words, n)
    assert m.all()
    # two guards must both hold
    m = O.prune_mask(sp, _clause(guards=((2, 0), (0, 1)), terms=((1, 1),), rhs=K + 1), words, n)
    assert m.sum() == n - K
    # empty sum: 0 >= 0 holds, 0 >= 1 fails everywhere
    assert O.prune_mask(sp, _clause(rhs=0), words, n).all()
    assert not O.prune_mask(sp, _clause(rhs=1), words, n).any()
    # several clauses AND together
    cl = np.concatenate([_clause(terms=((0, 1), (1, -1))), _clause(terms=((1, 1),), rhs=K)])
    m = O.prune_mask(sp, cl, words, n)
    assert m.sum() == 3 * 1  # only a = b = K survives, for each category


def test_prune_exact_with_large_coefficients():
    """Exact integer arithmetic: 2^40 a - 2^40 b - 1 >= 0 iff a > b (float64 would not tell)."""
    vals = np.array([[2 ** 20, 2 ** 20], [2 ** 20 + 1, 2 ** 20], [5, 7]]).T
    words = _words_int(vals)
    sp = _space((INT_UNIFORM, 0, 1, 2 ** 21), (INT_UNIFORM, 0, 1, 2 ** 21))
    m = O.prune_mask(sp, _clause(terms=((0, 2 ** 40), (1, -(2 ** 40))), rhs=1), words, 3)
    assert m.tolist() == [False, True, False]


def test_prune_fail_fraction_of_ten_parameter_space():
    """The ten-parameter vLLM space loses about 40% of a uniform pool."""
    inst = make_instance("d10-ei", seeds("d10-ei")[0], n_cand=1 << 16)
    m = O.prune_mask(inst.space, inst.clauses, inst.cand, inst.n_cand)
    assert abs((1.0 - m.mean()) - 0.40) <= 0.03


# ------------------------------------------------------------------ Eq. (3)

def _load_forest(path):
    trees = {}
    cases = []
    for line in open(path):
        f = line.split()
        if not f or f[0].startswith("#"):
            continue
        if f[0] == "node":
            t, i = int(f[1]), int(f[2])
            if f[3] == "split":
                trees.setdefault(t, {})[i] = (float(f[5]), int(f[6]), int(f[4]), 0)
            else:
                trees.setdefault(t, {})[i] = (float(f[4]), 0, 0, O.NODE_LEAF)
        elif f[0] == "case":
            cases.append((float(f[1]), float(f[2]), int(f[3])))
    nodes, offs = [], [0]
    for t in sorted(trees):
        for i in sorted(trees[t]):
            nodes.append(trees[t][i])
        offs.append(len(nodes))
    arr = np.zeros(len(nodes), NODE_DTYPE)
    for j, nd in enumerate(nodes):
        arr[j] = nd
    return arr, np.array(offs, np.int32), cases


def test_forest_hand_built(golden_dir):
    nodes, offs, cases = _load_forest(os.path.join(golden_dir, "forest_hand.txt"))
    sp = _space((CONTINUOUS, 0, 0, 100), (CONTINUOUS, 0, 0, 100))
    x = np.array([[c[0], c[1]] for c in cases], np.float32)
    words = np.ascontiguousarray(x.T).view(np.uint32)
    want = [c[2] for c in cases]
    assert O.rf_votes(nodes, offs, sp, words, len(cases)).tolist() == want
    assert [O.rf_votes_one(nodes, offs, xi.astype(np.float64)) for xi in x] == want


def test_forest_constant_leaves_and_tree_order():
    rng = Stream(7, "forest-test")
    inst = make_instance("tiny", 1001, n_cand=512)
    # constant forest: every leaf votes c => votes = T c
    nodes = inst.nodes.copy()
    leaf = (nodes["flags"] & O.NODE_LEAF) != 0
    nodes["val"][leaf] = 17
    v = O.rf_votes(nodes, inst.tree_offset, inst.space, inst.cand, inst.n_cand)
    assert (v == 17 * inst.n_trees).all()
    # reversing the tree order does not change the votes
    T = inst.n_trees
    perm = np.array(rng.integers(0, 1000, T).argsort())
    parts = [inst.nodes[inst.tree_offset[t]:inst.tree_offset[t + 1]] for t in perm]
    offs = np.zeros(T + 1, np.int32)
    offs[1:] = np.cumsum([len(p) for p in parts])
    v1 = O.rf_votes(inst.nodes, inst.tree_offset, inst.space, inst.cand, inst.n_cand)
    v2 = O.rf_votes(np.concatenate(parts), offs, inst.space, inst.cand, inst.n_cand)
    assert (v1 == v2).all()
    # the recursive walk agrees with the vectorised one
    x = O.decode(inst.space, inst.cand, 64)
    assert [O.rf_votes_one(inst.nodes, inst.tree_offset, xi) for xi in x] == v1[:64].tolist()


def test_tree_grown_to_purity_reproduces_labels():
    """A single CART tree without bootstrap, grown without a depth limit on
    distinct points, sends every training point to a leaf of its own label."""
    from workloads.generate import _grow, _layout
    w = WORKLOADS["d8-ehvi2"]
    st = Stream(11, "purity")
    from workloads.generate import draw_configs, stored_values
    X = stored_values(w, draw_configs(w, st, 64))
    lab = (st.uniform(64) < 0.5).astype(np.float64)
    tree = _layout(_grow(X, lab, 0, 64, 255))
    offs = np.array([0, len(tree)], np.int32)
    words = draw_configs(w, Stream(11, "purity"), 64)
    sp = np.zeros(w.d, PARAM_DTYPE)
    for i, p in enumerate(w.params):
        sp[i] = (p.kind, p.n_choices, p.lo, p.hi)
    v = O.rf_votes(tree, offs, sp, words, 64)
    assert (v == 255 * lab).all()


def test_pof_threshold_inclusive():
    T, V = 100, 255
    thr = 10 * V * T // 20  # Delta = 0.5 -> votes >= 12750
    v = np.array([thr - 1, thr, thr + 1, 0, V * T])
    assert O.pof_feasible(v, T, V, 10, 20).tolist() == [False, True, True, False, True]
    # Delta = 0.25 and 0.75 (the bounds of Algorithm 1)
    assert O.pof_feasible(np.array([V * T // 4]), T, V, 5, 20).tolist() == [True]
    assert O.pof_feasible(np.array([3 * V * T // 4 - 1]), T, V, 15, 20).tolist() == [False]


# ------------------------------------------------------------------ GP, Section 4.3

@pytest.mark.parametrize("nu,kernel", [(2.5, O.MATERN52), (1.5, O.MATERN32)])
def test_matern_matches_bessel_form(nu, kernel):
    """k(r) = s 2^(1-nu)/Gamma(nu) (sqrt(2 nu) r)^nu K_nu(sqrt(2 nu) r)."""
    r = np.linspace(1e-3, 8.0, 400)
    z = math.sqrt(2 * nu) * r
    ref = 1.7 * 2 ** (1 - nu) / special.gamma(nu) * z ** nu * special.kv(nu, z)
    assert np.allclose(O.matern(r, 1.7, kernel), ref, rtol=1e-12, atol=1e-14)
    assert O.matern(0.0, 1.7, kernel) == pytest.approx(1.7)
    assert np.all(np.diff(O.matern(r, 1.0, kernel)) < 0)


def test_features_and_distance():
    sp = _space((INT_LOG, 0, 4, 4096), (INT_UNIFORM, 0, 2, 10), (CONTINUOUS, 0, 0.5, 1.0),
                (CATEGORICAL, 3, 0, 0))
    x = np.array([[4, 2, 0.5, 0], [4096, 10, 1.0, 2], [128, 6, 0.75, 1]], np.float64)
    u, cat = O.gp_features(sp, x)
    assert np.allclose(u[:, :3], [[0, 0, 0], [1, 1, 1], [0.5, 0.5, 0.5]])
    assert cat.tolist() == [False, False, False, True]
    ell = np.array([0.5, 1.0, 2.0, 0.25])
    r = O.scaled_distance(u, u, cat, ell)
    # rows 0 and 1: (1/0.5)^2 + 1 + (1/2)^2 + categorical 1/0.0625
    assert r[0, 1] ** 2 == pytest.approx(4 + 1 + 0.25 + 16)
    assert np.allclose(r, r.T) and np.allclose(np.diag(r), 0)


def _toy_gp(n, seed=3, noise=1e-3, ell=0.4, d=3):
    st = Stream(seed, "toy-gp")
    sp = _space(*[(CONTINUOUS, 0, 0.0, 1.0)] * d)
    X = st.uniform(n * d).reshape(d, n).astype(np.float32)
    y = st.normal(n).astype(np.float32)
    gp = O.GP(sp, X.view(np.uint32), y, np.full(d, ell), 1.0, noise)
    return sp, X, y, gp


def test_gp_single_observation_closed_form():
    """n = 1: mu = k y / (s + tau^2), sigma^2 = s - k^2 / (s + tau^2)."""
    sp, X, y, gp = _toy_gp(1, noise=0.3)
    st = Stream(5, "cands")
    C = st.uniform(3 * 50).reshape(3, 50).astype(np.float32)
    mu, var = gp.posterior(C.view(np.uint32))
    k = gp.cov(O.gp_features(sp, O.decode(sp, C.view(np.uint32)))[0], gp.u_obs)[:, 0]
    assert np.allclose(mu, k * y[0] / 1.3, rtol=1e-12)
    assert np.allclose(var, 1.0 - k * k / 1.3, rtol=1e-12)


def test_gp_interpolates_as_noise_vanishes():
    sp, X, y, gp = _toy_gp(12, noise=1e-10)
    mu, var = gp.posterior(X.view(np.uint32))
    assert np.allclose(mu, y, atol=1e-5)
    assert np.all(var < 1e-6)


def test_gp_far_field_and_bounds():
    sp, X, y, gp = _toy_gp(20, ell=0.05)
    st = Stream(9, "far")
    C = st.uniform(3 * 200).reshape(3, 200).astype(np.float32)
    far = (C + 5.0).astype(np.float32)  # 100 lengthscales from every observation
    mu, var = gp.posterior(far.view(np.uint32))
    assert np.all(np.abs(mu) < 1e-12) and np.allclose(var, 1.0, atol=1e-12)
    sp, X, y, gp = _toy_gp(40, ell=0.3)
    mu, var = gp.posterior(C.view(np.uint32))
    assert np.all(var >= 0) and np.all(var <= 1.0 + 1e-12)


def test_gp_permutation_invariant():
    sp, X, y, gp = _toy_gp(25)
    perm = np.array(Stream(2, "perm").integers(0, 10 ** 6, 25).argsort())
    gp2 = O.GP(sp, np.ascontiguousarray(X[:, perm]).view(np.uint32), y[perm], np.full(3, 0.4), 1.0, 1e-3)
    C = Stream(4, "c").uniform(300).reshape(3, 100).astype(np.float32).view(np.uint32)
    m1, v1 = gp.posterior(C)
    m2, v2 = gp2.posterior(C)
    assert np.allclose(m1, m2, rtol=1e-10, atol=1e-12) and np.allclose(v1, v2, rtol=1e-10, atol=1e-12)


def _gauss_jordan_inverse(A):
    A = np.array(A, np.float64)
    n = len(A)
    M = np.concatenate([A, np.eye(n)], axis=1)
    for c in range(n):
        p = c + int(np.argmax(np.abs(M[c:, c])))
        M[[c, p]] = M[[p, c]]
        M[c] /= M[c, c]
        for r in range(n):
            if r != c:
                M[r] -= M[r, c] * M[c]
    return M[:, n:]


@pytest.mark.parametrize("n", [2, 5, 8])
def test_gp_matches_explicit_inverse(n):
    """The Cholesky route equals the printed formulas with an explicit inverse."""
    sp, X, y, gp = _toy_gp(n, noise=0.05)
    C = Stream(8, "c").uniform(3 * 40).reshape(3, 40).astype(np.float32).view(np.uint32)
    u, _ = O.gp_features(sp, O.decode(sp, C))
    Kinv = _gauss_jordan_inverse(gp.cov(gp.u_obs, gp.u_obs) + 0.05 * np.eye(n))
    ks = gp.cov(u, gp.u_obs)
    mu_ref = ks @ Kinv @ y.astype(np.float64)
    var_ref = 1.0 - np.einsum("ij,jk,ik->i", ks, Kinv, ks)
    mu, var = gp.posterior(C)
    assert np.allclose(mu, mu_ref, rtol=1e-10, atol=1e-12)
    assert np.allclose(var, var_ref, rtol=1e-9, atol=1e-12)


# ------------------------------------------------------------------ EI, Eq. (6)

def test_ei_closed_form_matches_quadrature():
    xi = 1e-4
    for mu, sd, yb in [(0.0, 1.0, 0.0), (-1.3, 0.2, 0.5), (2.0, 0.5, 1.0), (0.3, 3.0, 2.0), (-4, 0.7, 0.0)]:
        f = lambda t: max(0.0, mu + sd * t + xi - yb) * math.exp(-0.5 * t * t) / math.sqrt(2 * math.pi)
        lo = (yb - xi - mu) / sd
        q, _ = integrate.quad(f, max(lo, -12.0), 12.0, epsabs=1e-13, epsrel=1e-12, limit=200)
        assert O.expected_improvement(mu, sd * sd, yb, xi) == pytest.approx(q, rel=1e-9, abs=1e-12)


def test_ei_limits_and_monotonicity():
    a = np.array([-1.0, 0.0, 0.5])
    assert np.allclose(O.expected_improvement(a, 0.0, 0.0, 0.0), np.maximum(a, 0))
    assert np.allclose(O.expected_improvement(a, 1e-24, 0.0, 0.0), np.maximum(a, 0), atol=1e-11)
    mus = np.linspace(-3, 3, 50)
    assert np.all(np.diff(O.expected_improvement(mus, 0.25, 0.0)) > 0)
    sds = np.linspace(0.01, 3, 50)
    assert np.all(np.diff(O.expected_improvement(0.2, sds ** 2, 0.5)) > 0)


# ------------------------------------------------------------------ HV, EHVI, Eq. (7), Eq. (8)

def _hv2d_rectangles(points, ref):
    """Section 4.4: sum of rectangles between the sorted front and r."""
    P = [p for p in points if p[0] > ref[0] and p[1] > ref[1]]
    P.sort(key=lambda p: -p[0])
    hv, top = 0.0, ref[1]
    for x, y in P:
        if y > top:
            hv += (x - ref[0]) * (y - top)
            top = y
    return hv


def _hv_lattice(points, ref, top):
    """Brute force on integers: count unit cells [z, z+1) dominated by some point."""
    M = len(ref)
    count = 0
    for z in itertools.product(*[range(ref[j], top) for j in range(M)]):
        if any(all(p[j] >= z[j] + 1 for j in range(M)) for p in points):
            count += 1
    return count


def test_hv_worked_example(golden_dir):
    pts, hvis = [], []
    for line in open(os.path.join(golden_dir, "hv_2d_worked.txt")):
        f = line.split()
        if not f or f[0].startswith("#"):
            continue
        if f[0] == "ref":
            ref = np.array([float(f[1]), float(f[2])])
        elif f[0] == "point":
            pts.append([float(f[1]), float(f[2])])
        elif f[0] == "hv":
            hv = float(f[1])
        elif f[0] == "hvi":
            hvis.append(([float(f[1]), float(f[2])], float(f[3])))
    pts = np.array(pts)
    assert O.hypervolume(pts, ref) == pytest.approx(hv)
    front = O.pareto_front(pts, ref)
    assert len(front) == 3
    lo, hi = O.nondominated_cells(front, ref)
    for y, want in hvis:
        assert O.hvi_cells(np.array([y]), lo, hi)[0] == pytest.approx(want)


def test_single_point_hv_eq8(golden_dir):
    for line in open(os.path.join(golden_dir, "hv_single_point.txt")):
        f = line.split()
        if not f or f[0].startswith("#"):
            continue
        y1, y2, r1, r2, want = map(float, f)
        assert O.hypervolume(np.array([[y1, y2]]), np.array([r1, r2])) == pytest.approx(want)


@pytest.mark.parametrize("M,top,npts", [(2, 12, 9), (3, 7, 8)])
def test_hv_lattice_brute_force(M, top, npts):
    st = Stream(M, "lattice")
    for trial in range(4):
        pts = st.integers(1, top, npts * M).reshape(npts, M)
        ref = np.zeros(M, np.int64)
        want = _hv_lattice(pts.tolist(), ref.tolist(), top)
        assert O.hypervolume(pts.astype(float), ref.astype(float)) == pytest.approx(want)
        if M == 2:
            assert _hv2d_rectangles(pts.astype(float).tolist(), [0.0, 0.0]) == pytest.approx(want)


@pytest.mark.parametrize("M", [2, 3])
def test_hvi_by_cells_equals_hv_difference(M):
    st = Stream(40 + M, "hvi")
    ref = np.zeros(M)
    pts = st.uniform(10 * M).reshape(10, M) * 4.0
    front = O.pareto_front(pts, ref)
    base = O.hypervolume(front, ref)
    lo, hi = O.nondominated_cells(front, ref)
    ys = st.uniform(60 * M).reshape(60, M) * 5.0 - 0.5
    got = O.hvi_cells(ys, lo, hi)
    want = [O.hypervolume(np.vstack([front, y]), ref) - base for y in ys]
    assert np.allclose(got, want, rtol=1e-12, atol=1e-12)
    # permuting the points leaves HV unchanged
    perm = np.array(st.integers(0, 10 ** 6, len(pts)).argsort())
    assert O.hypervolume(pts[perm], ref) == pytest.approx(O.hypervolume(pts, ref), rel=1e-14)
    # a dominated point improves nothing
    assert O.hvi_cells(front[:1] * 0.999, lo, hi)[0] == pytest.approx(0.0, abs=1e-14)
    # cells clipped to a bounding box plus HV fill the box
    box = np.full(M, 6.0)
    clipped = np.prod(np.maximum(np.minimum(hi, box) - lo, 0), axis=1).sum()
    assert clipped + base == pytest.approx(np.prod(box - ref), rel=1e-12)


def test_empty_front_single_cell():
    ref = np.array([0.5, -1.0])
    lo, hi = O.nondominated_cells(np.zeros((0, 2)), ref)
    assert len(lo) == 1
    y = np.array([[1.5, 2.0], [0.0, 3.0]])
    assert np.allclose(O.hvi_cells(y, lo, hi), [3.0, 0.0])


def _ehvi_analytic(mu, sd, lo, hi):
    """Independent Gaussians: E prod_j clip_j = prod_j E clip_j per cell, with
    E[max(0, min(Y, u) - l)] = int_l^u P(Y > t) dt in closed form."""
    def g(t, m, s):  # int_{-inf}^{t} Phi((x - m)/s) dx
        z = (t - m) / s
        return s * (z * O.norm_cdf(z) + O.norm_pdf(z))
    tot = 0.0
    for l, u in zip(lo, hi):
        prod = 1.0
        for j in range(len(mu)):
            inner = (u[j] - l[j]) if np.isfinite(u[j]) else None
            # int_l^u (1 - Phi) = (u - l) - [G(u) - G(l)], G = int Phi
            if np.isfinite(u[j]):
                val = (u[j] - l[j]) - (g(u[j], mu[j], sd[j]) - g(l[j], mu[j], sd[j]))
            else:
                # int_l^inf (1 - Phi((t-m)/s)) dt = s psi((m - l)/s)
                z = (mu[j] - l[j]) / sd[j]
                val = sd[j] * (z * O.norm_cdf(z) + O.norm_pdf(z))
            prod *= val
        tot += prod
    return tot


@pytest.mark.parametrize("M", [2, 3])
def test_mc_ehvi_converges_to_analytic(M):
    st = Stream(60 + M, "ehvi-conv")
    ref = np.zeros(M)
    front = O.pareto_front(st.uniform(8 * M).reshape(8, M) * 2.0, ref)
    lo, hi = O.nondominated_cells(front, ref)
    mu = np.full(M, 1.2)
    sd = np.array([0.5, 0.8, 0.3][:M])
    S = 40000
    eps = st.normal(S * M).reshape(S, M)
    vals = O.hvi_cells(mu + sd * eps, lo, hi)
    est = vals.mean()
    se = vals.std() / math.sqrt(S)
    assert abs(est - _ehvi_analytic(mu, sd, lo, hi)) < 4 * se
    # the oracle's MC EHVI is that mean, and its exact EHVI is the test's own closed form
    e = O.ehvi_mc(mu[None, :], (sd ** 2)[None, :], eps, front, ref)[0]
    assert e == pytest.approx(est, rel=1e-12)
    x = O.ehvi_analytic(mu[None, :], (sd ** 2)[None, :], front, ref)[0]
    assert x == pytest.approx(_ehvi_analytic(mu, sd, lo, hi), rel=1e-10)
    assert abs(est - x) < 4 * se


def test_exact_ehvi_limits_and_quadrature():
    """sigma -> 0 gives the deterministic HVI(mu); for M = 2 the exact EHVI
    equals 2-D quadrature of HVI(y) against the product density."""
    st = Stream(71, "ehvi-exact")
    ref = np.zeros(2)
    front = O.pareto_front(st.uniform(12).reshape(6, 2) * 2.0, ref)
    lo, hi = O.nondominated_cells(front, ref)
    for mu in ([1.1, 0.7], [2.5, 0.1], [-0.3, 1.9]):
        mu = np.array(mu)
        got = O.ehvi_analytic(mu[None, :], np.zeros((1, 2)), front, ref)[0]
        assert got == pytest.approx(O.hvi_cells(mu, lo, hi)[0], rel=1e-12, abs=1e-14)
    mu, sd = np.array([1.0, 0.8]), np.array([0.4, 0.25])
    dens = lambda y, m, s: math.exp(-0.5 * ((y - m) / s) ** 2) / (s * math.sqrt(2 * math.pi))
    # HVI is piecewise bilinear with kinks on the grid lines: nested quad with those breakpoints
    kinks = [np.unique(np.concatenate([[0.0], front[:, j]])) for j in range(2)]
    box = [(mu[j] - 9 * sd[j], mu[j] + 9 * sd[j]) for j in range(2)]

    def inner(y1):
        g = lambda y0: O.hvi_cells(np.array([y0, y1]), lo, hi)[0] * dens(y0, mu[0], sd[0])
        pts = [k for k in kinks[0] if box[0][0] < k < box[0][1]]
        return integrate.quad(g, *box[0], points=pts, epsabs=1e-12, epsrel=1e-10, limit=200)[0]

    pts = [k for k in kinks[1] if box[1][0] < k < box[1][1]]
    q, _ = integrate.quad(lambda y1: inner(y1) * dens(y1, mu[1], sd[1]), *box[1], points=pts,
                          epsabs=1e-11, epsrel=1e-9, limit=200)
    got = O.ehvi_analytic(mu[None, :], (sd ** 2)[None, :], front, ref)[0]
    assert got == pytest.approx(q, rel=1e-6, abs=1e-9)
    # psi(a) = E[max(0, Y - a)] against quadrature
    for m, s_, a in [(0.3, 0.7, 0.1), (-1.0, 0.2, 0.5), (2.0, 1.5, -1.0)]:
        qq, _ = integrate.quad(lambda y: max(0.0, y - a) * dens(y, m, s_), a, m + 14 * s_, epsabs=1e-13, limit=200)
        assert float(O.expected_excess(m, s_, a)) == pytest.approx(qq, rel=1e-9, abs=1e-13)


# ------------------------------------------------------------------ top-q, Section 4.7

def test_topq_against_repeated_argmax():
    st = Stream(77, "topq")
    for trial in range(20):
        n = int(st.integers(1, 300, 1)[0])
        acq = np.round(st.normal(n), 1)  # many ties
        acq[st.uniform(n) < 0.1] = -np.inf
        acq[st.uniform(n) < 0.05] = np.nan
        mask = st.uniform(n) < 0.8
        q = int(st.integers(1, 40, 1)[0])
        idx, val, cnt = O.select_topq(acq, mask, q)
        # brute force: q rounds of "largest value, lowest index" over the eligible set
        alive = [i for i in range(n) if mask[i] and not np.isnan(acq[i]) and acq[i] > -np.inf]
        want = []
        for _ in range(q):
            if not alive:
                break
            best = alive[0]
            for i in alive:
                if acq[i] > acq[best]:
                    best = i
            want.append(best)
            alive.remove(best)
        assert idx.tolist() == want and cnt == len(want)


# ------------------------------------------------------------------ fantasies (refit form)

def test_fantasy_refit_properties():
    """Kriging believer: conditioning on y_p = mu(x_p) leaves mu unchanged;
    sigma^2(x_p) becomes s t / (s + t) (s = sigma^2(x_p), t = tau^2); the
    refit variance equals the rank-1 downdate sigma^2 - c(x)^2 with
    c(x) = k_post(x, x_p) / sqrt(s + t)."""
    sp, X, y, gp = _toy_gp(30, noise=2e-3)
    C = Stream(12, "c").uniform(3 * 300).reshape(3, 300).astype(np.float32).view(np.uint32)
    u, _ = O.gp_features(sp, O.decode(sp, C))
    mu0, var0 = gp.posterior_u(u)
    p = 17
    kstar = gp.cov(u, gp.u_obs)
    Kn = gp.cov(gp.u_obs, gp.u_obs) + 2e-3 * np.eye(30)
    kpost = gp.cov(u, u[p:p + 1])[:, 0] - kstar @ np.linalg.solve(Kn, kstar[p])
    c = kpost / math.sqrt(var0[p] + 2e-3)
    gp.add_observations(u[p:p + 1], [mu0[p]])
    mu1, var1 = gp.posterior_u(u)
    assert np.allclose(mu1, mu0, rtol=1e-9, atol=1e-11)
    s, t = var0[p], 2e-3
    assert var1[p] == pytest.approx(s * t / (s + t), rel=1e-8)
    assert np.allclose(var1, np.maximum(var0 - c * c, 0), rtol=1e-8, atol=1e-11)


def _hv2(points, ref):
    """2-D hypervolume by the textbook sweep: points strictly above r, taken
    in decreasing first objective, each adding the strip of its second
    objective above the best one seen so far."""
    P = sorted((p for p in np.asarray(points, np.float64) if p[0] > ref[0] and p[1] > ref[1]),
               key=lambda p: (-p[0], -p[1]))
    hv, top = 0.0, float(ref[1])
    for p0, p1 in P:
        if p1 > top:
            hv += (p0 - ref[0]) * (p1 - top)
            top = p1
    return hv


def _fantasy_from_scratch(inst, q, feasible):
    """Sequential kriging-believer picks recomputed step by step from the
    definitions, sharing nothing with the oracle's loop but GP and the
    decoding: at step j a NEW GP per objective on the observations plus the
    previous picks' words (fantasised values, noise tau^2), the fantasised
    value of a pick taken as that step's own posterior mean at it, the front
    as the points (observed and fantasised) no other point dominates, EHVI as
    the mean over the base samples of HV(front + y_s) - HV(front) by the 2-D
    sweep, picked candidates excluded, argmax with the lowest index."""
    M = inst.n_obj
    words = inst.cand[:, :inst.n_cand]
    eligible = np.asarray(feasible, bool).copy()
    picks, acqs, vars_, fvals, fronts = [], [], [], [], []
    repick_needed = False
    for j in range(q):
        xw = np.concatenate([inst.x_obs, words[:, picks]], axis=1) if picks else inst.x_obs
        gps = [O.GP(inst.space, xw, np.concatenate([inst.y_obs[m].astype(np.float64), [f[m] for f in fvals]]),
                    inst.lengthscale[m], inst.signal_var[m], inst.noise_var[m]) for m in range(M)]
        mv = [gp.posterior(words) for gp in gps]
        mu = np.stack([a for a, _ in mv], 1)
        var = np.stack([b for _, b in mv], 1)
        pts = np.concatenate([inst.y_obs.T.astype(np.float64), np.array(fvals).reshape(-1, M)])
        front = [p for p in pts if p[0] > inst.ref[0] and p[1] > inst.ref[1]
                 and not any(np.all(z >= p) and np.any(z > p) for z in pts)]
        base = _hv2(front, inst.ref)
        sd = np.sqrt(var)
        a = np.full(len(mu), -np.inf)
        for i in range(len(mu)):
            if feasible[i]:
                ys = mu[i] + sd[i] * inst.eps
                a[i] = np.mean([_hv2(front + [y], inst.ref) - base for y in ys])
        val = np.where(eligible, a, -np.inf)
        if not np.any(np.isfinite(val)):
            break
        p = int(np.flatnonzero(val == val.max())[0])
        repick_needed |= bool(picks) and int(np.flatnonzero(a == a[feasible].max())[0]) in picks
        picks.append(p)
        acqs.append(a)
        vars_.append(var)
        fronts.append(np.array(front).reshape(-1, M))
        fvals.append(np.array([gp.posterior(words[:, [p]])[0][0] for gp in gps]))
        eligible[p] = False
    return picks, acqs, vars_, fronts, repick_needed


@pytest.mark.parametrize("noise", [None, 0.3])
def test_fantasy_picks_equal_a_from_scratch_recomputation(noise):
    """Pins the oracle's sequential-pick loop (refit GP, fantasised front,
    exclusion, argmax) against a recomputation from scratch at every step.
    With a large noise variance a picked candidate keeps a high EHVI after
    its own fantasy, so the exclusion of picked candidates decides a pick."""
    import dataclasses
    inst = make_instance("tiny", seeds("tiny")[2], n_cand=160)
    if noise is not None:
        inst = dataclasses.replace(inst, noise_var=np.full(inst.n_obj, noise, np.float32))
    feas = Stream(77, "feas").uniform(inst.n_cand) < 0.8
    q = 5
    ref = O.fantasy_picks(inst, q, feas)
    picks, acqs, vars_, fronts, repick = _fantasy_from_scratch(inst, q, feas)
    assert ref["picks"] == picks
    for j in range(q):
        ok = np.isfinite(acqs[j])
        assert np.array_equal(ok, feas)
        want = np.where(np.isin(np.arange(inst.n_cand), picks[:j]), -np.inf, acqs[j])
        got = ref["acq"][j]
        both = np.isfinite(got) & np.isfinite(want)
        assert np.array_equal(np.isfinite(got), np.isfinite(want))
        assert np.allclose(got[both], want[both], rtol=1e-9, atol=1e-12)
        assert np.allclose(ref["var"][j], vars_[j], rtol=1e-8, atol=1e-12)
        f_ref = np.array(sorted(map(tuple, ref["fronts"][j])))
        f_new = np.array(sorted(map(tuple, fronts[j])))
        assert f_ref.shape == f_new.shape and np.allclose(f_ref, f_new, rtol=1e-10, atol=1e-12)
    if noise is not None:
        assert repick, "the case must exercise the exclusion of picked candidates"


def test_fantasy_picks_on_a_subset_equal_the_whole_pool():
    """Forced replay evaluated at a subset of the pool gives, at those
    candidates, the values of the whole-pool run (the refits and fronts do
    not depend on which candidates are evaluated)."""
    inst = make_instance("tiny", seeds("tiny")[0], n_cand=200)
    feas = Stream(5, "feas").uniform(inst.n_cand) < 0.9
    full = O.fantasy_picks(inst, 4, feas)
    sub = np.sort(Stream(6, "sub").u64(40) % np.uint64(inst.n_cand)).astype(np.int64)
    part = O.fantasy_picks(inst, 4, feas, forced=full["picks"], subset=sub)
    assert part["picks"] == full["picks"]
    assert set(full["picks"]) <= set(part["index"].tolist())
    for j in range(4):
        assert np.allclose(part["acq"][j], full["acq"][j][part["index"]], rtol=1e-12, atol=1e-15)
        assert np.allclose(part["var"][j], full["var"][j][part["index"]], rtol=1e-12, atol=1e-15)


def _hand_instance(targets, q_noise=1e-8):
    """One observation x = 0 with y = (1, -1), one continuous parameter in
    [0, 1], both objectives with lengthscale 0.25, s_f^2 = 1, tau^2 = 1e-8;
    candidate i sits where the Matern-5/2 covariance with the observation is
    targets[i], so its posterior mean is (k_i, -k_i) / (1 + tau^2)."""
    from types import SimpleNamespace
    from scipy.optimize import brentq
    from workloads.generate import PARAM_DTYPE
    space = np.zeros(1, PARAM_DTYPE)
    space[0] = (3, 0, 0.0, 1.0)
    ell = 0.25
    xs = [brentq(lambda x: float(O.matern(x / ell, 1.0)) - t, 0.0, 1.0, xtol=1e-15) for t in targets]
    n = len(xs)
    cand = np.zeros((1, (n + 3) // 4 * 4), np.uint32)
    cand[0, :n] = np.array(xs, np.float32).view(np.uint32)
    k = np.array([float(O.matern(np.float32(x) / ell, 1.0)) for x in xs])
    inst = SimpleNamespace(n_cand=n, cand=cand, space=space, x_obs=np.zeros((1, 1), np.uint32),
                           y_obs=np.array([[1.0], [-1.0]], np.float32), lengthscale=np.full((2, 1), ell, np.float32),
                           signal_var=np.ones(2, np.float32), noise_var=np.full(2, q_noise, np.float32), n_obj=2,
                           eps=np.zeros((1, 2), np.float32), ref=np.array([-1.0, -1.5], np.float32))
    return inst, k


def test_fantasy_picks_hand_worked_one_observation():
    """n = 1, M = 2, a single base sample eps = 0 (EHVI = HVI at the mean),
    r = (-1, -1.5), candidates with k = 0.5, 0.2, 0.8, 0.25 (means (k, -k)).
    Worked by hand from the rectangles of Section 4.4:
      step 1: HVI = (k + 1)(1 - k) = 0.75, 0.96, 0.36, 0.9375 -> index 1;
      step 2 (front + (0.2, -0.2)): k = 0.5 keeps (0.5 - 0.2) x (1 - 0.5)
              = 0.15, k = 0.8 keeps 0.6 x 0.2 = 0.12, k = 0.25 keeps
              0.05 x 0.75 = 0.0375 -> index 0 (a loop that kept the front
              unchanged would take k = 0.25, index 3, the second-best value
              of step 1);
      step 3 (front + (0.5, -0.5)): k = 0.8 keeps 0.3 x 0.2 = 0.06, k = 0.25
              keeps 0.05 x 0.25 = 0.0125 -> index 2;
      step 4: index 3 with 0.0125;
    and with q = 5 the loop stops after 4 picks (the candidates run out)."""
    inst, k = _hand_instance([0.5, 0.2, 0.8, 0.25])
    feas = np.ones(4, bool)
    r2 = O.fantasy_picks(inst, 2, feas)
    assert r2["picks"] == [1, 0]
    assert np.allclose(r2["acq"][0], [0.75, 0.96, 0.36, 0.9375], atol=2e-6)
    assert np.allclose(r2["acq"][1][[0, 2, 3]], [0.15, 0.12, 0.0375], atol=2e-6)
    assert r2["acq"][1][1] == -np.inf
    r5 = O.fantasy_picks(inst, 5, feas)
    assert r5["picks"] == [1, 0, 2, 3]
    assert r5["acq"][2][2] == pytest.approx(0.06, abs=2e-6)
    assert r5["acq"][2][3] == pytest.approx(0.0125, abs=2e-6)
    assert r5["acq"][3][3] == pytest.approx(0.0125, abs=2e-6)
    # the fronts: the observation, then each fantasised mean (k, -k)
    assert len(r5["fronts"][3]) == 4
    assert np.allclose(sorted(r5["fronts"][3][:, 0]), sorted([1.0, k[1], k[0], k[2]]), atol=1e-7)


# ------------------------------------------------------------------ MACE (Sections 4.5 and 4.7)

def test_pi_closed_form_matches_quadrature():
    """PI = P(f + xi > y+) is the Gaussian density integrated above y+ - xi."""
    xi = 1e-4
    for mu, sd, yb in [(0.0, 1.0, 0.0), (-1.3, 0.2, 0.5), (2.0, 0.5, 1.0), (0.3, 3.0, 2.0), (-4, 0.7, 0.0)]:
        pdf = lambda y: math.exp(-0.5 * ((y - mu) / sd) ** 2) / (sd * math.sqrt(2 * math.pi))
        lo = yb - xi
        q, _ = integrate.quad(pdf, lo, mu + 14 * sd, epsabs=1e-14, epsrel=1e-12, limit=200) if lo < mu + 14 * sd else (0.0, 0)
        assert O.probability_of_improvement(mu, sd * sd, yb, xi) == pytest.approx(q, rel=1e-9, abs=1e-13)


def test_pi_is_the_mean_derivative_of_ei():
    """d EI / d mu = Phi(z) = PI: ties the two closed forms to each other."""
    h = 1e-6
    for mu, var, yb in [(0.1, 0.3, 0.4), (-2.0, 1.5, 0.0), (1.2, 0.01, 1.0)]:
        d = (O.expected_improvement(mu + h, var, yb) - O.expected_improvement(mu - h, var, yb)) / (2 * h)
        assert float(d) == pytest.approx(float(O.probability_of_improvement(mu, var, yb)), abs=1e-8)


def test_pi_and_ucb_limits():
    # sigma = 0: a certain event exactly when mu + xi > y+ (strict)
    assert np.array_equal(O.probability_of_improvement(np.array([0.5, 1.0, 1.5]), 0.0, 1.0, 0.0), [0.0, 0.0, 1.0])
    assert np.allclose(O.upper_confidence_bound(np.array([0.5, -2.0]), 0.0, 7.0), [0.5, -2.0])
    # mu + kappa sigma is the Phi(kappa) quantile of N(mu, sigma^2) (library quantile)
    from scipy.stats import norm
    for mu, sd, kappa in [(0.3, 0.2, 1.5), (-1.0, 2.0, 0.5), (2.0, 0.1, 3.0)]:
        want = norm.ppf(norm.cdf(kappa), loc=mu, scale=sd)
        assert O.upper_confidence_bound(mu, sd * sd, kappa) == pytest.approx(want, rel=1e-9)
    mus = np.linspace(-3, 3, 40)
    assert np.all(np.diff(O.probability_of_improvement(mus, 0.3, 0.0)) > 0)
    A = O.mace_acquisitions(np.array([0.1]), np.array([0.04]), 0.2, 1e-4, 2.0)
    assert A.shape == (3, 1) and A[0, 0] == pytest.approx(0.5)


def _front_2d_sweep(P):
    """Textbook 2-D maxima: sort by x descending (y descending on ties) and
    keep a point when its y is at least the best y seen among points with a
    strictly larger x, and it equals the previous kept point or beats every
    y seen so far."""
    order = sorted(range(len(P)), key=lambda i: (-P[i][0], -P[i][1]))
    keep, best_y, prev = [], -math.inf, None
    for i in order:
        x, y = P[i]
        if y > best_y or (prev is not None and (x, y) == prev):
            keep.append(i)
            prev = (x, y)
        best_y = max(best_y, y)
    return sorted(keep)


def test_nondominated_matches_2d_sweep():
    st = Stream(41, "front2d")
    for trial in range(20):
        n = 1 + trial * 7
        P = np.floor(st.uniform(2 * n).reshape(n, 2) * (3 + trial)).tolist()
        got = np.nonzero(O.nondominated(np.array(P)))[0].tolist()
        assert got == _front_2d_sweep([tuple(p) for p in P])


@pytest.mark.parametrize("M", [3, 4])
def test_nondominated_is_the_maxima_set(M):
    """The unique set that is mutually non-dominating and dominates every
    other point; permutation-invariant; unchanged by a dominated point;
    duplicates of front points all kept."""
    st = Stream(42 + M, "frontMd")
    dom = lambda a, b: all(x >= y for x, y in zip(a, b)) and any(x > y for x, y in zip(a, b))
    for trial in range(12):
        n = 5 + 9 * trial
        Y = np.floor(st.uniform(M * n).reshape(n, M) * 4)
        f = O.nondominated(Y)
        F = [tuple(Y[i]) for i in np.nonzero(f)[0]]
        assert f.any()
        for i in range(n):
            dominated = any(dom(tuple(Y[j]), tuple(Y[i])) for j in range(n))
            assert f[i] == (not dominated)
            if not f[i]:
                assert any(dom(p, tuple(Y[i])) for p in F)
        perm = np.argsort(st.uniform(n))
        assert np.array_equal(O.nondominated(Y[perm]), f[perm])
        worst = Y.min(axis=0) - 1
        assert np.array_equal(O.nondominated(np.vstack([Y, worst]))[:n], f)
        i0 = int(np.nonzero(f)[0][0])
        f2 = O.nondominated(np.vstack([Y, Y[i0]]))
        assert f2[-1] and np.array_equal(f2[:n], f)


def test_splitmix64_published_outputs(golden_dir):
    lines = [l for l in open(os.path.join(golden_dir, "splitmix64_seed0.txt")) if not l.startswith("#")]
    assert lines[0].split() == ["seed", "0"]
    want = [int(l, 16) for l in lines[1:]]
    assert [O.splitmix64(0, i) for i in range(len(want))] == want


def test_mace_select_draws_from_the_front():
    st = Stream(44, "mace")
    n = 400
    A = np.floor(st.uniform(3 * n).reshape(3, n) * 6)
    mask = st.uniform(n) < 0.8
    A[0, 5] = np.nan
    A[1, 6] = -np.inf
    picks, front, cnt = O.mace_select(A, mask, 4, seed=7)
    ok = mask.copy()
    ok[[5, 6]] = False
    idx = np.nonzero(ok)[0]
    assert np.array_equal(front, idx[O.nondominated(A[:, idx].T)])
    assert cnt == min(4, len(front)) and set(picks) <= set(front) and len(set(picks)) == cnt
    keys = [O.splitmix64(7, int(i)) for i in picks]
    assert keys == sorted(keys)
    assert all(O.splitmix64(7, int(i)) > keys[-1] for i in set(front) - set(picks))
    # a front smaller than k comes back whole; nothing eligible gives nothing
    p2, f2, c2 = O.mace_select(A, mask, len(front) + 3, seed=1)
    assert c2 == len(front) and sorted(p2) == sorted(front)
    p3, f3, c3 = O.mace_select(A, np.zeros(n, bool), 4, seed=1)
    assert c3 == 0 and len(p3) == 0 and len(f3) == 0
    # over many seeds every front member is drawn about k / F of the time
    F = len(front)
    counts = np.zeros(n)
    for s in range(2000):
        counts[O.mace_select(A, mask, 2, seed=s)[0]] += 1
    freq = counts[front] / 2000
    assert np.all(np.abs(freq - 2 / F) < 5 * math.sqrt((2 / F) * (1 - 2 / F) / 2000) + 1e-9)


# ------------------------------------------------------------------ input warping (Section 4.3)

def test_kumaraswamy_cdf_is_the_integral_of_its_density():
    for a, b in [(0.5, 2.0), (1.7, 0.6), (3.0, 3.0), (1.0, 1.0)]:
        pdf = lambda x: a * b * x ** (a - 1) * (1 - x ** a) ** (b - 1)
        for u in (0.05, 0.3, 0.77, 0.999):
            q, _ = integrate.quad(pdf, 0.0, u, epsabs=1e-13, epsrel=1e-11, limit=200)
            assert float(O.kumaraswamy_cdf(u, a, b)) == pytest.approx(q, rel=1e-8, abs=1e-12)
    u = np.linspace(0, 1, 101)
    assert np.allclose(O.kumaraswamy_cdf(u, 1.0, 1.0), u, atol=1e-15)
    w = O.kumaraswamy_cdf(u, 2.3, 0.4)
    assert w[0] == 0.0 and w[-1] == 1.0 and np.all(np.diff(w) > 0)


def test_warped_gp_is_the_plain_gp_on_warped_features():
    """The warp acts once on both the observations and the candidates."""
    sp, X, y, gp = _toy_gp(20, noise=1e-3)
    st = Stream(81, "warp")
    warp = np.exp(st.normal(2 * len(sp)).reshape(len(sp), 2) * 0.4)
    Xw = X.view(np.uint32)
    gw = O.GP(sp, Xw, y, gp.lengthscale, gp.signal_var, gp.noise_var, gp.kernel, warp=warp)
    C = st.uniform(3 * 200).reshape(3, 200).astype(np.float32).view(np.uint32)
    u, cat = O.gp_features(sp, O.decode(sp, C))
    plain = O.GP(sp, Xw, y, gp.lengthscale, gp.signal_var, gp.noise_var, gp.kernel)
    plain.u_obs = gw.warped(plain.u_obs)
    plain._factor()
    m1, v1 = gw.posterior_u(u)
    m2, v2 = plain.posterior_u(gw.warped(u))
    assert np.allclose(m1, m2, rtol=1e-12, atol=1e-13) and np.allclose(v1, v2, rtol=1e-12, atol=1e-13)
    # one observation, one ordinal dimension: the closed form on warped coordinates
    sp1 = sp[:1]
    x1 = np.ascontiguousarray(Xw[:1, :1])
    g1 = O.GP(sp1, x1, y[:1], gp.lengthscale[:1], 1.0, 0.1, O.MATERN52, warp=warp[:1])
    c1 = np.ascontiguousarray(C[:1, :5])
    uc, _ = O.gp_features(sp1, O.decode(sp1, c1))
    uo, _ = O.gp_features(sp1, O.decode(sp1, x1))
    a_, b_ = warp[0]
    wc = 1 - (1 - uc[:, 0] ** a_) ** b_
    wo = 1 - (1 - uo[0, 0] ** a_) ** b_
    r = np.abs(wc - wo) / gp.lengthscale[0]
    k = (1 + math.sqrt(5) * r + 5 * r * r / 3) * np.exp(-math.sqrt(5) * r)
    mu, var = g1.posterior_u(uc)
    assert np.allclose(mu, k * y[0] / 1.1, rtol=1e-12) and np.allclose(var, 1 - k * k / 1.1, rtol=1e-10, atol=1e-14)


# ------------------------------------------------------------------ Sobol sampling and the Delta controller (Algorithm 1)

def _totient(m):
    r, p, x = m, 2, m
    while p * p <= x:
        if x % p == 0:
            while x % p == 0:
                x //= p
            r -= r // p
        p += 1
    if x > 1:
        r -= r // x
    return r


def test_primitive_polynomials_count_and_period():
    """There are phi(2^s - 1) / s primitive polynomials of degree s; each
    drives a shift register through all 2^s - 1 nonzero states."""
    polys = O.primitive_polynomials(1 + 1 + 2 + 2 + 6 + 6 + 18)
    by_degree = {}
    for s, a in polys:
        by_degree.setdefault(s, []).append(a)
    for s in range(1, 8):
        assert len(by_degree.get(s, [])) == _totient((1 << s) - 1) // s, s
    for s, a in polys:
        taps = [(a >> (s - 1 - i)) & 1 for i in range(1, s)]  # a_1 .. a_(s-1)
        state = [0] * (s - 1) + [1]
        seen = set()
        for _ in range((1 << s) - 1):
            seen.add(tuple(state))
            # x^s = a_1 x^(s-1) + ... + a_(s-1) x + 1 over GF(2): the linear recurrence of the register
            new = state[0]
            for i, t in enumerate(taps):
                new ^= t & state[s - 1 - i]
            state = state[1:] + [new]
        assert len(seen) == (1 << s) - 1, (s, a)


def test_sobol_first_dimension_is_van_der_corput():
    X = O.sobol_integers(1, 300, skip=17)
    for r in range(300):
        i = 17 + r
        rev = int(format(i, "032b")[::-1], 2)
        assert int(X[r, 0]) == rev


@pytest.mark.parametrize("m", [1, 3, 6, 8])
def test_sobol_net_properties(m):
    """Each dimension alone is a (0, 1)-sequence, and the first two
    dimensions a (0, 2)-sequence: the first 2^m points fill every
    elementary box of volume 2^-m exactly once."""
    n = 1 << m
    X = O.sobol_integers(6, n).astype(object)
    for j in range(6):
        assert sorted(int(x) >> (32 - m) for x in X[:, j]) == list(range(n))
    for a in range(m + 1):
        b = m - a
        cells = {(int(x0) >> (32 - a), int(x1) >> (32 - b)) for x0, x1 in X[:, :2]}
        assert len(cells) == n, (m, a)


def test_sobol_skip_and_configs():
    full = O.sobol_integers(4, 96)
    assert np.array_equal(O.sobol_integers(4, 40, skip=56), full[56:])
    sp = _space((INT_LOG, 0, 1, 1024), (INT_UNIFORM, 0, 3, 9), (CATEGORICAL, 4, 0, 0), (CONTINUOUS, 0, 0.5, 0.95))
    w = O.sobol_configs(sp, 64)
    v = w.view(np.int32)
    assert v[0].min() >= 1 and v[0].max() <= 1024
    assert np.array_equal(np.bincount(v[1] - 3, minlength=7)[:7] > 0, np.ones(7, bool))
    assert v[2, :4].tolist() == [0, 2, 1, 3]     # floor(4 u) of the third dimension: 0, .5, .25, .75
    f = w[3].view(np.float32)
    assert f.min() >= 0.5 and f.max() < 0.95


def test_sobol_configs_mapping_values():
    """The mappings of the shortfall fill (Section 4.6) at the first eight
    points of the first dimension (the van der Corput points k / 8, pinned
    above), worked by hand: integer log-uniform on [1, 1024] is 1024^u =
    2^(10 u) rounded (2^1.25 = 2.38, 2^2.5 = 5.66, 2^3.75 = 13.45, 2^6.25 =
    76.1, 2^7.5 = 181.02, 2^8.75 = 430.5 + 0.04); integer uniform on [3, 9]
    is 3 + floor(7 u); a categorical of 5 choices floor(5 u); continuous on
    [0.5, 0.95] is 0.5 + 0.45 u."""
    u = [0.0, 0.5, 0.25, 0.75, 0.125, 0.625, 0.375, 0.875]  # points 0 .. 7
    log_at = {0.0: 1, 0.125: 2, 0.25: 6, 0.375: 13, 0.5: 32, 0.625: 76, 0.75: 181, 0.875: 431}
    uni_at = {0.0: 3, 0.125: 3, 0.25: 4, 0.375: 5, 0.5: 6, 0.625: 7, 0.75: 8, 0.875: 9}
    cat_at = {0.0: 0, 0.125: 0, 0.25: 1, 0.375: 1, 0.5: 2, 0.625: 3, 0.75: 3, 0.875: 4}
    for kind, lo, hi, want in ((INT_LOG, 1, 1024, log_at), (INT_UNIFORM, 3, 9, uni_at)):
        w = O.sobol_configs(_space((kind, 0, lo, hi)), 8).view(np.int32)[0]
        assert w.tolist() == [want[x] for x in u], kind
    w = O.sobol_configs(_space((CATEGORICAL, 5, 0, 0)), 8).view(np.int32)[0]
    assert w.tolist() == [cat_at[x] for x in u]
    f = O.sobol_configs(_space((CONTINUOUS, 0, 0.5, 0.95)), 8).view(np.float32)[0]
    assert f.tolist() == [float(np.float32(0.5 + 0.45 * x)) for x in u]


def test_delta_controller_trajectory():
    """Worked by hand from Algorithm 1 with k = 2 and step 0.05."""
    d, c = 0.5, 0
    steps = []
    for invalid in (False, False, False, True, False, False, False, False, False):
        d, c = O.delta_update(d, c, 2, invalid)
        steps.append((round(d, 10), c))
    assert steps == [(0.5, 2), (0.5, 4), (0.45, 1), (0.5, 0), (0.5, 2), (0.5, 4), (0.45, 1), (0.45, 3), (0.4, 0)]
    # bounds: never above 0.75 after invalid results, never below 0.25
    d, c = 0.72, 0
    d, c = O.delta_update(d, c, 1, True)
    assert d == 0.75
    d = 0.26
    for _ in range(10):
        d, c = O.delta_update(d, c, 5, False)
    assert d == 0.25


# ------------------------------------------------------------------ forest training (Algorithm 1, Section 4.6)

def test_cart_hand_worked(golden_dir):
    lines = [l.split() for l in open(os.path.join(golden_dir, "cart_hand.txt")) if not l.startswith("#")]
    s = [float(v) for v in lines[0][1:]]
    X = np.array([s[i:i + 2] for i in range(0, len(s), 3)], np.float32)
    y = np.array(s[2::3], np.int64)
    want = [(float(a), int(b), int(c), bool(int(d))) for _, a, b, c, d in lines[1:]]
    assert O.train_cart(X, y, np.arange(len(y)), 4, 255) == want


def _split_sse_brute(X, y, samp, f, v):
    left = [i for i in samp if X[i, f] <= v]
    right = [i for i in samp if X[i, f] > v]
    sse = lambda g: sum((y[i] - np.mean([y[j] for j in g])) ** 2 for i in g) if g else 0.0
    return sse(left) + sse(right)


def test_cart_splits_are_optimal_and_leaves_round():
    """Every split minimises the summed squared error over all splits of its
    node's samples (brute force with floating means); leaves hold
    round(V p / m); the tree ignores the order of the bootstrap list; grown
    to purity without bootstrap it reproduces its labels."""
    st = Stream(91, "cart")
    n, d = 60, 4
    X = np.floor(st.uniform(n * d).reshape(n, d) * 7).astype(np.float32)
    y = (st.uniform(n) < 0.4).astype(np.int64)
    boot = st.integers(0, n - 1, n)
    tree = O.train_cart(X, y, boot, 5, 255)
    # walk the tree again, node by node, to recover each node's samples
    node_samples = {0: list(boot)}
    for k, (val, left, f, leaf) in enumerate(tree):
        samp = node_samples[k]
        if leaf:
            p, m = sum(y[i] for i in samp), len(samp)
            assert val == math.floor(255 * p / m + 0.5)
            continue
        got = _split_sse_brute(X, y, samp, f, val)
        for g in range(d):
            for v in sorted(set(X[samp, g]))[:-1]:
                assert got <= _split_sse_brute(X, y, samp, g, v) + 1e-9
        node_samples[left] = [i for i in samp if X[i, f] <= val]
        node_samples[left + 1] = [i for i in samp if X[i, f] > val]
    assert O.train_cart(X, y, boot[::-1], 5, 255) == tree
    Xp = (X + np.arange(n, dtype=np.float32)[:, None] * np.float32(0.001)).astype(np.float32)
    full = O.train_cart(Xp, y, np.arange(n), 64, 1)
    for i in range(n):
        k = 0
        while not full[k][3]:
            k = full[k][1] + (0 if Xp[i, full[k][2]] <= full[k][0] else 1)
        assert full[k][0] == y[i]


def test_cart_signed_zero_is_one_value():
    """-0 and +0 are one feature value (x <= v cannot separate them): they
    form one candidate and the threshold is stored as +0, whichever of the
    two the samples carry; the split matches the one with +0 everywhere."""
    X = np.array([[-1.0], [-0.0], [0.0], [-0.0], [2.0]], np.float32)
    y = np.array([0, 0, 1, 1, 1])
    tree = O.train_cart(X, y, np.arange(5), 4, 255)
    Xp = X + np.float32(0.0)  # -0 + 0 = +0; the other values unchanged
    assert np.signbit(X).sum() == 3 and np.signbit(Xp).sum() == 1
    assert tree == O.train_cart(Xp, y, np.arange(5), 4, 255)
    zeros = [t for t in tree if not t[3] and t[0] == 0.0]
    assert zeros and all(math.copysign(1.0, t[0]) == 1.0 for t in zeros)


# ------------------------------------------------------------------ GP hyperparameters by MLE (Section 4.3)

def _mle_case(name="d8-ehvi2", n=24, m=0):
    inst = make_instance(name, seeds(name)[0], n_cand=16)
    x = np.ascontiguousarray(inst.x_obs[:, :n])
    y = np.asarray(inst.y_obs[m, :n], np.float64)
    theta = np.concatenate([np.log(inst.lengthscale[m].astype(np.float64)),
                            [math.log(float(inst.signal_var[m])), math.log(max(float(inst.noise_var[m]), 1e-3))]])
    return inst, x, y, theta


@pytest.mark.parametrize("kernel", [0, 1])
def test_lml_equals_gaussian_log_density(kernel):
    """The log marginal likelihood is the log density of y under
    N(0, K + tau^2 I): scipy's multivariate normal, with K from the
    (separately pinned) GP covariance."""
    from scipy.stats import multivariate_normal
    inst, x, y, theta = _mle_case()
    d = inst.d
    lml, _ = O.log_marginal_likelihood(inst.space, x, y, theta, kernel)
    gp = O.GP(inst.space, x, y, np.exp(theta[:d]), math.exp(theta[d]), math.exp(theta[d + 1]), kernel)
    K = gp.cov(gp.u_obs, gp.u_obs) + math.exp(theta[d + 1]) * np.eye(len(y))
    want = multivariate_normal(mean=np.zeros(len(y)), cov=K).logpdf(y)
    assert lml == pytest.approx(want, rel=1e-10, abs=1e-9)


@pytest.mark.parametrize("kernel,name", [(0, "d8-ehvi2"), (1, "d8-ehvi2"), (0, "d10-ei")])
def test_lml_gradient_matches_finite_differences(kernel, name):
    """Every component of the analytic gradient (ordinal and categorical
    lengthscales, signal and noise variance) equals a central difference of
    the log marginal likelihood."""
    inst, x, y, theta = _mle_case(name, n=20)
    _, g = O.log_marginal_likelihood(inst.space, x, y, theta, kernel)
    h = 1e-5
    for p in range(len(theta)):
        tp, tm = theta.copy(), theta.copy()
        tp[p] += h
        tm[p] -= h
        fd = (O.log_marginal_likelihood(inst.space, x, y, tp, kernel)[0] -
              O.log_marginal_likelihood(inst.space, x, y, tm, kernel)[0]) / (2 * h)
        assert g[p] == pytest.approx(fd, rel=1e-5, abs=1e-6), p


def test_lml_one_observation_closed_form_and_noise_mle():
    """n = 1: lml = -y^2 / (2 v) - log(v) / 2 - log(2 pi) / 2 with
    v = s_f^2 + tau^2, d lml / d ln tau^2 = tau^2 (y^2 / v^2 - 1 / v) / 2;
    fitting tau^2 alone reaches v = y^2, the closed-form maximiser."""
    space = np.zeros(2, PARAM_DTYPE)
    space["kind"] = CONTINUOUS
    space["hi"] = 1.0
    x = np.array([[np.float32(0.3).view(np.uint32)], [np.float32(0.7).view(np.uint32)]], np.uint32)
    y = np.array([2.5])
    sf2, tau2 = 1.0, 0.5
    theta = np.array([0.0, 0.0, math.log(sf2), math.log(tau2)])
    lml, g = O.log_marginal_likelihood(space, x, y, theta)
    v = sf2 + tau2
    assert lml == pytest.approx(-y[0] ** 2 / (2 * v) - 0.5 * math.log(v) - 0.5 * math.log(2 * math.pi), rel=1e-14)
    assert g[3] == pytest.approx(0.5 * tau2 * (y[0] ** 2 / v ** 2 - 1 / v), rel=1e-12)
    assert g[2] == pytest.approx(0.5 * sf2 * (y[0] ** 2 / v ** 2 - 1 / v), rel=1e-12)
    assert g[0] == 0.0 and g[1] == 0.0
    free = np.array([0, 0, 0, 1])
    th, best = O.fit_hyperparameters(space, x, y, theta, [-9] * 4, [9] * 4, free, 400, 0.1)
    assert math.exp(th[3]) == pytest.approx(y[0] ** 2 - sf2, rel=1e-4)
    assert np.array_equal(th[:3], theta[:3])


def test_fit_increases_lml_and_respects_bounds():
    """The fit ends with a larger likelihood than its start, inside the
    bounds, with frozen parameters untouched and the free ones at a
    stationary point or a bound."""
    inst, x, y, theta = _mle_case(n=30)
    P = len(theta)
    lo = np.full(P, -4.0)
    hi = np.full(P, 3.0)
    lo[-1] = math.log(1e-4)
    free = np.ones(P, int)
    free[0] = 0
    start = np.clip(theta + 0.5, lo, hi)
    l0, _ = O.log_marginal_likelihood(inst.space, x, y, start)
    th, l1 = O.fit_hyperparameters(inst.space, x, y, start, lo, hi, free, 1000, 0.05)
    assert l1 > l0 + 10.0
    assert np.all(th >= lo) and np.all(th <= hi) and th[0] == start[0]
    _, g = O.log_marginal_likelihood(inst.space, x, y, th)
    inside = (th > lo + 1e-9) & (th < hi - 1e-9) & (free == 1)
    at_bound = (free == 1) & ~inside
    assert inside.sum() >= 7 and np.all(np.abs(g[inside]) < 1e-6)
    # at a bound the gradient points outwards (the bound holds the maximiser back)
    assert np.all(np.where(th[at_bound] <= lo[at_bound] + 1e-9, g[at_bound] <= 0, g[at_bound] >= 0))
