"""Plain fp64 CPU oracle of the candidate-scoring path of SCOOT.

TEST INFRASTRUCTURE ONLY.  Only the tests, the smoke check and the
benchmark's CPU-baseline leg may import this module.  It shares no code
with the CUDA path: it takes the same seeded inputs (raw configuration words,
observed values, hyperparameters, forest nodes, base samples) and computes
every step on its own, slowly and directly, in float64.

Steps, in the order of one suggestion round (Section 4, Algorithm 1):

1. known-constraint pruning, Eq. (2) and the appendix on known constraints;
2. random-forest probability of feasibility, Eq. (3) (Section 4.6);
3. GP posterior mean and variance, the two equations of Section 4.3;
4. acquisition: EI, Eq. (6), or Monte-Carlo EHVI, Eq. (7), with the
   hypervolume of Section 4.4 (Fig. 4), or the exact EHVI expectation over
   independent Gaussian objectives;
5. top-q selection for parallel suggestion (Section 4.7);
6. sequential picks with kriging-believer fantasies (not in the paper; the
   refit form is used here: each pick is appended to the observations with
   its posterior mean as value and the GP is conditioned again);
7. MACE for single-objective suggestion (Sections 4.5 and 4.7): UCB, PI and
   EI on the same posterior, their Pareto front, and a random k-subset of it.
8. the tuning loop's Sobol sampling and Algorithm 1's threshold controller;
9. CART training of the feasibility forest (Algorithm 1, Section 4.6);
10. GP hyperparameters by maximum likelihood (Section 4.3).

Readings of points the paper leaves open are marked "Reading:".
Every function is pinned by the not-gpu tests against closed forms,
invariants, brute force or library routines; nothing here is "parity
unpinned".
"""
from __future__ import annotations

import math

import numpy as np
import scipy.linalg as sla
from scipy.special import erfc

INT_UNIFORM, INT_LOG, CATEGORICAL, CONTINUOUS = 0, 1, 2, 3
MATERN52, MATERN32 = 0, 1
NODE_LEAF = 1


# --------------------------------------------------------------------------
# decoding

def decode(space, words: np.ndarray, n: int | None = None) -> np.ndarray:
    """Stored values of candidates as float64 [n][d].

    Integers and category indices are int32 words; continuous values are
    float32 bit patterns (Section 3's mixed space of int / enum / float /
    bool parameters).
    """
    n = words.shape[1] if n is None else n
    cols = []
    for i in range(len(space)):
        w = np.ascontiguousarray(words[i, :n])
        if int(space[i]["kind"]) == CONTINUOUS:
            cols.append(w.view(np.float32).astype(np.float64))
        else:
            cols.append(w.view(np.int32).astype(np.float64))
    return np.stack(cols, axis=1) if cols else np.zeros((n, 0))


# --------------------------------------------------------------------------
# 1. known constraints, Eq. (2)

def prune_mask(space, clauses, words: np.ndarray, n: int) -> np.ndarray:
    """mask[i] = every clause c of C holds for candidate i (Eq. 2).

    Reading: a clause is "all guards hold => sum_t coef_t x[param_t] >= rhs",
    evaluated in exact integer arithmetic; the inclusive ">=" follows the
    appendix ("greater than or equal to").  The example constraint of
    Section 3 ("x[1] < x[3] if x[4] is False") is a clause with one guard.
    """
    x = decode(space, words, n)
    mask = np.ones(n, dtype=bool)
    for c in clauses:
        guard = np.ones(n, dtype=bool)
        for g in range(int(c["n_guard"])):
            p = int(c["guard_param"][g])
            guard &= x[:, p].astype(np.int64) == int(c["guard_value"][g])
        nt = int(c["n_term"])
        coefs = [int(c["coef"][t]) for t in range(nt)]
        if all(abs(k) < 2 ** 29 for k in coefs) and abs(int(c["rhs"])) < 2 ** 62:
            # every term is below 2^60 in magnitude (values are 32-bit), so
            # the int64 sum of at most four terms is exact
            lhs = np.zeros(n, dtype=np.int64)
            for t in range(nt):
                lhs += coefs[t] * x[:, int(c["term_param"][t])].astype(np.int64)
            holds = lhs >= int(c["rhs"])
        else:
            lhs = np.zeros(n, dtype=object)
            for t in range(nt):
                lhs = lhs + coefs[t] * x[:, int(c["term_param"][t])].astype(np.int64).astype(object)
            holds = np.array([int(v) >= int(c["rhs"]) for v in lhs], dtype=bool) if n else np.zeros(0, bool)
        mask &= (~guard) | holds
    return mask


# --------------------------------------------------------------------------
# 2. random-forest probability of feasibility, Eq. (3)

def tree_walk(nodes: np.ndarray, base: int, x: np.ndarray) -> float:
    """Leaf value of the regression tree whose root is nodes[base], for one
    configuration x, by recursion from the root.

    Reading: an internal node sends x to its left child when x[feat] <= thr;
    the right child sits right after the left one; child indices are
    relative to the tree's root.
    """
    return _walk_from(nodes, base, 0, x)


def _walk_from(nodes, tree_base, idx, x):
    nd = nodes[tree_base + idx]
    if int(nd["flags"]) & NODE_LEAF:
        return float(nd["val"])
    left = int(nd["left"])
    return _walk_from(nodes, tree_base, left if x[int(nd["feat"])] <= float(nd["val"]) else left + 1, x)


def rf_votes_one(nodes, tree_offset, x: np.ndarray) -> int:
    """Sum over trees of the integer leaf votes for one configuration."""
    total = 0
    for t in range(len(tree_offset) - 1):
        total += int(_walk_from(nodes, int(tree_offset[t]), 0, x))
    return total


def rf_votes(nodes, tree_offset, space, words, n: int) -> np.ndarray:
    """Votes for all n candidates: the same tree walk, vectorised over candidates."""
    x = decode(space, words, n)
    votes = np.zeros(n, dtype=np.int64)
    for t in range(len(tree_offset) - 1):
        base = int(tree_offset[t])
        size = int(tree_offset[t + 1]) - base
        tree = nodes[base:base + size]
        idx = np.zeros(n, dtype=np.int64)
        active = np.arange(n)          # candidates not yet at a leaf
        for _ in range(size + 1):
            node = idx[active]
            leaf = (tree["flags"][node] & NODE_LEAF) != 0
            active, node = active[~leaf], node[~leaf]
            if len(active) == 0:
                break
            xv = x[active, tree["feat"][node].astype(np.int64)]
            left = tree["left"][node].astype(np.int64)
            idx[active] = np.where(xv <= tree["val"][node].astype(np.float64), left, left + 1)
        votes += tree["val"][idx].astype(np.float64).astype(np.int64)
    return votes


def pof_feasible(votes, n_trees: int, leaf_scale: int, delta_num: int, delta_den: int):
    """POF(x) >= Delta (Eq. 3) with POF = votes / (leaf_scale * T), Delta = num / den.

    Reading: the forest regresses a 0/1 feasibility label; each leaf stores
    round(leaf_scale * mean label) so POF is an exact rational and the
    test is the exact integer comparison den * votes >= num * scale * T.
    """
    v = np.asarray(votes, dtype=object)
    lhs = v * int(delta_den)
    rhs = int(delta_num) * int(leaf_scale) * int(n_trees)
    return np.array([int(a) >= rhs for a in lhs], dtype=bool)


# --------------------------------------------------------------------------
# 3. GP posterior (Section 4.3)

def gp_features(space, x: np.ndarray):
    """Coordinates on which the covariance acts.

    Reading (the paper does not say): integer log-uniform parameters on a log
    scale, (ln v - ln lo) / (ln hi - ln lo); integer uniform and continuous
    ones linearly, (v - lo) / (hi - lo); categoricals by their index, compared
    for equality only.
    """
    u = np.array(x, dtype=np.float64, copy=True)
    is_cat = np.zeros(len(space), dtype=bool)
    for i in range(len(space)):
        kind = int(space[i]["kind"])
        lo, hi = float(space[i]["lo"]), float(space[i]["hi"])
        if kind == INT_LOG:
            u[:, i] = (np.log(x[:, i]) - math.log(lo)) / (math.log(hi) - math.log(lo))
        elif kind in (INT_UNIFORM, CONTINUOUS):
            u[:, i] = (x[:, i] - lo) / (hi - lo) if hi > lo else 0.0
        else:
            is_cat[i] = True
    return u, is_cat


def scaled_distance(ua, ub, is_cat, lengthscale) -> np.ndarray:
    """r[a, b] with r^2 = sum_c ((ua_c - ub_c) / l_c)^2 over ordinal dims plus
    sum_c [ua_c != ub_c] / l_c^2 over categorical dims (ARD lengthscales)."""
    r2 = np.zeros((ua.shape[0], ub.shape[0]))
    for c in range(ua.shape[1]):
        ell = float(lengthscale[c])
        if is_cat[c]:
            r2 += (ua[:, c][:, None] != ub[:, c][None, :]).astype(np.float64) / (ell * ell)
        else:
            diff = (ua[:, c][:, None] - ub[:, c][None, :]) / ell
            r2 += diff * diff
    return np.sqrt(r2)


def matern(r, signal_var: float, kernel: int = MATERN52):
    """Matern covariance of smoothness 5/2 (default) or 3/2.

    k_{5/2}(r) = s (1 + sqrt5 r + 5 r^2 / 3) exp(-sqrt5 r);
    k_{3/2}(r) = s (1 + sqrt3 r) exp(-sqrt3 r)  (the paper's kernel, Section 4.3).
    """
    r = np.asarray(r, dtype=np.float64)
    if kernel == MATERN52:
        a = math.sqrt(5.0) * r
        return signal_var * (1.0 + a + a * a / 3.0) * np.exp(-a)
    if kernel == MATERN32:
        a = math.sqrt(3.0) * r
        return signal_var * (1.0 + a) * np.exp(-a)
    raise ValueError(kernel)


def kumaraswamy_cdf(u, a, b):
    """Input warping of Section 4.3 (the Kumaraswamy CDF of the warping work
    the paper cites): w(u) = 1 - (1 - u^a)^b on [0, 1], a, b > 0."""
    u = np.clip(np.asarray(u, np.float64), 0.0, 1.0)
    return 1.0 - (1.0 - u ** a) ** b


class GP:
    """One objective's GP conditioned on the observations (Section 4.3).

    ``warp`` ([d][2], optional) gives each parameter's Kumaraswamy (a, b);
    ordinal features are warped before the distance, categoricals never."""

    def __init__(self, space, x_obs_words, y, lengthscale, signal_var, noise_var,
                 kernel: int = MATERN52, warp=None):
        self.space = space
        self.warp = None if warp is None else np.asarray(warp, np.float64)
        self.kernel = kernel
        self.lengthscale = np.asarray(lengthscale, np.float64)
        self.signal_var = float(signal_var)
        self.noise_var = float(noise_var)
        x = decode(space, x_obs_words)
        self.u_obs, self.is_cat = gp_features(space, x)
        self.y = np.asarray(y, np.float64)
        self._factor()

    def _factor(self):
        n = len(self.y)
        K = self.cov(self.u_obs, self.u_obs) + self.noise_var * np.eye(n)
        self.chol = np.linalg.cholesky(K)            # K + tau^2 I = L L^T
        self.alpha = sla.cho_solve((self.chol, True), self.y)  # (K + tau^2 I)^{-1} Y

    def warped(self, u):
        """Features with the ordinal coordinates warped (identity without warp)."""
        if self.warp is None:
            return u
        w = np.array(u, np.float64, copy=True)
        for c in np.nonzero(~self.is_cat)[0]:
            w[:, c] = kumaraswamy_cdf(u[:, c], self.warp[c, 0], self.warp[c, 1])
        return w

    def cov(self, ua, ub):
        return matern(scaled_distance(self.warped(ua), self.warped(ub), self.is_cat, self.lengthscale),
                      self.signal_var, self.kernel)

    def add_observations(self, u_new, y_new):
        """Condition again with extra (feature, value) pairs (plain refit)."""
        self.u_obs = np.concatenate([self.u_obs, u_new], axis=0)
        self.y = np.concatenate([self.y, np.asarray(y_new, np.float64)])
        self._factor()

    def posterior_u(self, u):
        """mu = k(x, X)(K + tau^2 I)^{-1} Y and
        sigma^2 = k(x, x) - k(x, X)(K + tau^2 I)^{-1} k(X, x), clamped at 0.

        Reading: sigma^2 is the variance of the latent f (tau^2 appears only
        inside the inverse, as printed)."""
        kstar = self.cov(u, self.u_obs)                      # [N][n]
        mu = kstar @ self.alpha
        v = sla.solve_triangular(self.chol, kstar.T, lower=True)   # L v = k*
        var = self.signal_var - np.sum(v * v, axis=0)
        return mu, np.maximum(var, 0.0)

    def posterior(self, words, n=None):
        u, _ = gp_features(self.space, decode(self.space, words, n))
        return self.posterior_u(u)

    def mean_condition(self, words, n=None):
        """sum_j |k(x, X_j) alpha_j|: the scale of the rounding error of any
        evaluation of mu as a dot product (used by the tests' tolerance)."""
        u, _ = gp_features(self.space, decode(self.space, words, n))
        return np.abs(self.cov(u, self.u_obs)) @ np.abs(self.alpha)


# --------------------------------------------------------------------------
# 4a. expected improvement, Eq. (6)

def norm_cdf(z):
    return 0.5 * erfc(-np.asarray(z, np.float64) / math.sqrt(2.0))


def norm_pdf(z):
    z = np.asarray(z, np.float64)
    return np.exp(-0.5 * z * z) / math.sqrt(2.0 * math.pi)


def expected_improvement(mu, var, y_best: float, xi: float = 1e-4):
    """EI(x) = E[max(0, f(x) + xi - f(x+))] for f(x) ~ N(mu, sigma^2).

    Closed form: with a = mu - y+ + xi and z = a / sigma,
    EI = a Phi(z) + sigma phi(z); EI = max(0, a) when sigma = 0.
    Reading: xi enters with the sign printed in Eq. (6); xi = 1e-4 (Section 4.5).
    """
    mu = np.asarray(mu, np.float64)
    sd = np.sqrt(np.maximum(np.asarray(var, np.float64), 0.0))
    a = mu - y_best + xi
    out = np.maximum(a, 0.0)
    pos = sd > 0
    z = np.where(pos, a / np.where(pos, sd, 1.0), 0.0)
    return np.where(pos, a * norm_cdf(z) + sd * norm_pdf(z), out)


# --------------------------------------------------------------------------
# 4b. hypervolume (Section 4.4) and Monte-Carlo EHVI, Eq. (7)

def pareto_front(Y: np.ndarray, ref: np.ndarray) -> np.ndarray:
    """Non-dominated points of Y (rows, maximised) that strictly dominate r.

    Points that do not lie strictly above r in every objective enclose no
    volume with r, so they are left out (they add 0, cf. Eq. 8)."""
    Y = np.asarray(Y, np.float64)
    ref = np.asarray(ref, np.float64)
    cand = [y for y in Y if np.all(y > ref)]
    front = []
    for i, y in enumerate(cand):
        dominated = False
        for j, z in enumerate(cand):
            if j != i and np.all(z >= y) and (np.any(z > y) or j < i):
                dominated = True   # a strictly better point, or an earlier duplicate
                break
        if not dominated:
            front.append(y)
    return np.array(front).reshape(-1, len(ref))


def nondominated_cells(front: np.ndarray, ref: np.ndarray):
    """The region {z >= r : no front point dominates z} as grid cells.

    The grid's coordinates on axis j are r_j, every front coordinate, and
    +inf.  Domination is constant inside a cell, so the region is exactly the
    union of the cells whose upper corner no front point weakly dominates
    (cells reaching +inf on some axis are never dominated).  Returns the
    cells' lower and upper corners, each [C][M].
    """
    front = np.asarray(front, np.float64).reshape(-1, len(ref))
    ref = np.asarray(ref, np.float64)
    M = len(ref)
    axes = []
    for j in range(M):
        c = np.unique(np.concatenate([[ref[j]], front[:, j]]))
        axes.append(np.concatenate([c, [np.inf]]))
    grids_lo = np.meshgrid(*[a[:-1] for a in axes], indexing="ij")
    grids_hi = np.meshgrid(*[a[1:] for a in axes], indexing="ij")
    lo = np.stack([g.ravel() for g in grids_lo], axis=1)
    hi = np.stack([g.ravel() for g in grids_hi], axis=1)
    if len(front):
        dom = np.zeros(len(lo), dtype=bool)
        for p in front:
            dom |= np.all(p[None, :] >= hi, axis=1)
        lo, hi = lo[~dom], hi[~dom]
    return lo, hi


def hypervolume(points: np.ndarray, ref: np.ndarray) -> float:
    """HV(P): volume dominated by P and dominating r (Section 4.4), by
    summing the grid cells whose upper corner some point dominates."""
    P = pareto_front(points, ref)
    if len(P) == 0:
        return 0.0
    ref = np.asarray(ref, np.float64)
    M = len(ref)
    axes = [np.unique(np.concatenate([[ref[j]], P[:, j]])) for j in range(M)]
    lo = np.stack([g.ravel() for g in np.meshgrid(*[a[:-1] for a in axes], indexing="ij")], 1)
    hi = np.stack([g.ravel() for g in np.meshgrid(*[a[1:] for a in axes], indexing="ij")], 1)
    dom = np.zeros(len(lo), dtype=bool)
    for p in P:
        dom |= np.all(p[None, :] >= hi, axis=1)
    return float(np.sum(np.prod(hi[dom] - lo[dom], axis=1)))


def hvi_cells(y: np.ndarray, lo: np.ndarray, hi: np.ndarray) -> np.ndarray:
    """HV(P u {y}) - HV(P) for rows y [K][M]: the volume of [r, y] that lies in
    the non-dominated region, sum_c prod_j max(0, min(y_j, hi_cj) - lo_cj)."""
    y = np.atleast_2d(np.asarray(y, np.float64))
    ext = np.minimum(y[:, None, :], hi[None, :, :]) - lo[None, :, :]
    return np.sum(np.prod(np.maximum(ext, 0.0), axis=2), axis=1)


def ehvi_mc(mu: np.ndarray, var: np.ndarray, eps: np.ndarray, front, ref) -> np.ndarray:
    """Monte-Carlo EHVI (Eq. 7) with common base samples.

    Reading: the expectation of Eq. (7) over the independent per-objective
    posteriors (Section 4.3: outputs modelled independently) is estimated with
    fixed base samples eps[S][M]: y_s = mu + sigma * eps_s, EHVI = mean_s HVI(y_s).
    mu, var: [N][M].
    """
    lo, hi = nondominated_cells(front, ref)
    mu = np.asarray(mu, np.float64)
    sd = np.sqrt(np.maximum(np.asarray(var, np.float64), 0.0))
    eps = np.asarray(eps, np.float64)
    out = np.empty(len(mu))
    for i in range(len(mu)):
        ys = mu[i][None, :] + sd[i][None, :] * eps
        out[i] = np.mean(hvi_cells(ys, lo, hi))
    return out


def expected_excess(mu, sd, a):
    """psi(a) = E[max(0, Y - a)] for Y ~ N(mu, sd^2): sd phi(z) + (mu - a) Phi(z)
    with z = (mu - a) / sd; max(0, mu - a) when sd = 0; 0 at a = +inf."""
    mu = np.asarray(mu, np.float64)
    sd = np.asarray(sd, np.float64)
    a = np.asarray(a, np.float64)
    fin = np.isfinite(a)
    d = np.where(fin, mu - np.where(fin, a, 0.0), 0.0)
    pos = sd > 0
    z = np.where(pos, d / np.where(pos, sd, 1.0), 0.0)
    val = np.where(pos, sd * norm_pdf(z) + d * norm_cdf(z), np.maximum(d, 0.0))
    return np.where(fin, val, 0.0)


def ehvi_analytic(mu: np.ndarray, var: np.ndarray, front, ref) -> np.ndarray:
    """EHVI (Eq. 7) as an exact expectation over independent Gaussian
    objectives, the closed form the paper's EHVI reference (Yang et al.)
    builds on: over the non-dominated cells [l, u),
      EHVI = sum_c prod_j E[max(0, min(Y_j, u_cj) - l_cj)],
    the expectation of a product of independent factors being the product of
    their expectations; each factor is int_l^u P(Y_j > t) dt = psi(l) - psi(u)
    with psi(a) = E[max(0, Y_j - a)].  mu, var: [N][M]."""
    lo, hi = nondominated_cells(front, ref)
    mu = np.asarray(mu, np.float64)
    sd = np.sqrt(np.maximum(np.asarray(var, np.float64), 0.0))
    out = np.empty(len(mu))
    for i in range(len(mu)):
        f = expected_excess(mu[i][None, :], sd[i][None, :], lo) - expected_excess(mu[i][None, :], sd[i][None, :], hi)
        out[i] = np.sum(np.prod(f, axis=1))
    return out


# --------------------------------------------------------------------------
# 5. top-q selection (Section 4.7)

def select_topq(acq, mask, q: int):
    """The q largest acquisition values among feasible candidates.

    Reading: order is value descending, then index ascending (lowest index
    wins a tie); candidates that are masked out, -inf or NaN are never
    selected; fewer than q eligible candidates return them all (the
    shortfall is filled by Sobol sampling outside this step, Section 4.6)."""
    acq = np.asarray(acq, np.float64)
    n = len(acq)
    ok = np.isfinite(acq) | (acq == np.inf)
    ok &= ~np.isnan(acq)
    if mask is not None:
        ok &= np.asarray(mask, bool)
    idx = np.nonzero(ok)[0]
    keys = sorted(idx.tolist(), key=lambda i: (-acq[i], i))
    take = keys[:q]
    return np.array(take, np.int64), acq[take], len(take)


# --------------------------------------------------------------------------
# whole round

def score_round(inst, acq_kind: str, xi: float = 1e-4, kernel: int = MATERN52,
                subset: np.ndarray | None = None, warp=None):
    """One suggestion round on an instance: masks, votes, posterior, acquisition.

    ``subset`` restricts the GP/acquisition work to those candidate indices
    (masks and votes are still computed for all of them)."""
    w = inst.workload
    n = inst.n_cand
    words = inst.cand
    mask_k = prune_mask(inst.space, inst.clauses, words, n)
    votes = rf_votes(inst.nodes, inst.tree_offset, inst.space, words, n)
    feas = mask_k & pof_feasible(votes, inst.n_trees, w.leaf_scale, w.delta_num, w.delta_den)
    sel = np.arange(n) if subset is None else np.asarray(subset)
    gps = [GP(inst.space, inst.x_obs, inst.y_obs[m], inst.lengthscale[m], inst.signal_var[m],
              inst.noise_var[m], kernel, warp=None if warp is None else warp[m]) for m in range(inst.n_obj)]
    sub_words = words[:, sel]
    mv = [gp.posterior(sub_words) for gp in gps]
    mu = np.stack([m for m, _ in mv], axis=1)
    var = np.stack([v for _, v in mv], axis=1)
    if acq_kind == "ei":
        a = expected_improvement(mu[:, 0], var[:, 0], float(np.max(inst.y_obs[0])), xi)
    elif acq_kind == "ehvi-exact":
        a = ehvi_analytic(mu, var, pareto_front(inst.y_obs.T, inst.ref), inst.ref)
    else:
        front = pareto_front(inst.y_obs.T, inst.ref)
        a = ehvi_mc(mu, var, inst.eps, front, inst.ref)
    a = np.where(feas[sel], a, -np.inf)
    return dict(mask_known=mask_k, votes=votes, feasible=feas, index=sel, mu=mu, var=var, acq=a)


# --------------------------------------------------------------------------
# 6. sequential picks with fantasies

def fantasy_picks(inst, q: int, feasible: np.ndarray, kernel: int = MATERN52,
                  forced: list | None = None, subset=None):
    """q sequential EHVI picks with kriging-believer fantasies (refit form).

    After each pick p the GP of every objective is conditioned again on the
    observations plus (x_p, mu(x_p)) with noise tau^2, the front is rebuilt
    with mu(x_p) added, and EHVI is recomputed over the pool with the picked
    candidates excluded.  ``forced`` replays a given pick sequence (to follow
    another implementation's choices step by step) instead of taking argmax.
    ``subset`` (pool indices; with ``forced`` only) evaluates the steps at
    those candidates and the forced picks alone, for pools too large to
    evaluate whole.  Returns the picks, the evaluated indices and the
    acquisition, variance, mean and front of each step (arrays over the
    evaluated indices).
    """
    n = inst.n_cand
    words = inst.cand[:, :n]
    if subset is None:
        sel = np.arange(n)
    else:
        if forced is None:
            raise ValueError("subset needs forced picks")
        sel = np.unique(np.concatenate([np.asarray(subset, np.int64), np.asarray(forced[:q], np.int64)]))
    where = {int(i): k for k, i in enumerate(sel)}
    gps = [GP(inst.space, inst.x_obs, inst.y_obs[m], inst.lengthscale[m],
              inst.signal_var[m], inst.noise_var[m], kernel) for m in range(inst.n_obj)]
    u_pool, _ = gp_features(inst.space, decode(inst.space, np.ascontiguousarray(words[:, sel]), len(sel)))
    mu0 = np.stack([gp.posterior_u(u_pool)[0] for gp in gps], axis=1)
    Yf = inst.y_obs.T.astype(np.float64)
    picks, acqs, mus, vars_, fronts = [], [], [], [], []
    eligible = np.asarray(feasible, bool)[sel].copy()
    for j in range(q):
        var = np.stack([gp.posterior_u(u_pool)[1] for gp in gps], axis=1)
        front = pareto_front(Yf, inst.ref)
        fronts.append(front)
        a = ehvi_mc(mu0, var, inst.eps, front, inst.ref)
        a = np.where(eligible, a, -np.inf)
        if forced is not None:
            if j >= len(forced):
                break
            p = int(forced[j])
        else:
            idx, _, cnt = select_topq(a, None, 1)
            if cnt == 0:
                break
            p = int(sel[idx[0]])
        k = where[p]
        picks.append(p)
        acqs.append(a)
        vars_.append(var)
        mus.append(mu0)
        eligible[k] = False
        for m, gp in enumerate(gps):
            gp.add_observations(u_pool[k:k + 1], [mu0[k, m]])
        Yf = np.concatenate([Yf, mu0[k:k + 1]], axis=0)
    return dict(picks=picks, index=sel, acq=acqs, var=vars_, mu=mus, fronts=fronts)


# --------------------------------------------------------------------------
# 7. MACE for single-objective suggestion (Sections 4.5 and 4.7)

def upper_confidence_bound(mu, var, kappa: float):
    """UCB(x) = mu(x) + beta * sigma(x), the UCB equation of Section 4.5.

    Reading: the coefficient multiplies sigma as printed; its value for
    tuning iteration t (beta_t of Section 4.5) is computed by the caller
    and passed in as ``kappa``."""
    sd = np.sqrt(np.maximum(np.asarray(var, np.float64), 0.0))
    return np.asarray(mu, np.float64) + float(kappa) * sd


def probability_of_improvement(mu, var, y_best: float, xi: float = 1e-4):
    """PI(x) = P(f(x) + xi > f(x+)) for f(x) ~ N(mu, sigma^2), the PI equation
    of Section 4.5: Phi((mu + xi - y+) / sigma).

    Reading: with sigma = 0 the event is certain when mu + xi > y+ and
    impossible otherwise (strict inequality, as printed)."""
    mu = np.asarray(mu, np.float64)
    sd = np.sqrt(np.maximum(np.asarray(var, np.float64), 0.0))
    a = mu - y_best + xi
    pos = sd > 0
    z = np.where(pos, a / np.where(pos, sd, 1.0), 0.0)
    return np.where(pos, norm_cdf(z), (a > 0).astype(np.float64))


def mace_acquisitions(mu, var, y_best: float, xi: float, kappa: float) -> np.ndarray:
    """The three acquisition values MACE ranks candidates by (Section 4.5):
    rows UCB, PI, EI, each to be maximised."""
    return np.stack([upper_confidence_bound(mu, var, kappa),
                     probability_of_improvement(mu, var, y_best, xi),
                     expected_improvement(mu, var, y_best, xi)])


def nondominated(Y) -> np.ndarray:
    """Boolean mask of the rows of Y (points, maximised) that no other row
    dominates: row j dominates row i when Y_j >= Y_i in every column and
    Y_j > Y_i in at least one.  Equal rows do not dominate each other, so
    duplicates of a front point are all on the front.  Straight from the
    definition: every pair is compared (in blocks of rows)."""
    Y = np.asarray(Y, np.float64)
    n = len(Y)
    out = np.ones(n, bool)
    for s in range(0, n, 256):
        blk = Y[s:s + 256]
        ge = np.all(Y[None, :, :] >= blk[:, None, :], axis=2)
        gt = np.any(Y[None, :, :] > blk[:, None, :], axis=2)
        out[s:s + 256] = ~np.any(ge & gt, axis=1)
    return out


_SM_GAMMA = 0x9E3779B97F4A7C15
_SM_MASK = (1 << 64) - 1


def splitmix64(seed: int, i: int) -> int:
    """Output i (0-based) of the SplitMix64 generator seeded with ``seed``
    (Steele, Lea and Flood, OOPSLA 2014, in the form Vigna publishes): the
    state after i + 1 steps is seed + (i + 1) * 0x9E3779B97F4A7C15, passed
    through the generator's 64-bit finaliser."""
    z = (seed + (i + 1) * _SM_GAMMA) & _SM_MASK
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & _SM_MASK
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & _SM_MASK
    return z ^ (z >> 31)


def mace_select(acq3, mask, k: int, seed: int):
    """k candidates drawn at random from the Pareto front of (UCB, PI, EI)
    (Section 4.7: for SOBO, the k suggestions are picked at random from the
    front of the three acquisition functions).

    Reading: eligible candidates are those with mask set whose three values
    are neither NaN nor -inf; the front is taken over eligible candidates
    only.  The random draw gives candidate i the key splitmix64(seed, i) and
    takes the k front members with the smallest keys (the lower index on
    equal keys), in that order: a uniformly random k-subset in random order.
    A front smaller than k is returned whole.

    Returns (picks, front indices in ascending order, number of picks)."""
    A = np.asarray(acq3, np.float64)
    n = A.shape[1]
    ok = ~np.any(np.isnan(A) | (A == -np.inf), axis=0)
    if mask is not None:
        ok &= np.asarray(mask, bool)[:n]
    idx = np.nonzero(ok)[0]
    front = idx[nondominated(A[:, idx].T)] if len(idx) else idx
    order = sorted(front.tolist(), key=lambda i: (splitmix64(seed, i), i))
    picks = np.array(order[:k], np.int64)
    return picks, np.sort(front).astype(np.int64), len(picks)


# --------------------------------------------------------------------------
# 8. the tuning loop's sampling and threshold control (Algorithm 1, Section 4.6)

def primitive_polynomials(count: int):
    """The first ``count`` primitive polynomials over GF(2) of degree >= 1,
    by degree, then by their middle coefficients read as a binary number.

    A polynomial x^s + a_1 x^(s-1) + ... + a_(s-1) x + 1 (bit mask with bits
    s and 0 set) is primitive when x has multiplicative order exactly
    2^s - 1 modulo it.  Returned as (s, a) with a = a_1 ... a_(s-1) as an
    integer (a_1 the most significant bit)."""
    def mulmod(p, q, poly, s):
        r = 0
        while q:
            if q & 1:
                r ^= p
            q >>= 1
            p <<= 1
            if p >> s & 1:
                p ^= poly
        return r

    def order_is_full(poly, s):
        e = (1 << s) - 1
        # x^k mod poly by repeated multiplication; the order divides 2^s - 1
        x = 1
        for k in range(1, e + 1):
            x = mulmod(x, 2, poly, s)
            if x == 1:
                return k == e
        return False

    out = []
    s = 1
    while len(out) < count:
        for a in range(1 << (s - 1)):
            poly = (1 << s) | (a << 1) | 1
            if order_is_full(poly, s):
                out.append((s, a))
                if len(out) == count:
                    break
        s += 1
    return out


def sobol_integers(d: int, n: int, skip: int = 0) -> np.ndarray:
    """Points skip .. skip + n - 1 of the d-dimensional Sobol sequence as
    32-bit integers X (the point is X / 2^32), uint64 array [n][d].

    Dimension 0 is the van der Corput sequence (V_k = 2^(32-k)).  Dimension
    j >= 1 uses the j-th primitive polynomial (degree s, coefficients a_i)
    with unit initial direction integers m_1 = ... = m_s = 1 and the
    recurrence m_k = 2 a_1 m_(k-1) xor 4 a_2 m_(k-2) xor ... xor
    2^(s-1) a_(s-1) m_(k-s+1) xor 2^s m_(k-s) xor m_(k-s); V_k = m_k 2^(32-k).
    Point i is the xor of V_k over the set bits k - 1 of i."""
    polys = primitive_polynomials(max(d - 1, 0))
    V = np.zeros((d, 33), dtype=object)
    for k in range(1, 33):
        V[0, k] = 1 << (32 - k)
    for j in range(1, d):
        s, a = polys[j - 1]
        m = [0] * 33
        for k in range(1, 33):
            if k <= s:
                m[k] = 1
            else:
                v = m[k - s] ^ (m[k - s] << s)
                for i in range(1, s):
                    if (a >> (s - 1 - i)) & 1:
                        v ^= m[k - i] << i
                m[k] = v
            V[j, k] = m[k] << (32 - k)
    out = np.zeros((n, d), dtype=np.uint64)
    for r in range(n):
        i = skip + r
        for j in range(d):
            x, k = 0, 1
            while i >> (k - 1):
                if (i >> (k - 1)) & 1:
                    x ^= V[j, k]
                k += 1
            out[r, j] = x
    return out


def sobol_configs(space, n: int, skip: int = 0) -> np.ndarray:
    """Sobol points mapped onto the search space as stored words [d][n]
    (Section 4.6: shortfall fill; Algorithm 1: initial design).

    Reading: with u = X / 2^32 in [0, 1) per dimension, in fp64:
    integer log-uniform: round(exp(ln lo + u (ln hi - ln lo))) clamped to
    [lo, hi] (half to even); integer uniform: lo + floor(u (hi - lo + 1));
    categorical: floor(u n_choices); continuous: lo + u (hi - lo), stored as
    float32."""
    d = len(space)
    X = sobol_integers(d, n, skip)
    words = np.zeros((d, n), np.uint32)
    for j in range(d):
        u = X[:, j].astype(np.float64) / 4294967296.0
        p = space[j]
        kind, lo, hi = int(p["kind"]), float(p["lo"]), float(p["hi"])
        if kind == INT_LOG:
            v = np.clip(np.rint(np.exp(math.log(lo) + u * (math.log(hi) - math.log(lo)))), lo, hi)
            words[j] = v.astype(np.int64).astype(np.int32).view(np.uint32)
        elif kind == INT_UNIFORM:
            v = np.minimum(lo + np.floor(u * (hi - lo + 1.0)), hi)
            words[j] = v.astype(np.int64).astype(np.int32).view(np.uint32)
        elif kind == CATEGORICAL:
            v = np.floor(u * int(p["n_choices"]))
            words[j] = v.astype(np.int64).astype(np.int32).view(np.uint32)
        else:
            words[j] = (lo + u * (hi - lo)).astype(np.float32).view(np.uint32)
    return words


def delta_update(delta: float, count: int, k: int, any_invalid: bool, step: float = 0.05):
    """Algorithm 1's feasibility-threshold controller after a batch of k
    suggestions: an invalid result raises Delta to min(0.75, max(0.5,
    Delta + step)) and clears the count of feasible suggestions; otherwise
    the count grows by k and, once it reaches 5, Delta drops to
    max(0.25, Delta - step) and the count loses 5.  Reading: the printed
    max(0.5, .) is applied literally (an invalid result lifts Delta to at
    least 0.5)."""
    if any_invalid:
        return min(0.75, max(0.5, delta + step)), 0
    count += k
    if count >= 5:
        delta = max(0.25, delta - step)
        count -= 5
    return delta, count


# --------------------------------------------------------------------------
# 9. random-forest training (Algorithm 1's TRAIN; Section 4.6)

def train_cart(feats: np.ndarray, labels: np.ndarray, boot: np.ndarray, max_depth: int, leaf_scale: int):
    """One regression tree on the bootstrap sample ``boot`` (indices into the
    observations), grown breadth first.

    feats [n][d] float32 (the stored values as floats), labels 0/1.
    Reading (CART with squared error, as the paper's sklearn forest): a node
    with m samples and p positives has SSE p (m - p) / m; it becomes a leaf
    at depth max_depth, when pure, or when no split separates its samples;
    otherwise it takes the split "x_f <= v" (v a sample value of feature f,
    not the node's largest) with the smallest SSE(left) + SSE(right),
    compared exactly as fractions, ties to the lower f, then the lower v
    (-0 and +0 count as one value, stored as +0).  A leaf stores round(leaf_scale p / m) (halves up) votes.  Nodes are
    numbered breadth first, so the children of a node are adjacent and
    follow it.  Returns a list of (val, left, feat, is_leaf), left counted
    from the tree's first node."""
    feats = np.asarray(feats, np.float32)
    labels = np.asarray(labels).astype(np.int64)
    nodes = []
    queue = [(list(int(i) for i in boot), 0)]
    head = 0
    while head < len(queue):
        samp, depth = queue[head]
        head += 1
        m = len(samp)
        p = int(sum(labels[i] for i in samp))
        best = None
        if depth < max_depth and 0 < p < m:
            for f in range(feats.shape[1]):
                vals = sorted({float(feats[i, f]) for i in samp})
                for v in vals[:-1]:
                    left = [i for i in samp if float(feats[i, f]) <= v]
                    nl, pl = len(left), int(sum(labels[i] for i in left))
                    nr, pr = m - nl, p - pl
                    # SSE(left) + SSE(right) = num / (nl nr)
                    num = pl * (nl - pl) * nr + pr * (nr - pr) * nl
                    den = nl * nr
                    key = (num, den)
                    if best is None or num * best[1] < best[0] * den:
                        best = (num, den, f, v)
        if best is None:
            votes = (2 * leaf_scale * p + m) // (2 * m)
            nodes.append([float(votes), 0, 0, True])
            continue
        _, _, f, v = best
        left = [i for i in samp if float(feats[i, f]) <= v]
        right = [i for i in samp if float(feats[i, f]) > v]
        child = len(queue)
        queue.append((left, depth + 1))
        queue.append((right, depth + 1))
        # -0 and +0 are one value ("x <= v" cannot tell them apart); the
        # threshold is stored as +0.
        nodes.append([0.0 if v == 0.0 else v, child, f, False])
    return [tuple(x) for x in nodes]


def train_forest(feats, labels, boot: np.ndarray, max_depth: int, leaf_scale: int):
    """Trees on the bootstrap samples boot [T][n] as (nodes structured array
    with fields val, left, feat, flags, and tree offsets [T + 1])."""
    trees = [train_cart(feats, labels, b, max_depth, leaf_scale) for b in boot]
    offs = np.zeros(len(trees) + 1, np.int32)
    offs[1:] = np.cumsum([len(t) for t in trees])
    out = np.zeros(offs[-1], dtype=[("val", "<f4"), ("left", "<u2"), ("feat", "u1"), ("flags", "u1")])
    k = 0
    for t in trees:
        for val, left, f, leaf in t:
            out[k] = (val, left, f, 1 if leaf else 0)
            k += 1
    return out, offs


# --------------------------------------------------------------------------
# 10. GP hyperparameters by maximum likelihood (Section 4.3)

def _matern_and_slope(r, kernel):
    """k(r) / s_f^2 and its derivative in r^2 (finite at r = 0):
    5/2: (1 + a + a^2/3) e^-a and -(5/6)(1 + a) e^-a, a = sqrt5 r;
    3/2: (1 + a) e^-a and -(3/2) e^-a, a = sqrt3 r."""
    r = np.asarray(r, np.float64)
    if kernel == MATERN52:
        a = math.sqrt(5.0) * r
        e = np.exp(-a)
        return (1.0 + a + a * a / 3.0) * e, -(5.0 / 6.0) * (1.0 + a) * e
    if kernel == MATERN32:
        a = math.sqrt(3.0) * r
        e = np.exp(-a)
        return (1.0 + a) * e, -1.5 * e
    raise ValueError(kernel)


def log_marginal_likelihood(space, x_obs_words, y, theta, kernel: int = MATERN52):
    """log p(y | X, theta) of the zero-mean GP of Section 4.3 and its
    gradient in theta = (ln l_1 .. ln l_d, ln s_f^2, ln tau^2).

    With K = s_f^2 k(r) + tau^2 I and alpha = K^{-1} y:
      lml = -y^T alpha / 2 - log det K / 2 - n log(2 pi) / 2,
      d lml / d theta_p = tr((alpha alpha^T - K^{-1}) dK/dtheta_p) / 2,
    dK/d ln s_f^2 = s_f^2 k(r), dK/d ln tau^2 = tau^2 I and
    dK/d ln l_c = -2 s_f^2 k'(r^2) D_c, where D_c is the term of feature c in
    r^2 ((u_c - u'_c)^2 / l_c^2, or [u_c != u'_c] / l_c^2 for a category).
    Returns (lml, grad[d + 2])."""
    theta = np.asarray(theta, np.float64)
    d = len(space)
    ell = np.exp(theta[:d])
    sf2, tau2 = math.exp(theta[d]), math.exp(theta[d + 1])
    u, is_cat = gp_features(space, decode(space, x_obs_words))
    y = np.asarray(y, np.float64)
    n = len(y)
    D = np.zeros((d, n, n))
    for c in range(d):
        if is_cat[c]:
            D[c] = (u[:, c][:, None] != u[:, c][None, :]).astype(np.float64) / (ell[c] * ell[c])
        else:
            diff = (u[:, c][:, None] - u[:, c][None, :]) / ell[c]
            D[c] = diff * diff
    r = np.sqrt(D.sum(axis=0))
    k, dk = _matern_and_slope(r, kernel)
    K = sf2 * k + tau2 * np.eye(n)
    L = np.linalg.cholesky(K)
    alpha = sla.cho_solve((L, True), y)
    Kinv = sla.cho_solve((L, True), np.eye(n))
    lml = -0.5 * y @ alpha - np.sum(np.log(np.diag(L))) - 0.5 * n * math.log(2.0 * math.pi)
    Wm = np.outer(alpha, alpha) - Kinv
    grad = np.zeros(d + 2)
    for c in range(d):
        grad[c] = 0.5 * np.sum(Wm * (-2.0 * sf2 * dk * D[c]))
    grad[d] = 0.5 * np.sum(Wm * (sf2 * k))
    grad[d + 1] = 0.5 * tau2 * np.trace(Wm)
    return float(lml), grad


def fit_hyperparameters(space, x_obs_words, y, theta0, lo, hi, free, steps: int, lr: float,
                        kernel: int = MATERN52):
    """Maximum-likelihood hyperparameters from the start theta0 by projected
    Adam ascent (Kingma and Ba's Adam: beta1 = 0.9, beta2 = 0.999,
    eps = 1e-8), `steps` steps with the step size decaying linearly,
    lr (1 - t / steps) at step t = 0 .. steps-1; after each step theta is
    clipped to [lo, hi]; parameters with free[p] == 0 stay at theta0.
    Reading: the paper learns tau^2 by maximum likelihood (Section 4.3);
    which parameters are free is the caller's choice (tau^2 alone is the
    paper's statement).  Returns (theta, lml) at the last step."""
    theta = np.array(theta0, np.float64)
    lo, hi = np.asarray(lo, np.float64), np.asarray(hi, np.float64)
    mask = np.asarray(free, bool).astype(np.float64)
    m1 = np.zeros_like(theta)
    m2 = np.zeros_like(theta)
    b1, b2, eps = 0.9, 0.999, 1e-8
    for t in range(steps):
        _, g = log_marginal_likelihood(space, x_obs_words, y, theta, kernel)
        g = g * mask
        m1 = b1 * m1 + (1.0 - b1) * g
        m2 = b2 * m2 + (1.0 - b2) * g * g
        mh = m1 / (1.0 - b1 ** (t + 1))
        vh = m2 / (1.0 - b2 ** (t + 1))
        step = lr * (1.0 - t / steps)
        theta = np.clip(theta + step * mh / (np.sqrt(vh) + eps), lo, hi)
    lml, _ = log_marginal_likelihood(space, x_obs_words, y, theta, kernel)
    return theta, lml
