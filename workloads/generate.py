"""Seeded synthetic instances of the candidate-scoring workloads.

Everything here is input synthesis: the candidate pool, the observed
configurations, synthetic objective surfaces standing in for stress-test
results, GP hyperparameters, a random forest trained on a synthetic crash
label, the reference point and the Monte-Carlo base samples.  None of the
scoring arithmetic (pruning, tree walks, the GP posterior, acquisition
values, hypervolumes, box decompositions, selection) lives here; the CUDA
path and the oracle each implement those on their own.

Recipe (per workload ``w`` and master seed ``seed``):

* pool: int-log v = round(exp(U(ln lo, ln hi))) clamped to [lo, hi];
  int-uniform and categorical uniform; continuous uniform, rounded to fp32;
* observations: ``w.n_obs`` configurations from the same distribution;
* surfaces: per objective m, g_m(u) = sum_i sin(3 w_mi u_i) + 0.5 ||u - c_m||^2
  on the [0, 1] coordinates u of a configuration (log scale for int-log,
  index/(k-1) for categoricals), w_mi ~ U(0.5, 2), c_m ~ U(0, 1)^d; the
  observed value is sign_m * (g_m + noise), noise ~ N(0, noise_sd^2) with
  correlation ``noise_rho`` between objectives; values are standardised per
  objective over the observations;
* GP hyperparameters: lengthscales lognormal(0, 0.5) per objective and
  dimension, signal variance 1, noise variance (noise_sd / sd_m)^2 with a
  1e-6 floor;
* objectives conflict (M > 1): the maximised objective m is
  conflict_scale/sqrt(d) * g_m(u) + tradeoff_m * t(u), t a weighted sum of
  the batching/memory coordinates shared by all objectives;
* reference point: the default configuration's objectives (Section 4.5),
  read as a default that every observation improves on: the componentwise
  minimum of the standardised observed objectives;
* crash label: a configuration is labelled infeasible when a weighted sum of
  its coordinates exceeds the (1 - infeasible_frac) quantile over the
  observations, then each label flips with probability ``label_flip``;
* forest: ``w.n_trees`` CART regression trees (bootstrap resample, all
  features, squared-error splits at midpoints between adjacent distinct
  values, grown to purity or ``w.max_depth``), leaves storing
  round(leaf_scale * mean label) as integer votes;
* Monte-Carlo base samples: eps[S][M] ~ N(0, 1).
"""
from __future__ import annotations

import functools
from dataclasses import dataclass

import numpy as np

from .configs import CATEGORICAL, CONTINUOUS, INT_LOG, INT_UNIFORM, WORKLOADS, Workload
from .rng import Stream

PARAM_DTYPE = np.dtype([("kind", "<i4"), ("n_choices", "<i4"), ("lo", "<f4"), ("hi", "<f4")])
CLAUSE_DTYPE = np.dtype([
    ("n_guard", "<i4"), ("guard_param", "<i4", (2,)), ("guard_value", "<i4", (2,)),
    ("n_term", "<i4"), ("term_param", "<i4", (4,)),
    ("coef", "<i8", (4,)), ("rhs", "<i8"),
])
NODE_DTYPE = np.dtype([("val", "<f4"), ("left", "<u2"), ("feat", "u1"), ("flags", "u1")])
NODE_LEAF = 1

assert PARAM_DTYPE.itemsize == 16 and CLAUSE_DTYPE.itemsize == 80 and NODE_DTYPE.itemsize == 8


@dataclass
class Instance:
    workload: Workload
    seed: int
    space: np.ndarray       # PARAM_DTYPE[d]
    clauses: np.ndarray     # CLAUSE_DTYPE[n_clauses]
    cand: np.ndarray        # uint32[d][ld] words (int32 or float32 bits)
    n_cand: int
    x_obs: np.ndarray       # uint32[d][n] words, same encoding as cand
    y_obs: np.ndarray       # float32[M][n], standardised, to be maximised
    lengthscale: np.ndarray # float32[M][d]
    signal_var: np.ndarray  # float32[M]
    noise_var: np.ndarray   # float32[M]
    ref: np.ndarray         # float32[M]
    nodes: np.ndarray       # NODE_DTYPE[total]
    tree_offset: np.ndarray # int32[T+1]
    eps: np.ndarray         # float32[S][M] (S may be 0)
    label_obs: np.ndarray   # float64[n] crash label used to train the forest (1 = ran)

    @property
    def d(self):
        return self.cand.shape[0]

    @property
    def ld(self):
        return self.cand.shape[1]

    @property
    def n_obs(self):
        return self.x_obs.shape[1]

    @property
    def n_obj(self):
        return self.y_obs.shape[0]

    @property
    def n_trees(self):
        return len(self.tree_offset) - 1


def space_array(w: Workload) -> np.ndarray:
    a = np.zeros(w.d, PARAM_DTYPE)
    for i, p in enumerate(w.params):
        a[i] = (p.kind, p.n_choices, p.lo, p.hi)
    return a


def clause_array(w: Workload) -> np.ndarray:
    a = np.zeros(len(w.clauses), CLAUSE_DTYPE)
    for i, c in enumerate(w.clauses):
        a[i]["n_guard"] = len(c.guards)
        for g, (p, v) in enumerate(c.guards):
            a[i]["guard_param"][g] = p
            a[i]["guard_value"][g] = v
        a[i]["n_term"] = len(c.terms)
        for t, (p, k) in enumerate(c.terms):
            a[i]["term_param"][t] = p
            a[i]["coef"][t] = k
        a[i]["rhs"] = c.rhs
    return a


def draw_configs(w: Workload, st: Stream, n: int, ld: int | None = None) -> np.ndarray:
    """n configurations as uint32 words [d][ld] (columns beyond n are zero)."""
    ld = n if ld is None else ld
    out = np.zeros((w.d, ld), np.uint32)
    for i, p in enumerate(w.params):
        if p.kind == INT_LOG:
            u = st.uniform(n)
            v = np.rint(np.exp(np.log(p.lo) + u * (np.log(p.hi) - np.log(p.lo))))
            v = np.clip(v, p.lo, p.hi).astype(np.int32)
            out[i, :n] = v.view(np.uint32)
        elif p.kind == INT_UNIFORM:
            v = st.integers(int(p.lo), int(p.hi), n).astype(np.int32)
            out[i, :n] = v.view(np.uint32)
        elif p.kind == CATEGORICAL:
            v = st.integers(0, p.n_choices - 1, n).astype(np.int32)
            out[i, :n] = v.view(np.uint32)
        elif p.kind == CONTINUOUS:
            v = (p.lo + st.uniform(n) * (p.hi - p.lo)).astype(np.float32)
            v = np.clip(v, np.float32(p.lo), np.float32(p.hi))
            out[i, :n] = v.view(np.uint32)
        else:
            raise ValueError(p.kind)
    return out


def stored_values(w: Workload, words: np.ndarray) -> np.ndarray:
    """Stored values as float64 [n][d]: ints and category indices exactly, floats widened."""
    cols = []
    for i, p in enumerate(w.params):
        if p.kind == CONTINUOUS:
            cols.append(words[i].view(np.float32).astype(np.float64))
        else:
            cols.append(words[i].view(np.int32).astype(np.float64))
    return np.stack(cols, axis=1)


def _truth_coords(w: Workload, vals: np.ndarray) -> np.ndarray:
    """[0,1] coordinates on which the synthetic surfaces are defined."""
    u = np.empty_like(vals)
    for i, p in enumerate(w.params):
        v = vals[:, i]
        if p.kind == INT_LOG:
            u[:, i] = (np.log(v) - np.log(p.lo)) / (np.log(p.hi) - np.log(p.lo))
        elif p.kind == CATEGORICAL:
            u[:, i] = v / max(1, p.n_choices - 1)
        else:
            u[:, i] = (v - p.lo) / (p.hi - p.lo)
    return u


# ---------------------------------------------------------------- forest (CART)

def _best_split(xs: np.ndarray, ys: np.ndarray):
    """Lowest weighted squared-error split over all features; None if none."""
    n, d = xs.shape
    order = np.argsort(xs, axis=0, kind="stable")
    xsorted = np.take_along_axis(xs, order, axis=0)
    ysorted = ys[order]
    cs = np.cumsum(ysorted, axis=0)
    cs2 = np.cumsum(ysorted * ysorted, axis=0)
    tot, tot2 = cs[-1], cs2[-1]
    nl = np.arange(1, n, dtype=np.float64)[:, None]
    nr = n - nl
    sl, sl2 = cs[:-1], cs2[:-1]
    sse = (sl2 - sl * sl / nl) + ((tot2 - sl2) - (tot - sl) ** 2 / nr)
    valid = xsorted[1:] > xsorted[:-1]
    sse = np.where(valid, sse, np.inf)
    k = int(np.argmin(sse))  # row-major over (position, feature): first best
    pos, feat = divmod(k, d)
    if not np.isfinite(sse[pos, feat]):
        return None
    lo_v, hi_v = xsorted[pos, feat], xsorted[pos + 1, feat]
    thr = np.float32(0.5 * (lo_v + hi_v))
    if not (float(thr) >= lo_v and float(thr) < hi_v):
        thr = np.float32(lo_v)
    return feat, thr


def _grow(xs, ys, depth, max_depth, leaf_scale):
    if depth >= max_depth or len(ys) < 2 or np.all(ys == ys[0]):
        return ("leaf", float(np.floor(leaf_scale * ys.mean() + 0.5)))
    split = _best_split(xs, ys)
    if split is None:
        return ("leaf", float(np.floor(leaf_scale * ys.mean() + 0.5)))
    feat, thr = split
    go_left = xs[:, feat] <= float(thr)
    return ("split", feat, thr,
            _grow(xs[go_left], ys[go_left], depth + 1, max_depth, leaf_scale),
            _grow(xs[~go_left], ys[~go_left], depth + 1, max_depth, leaf_scale))


def _layout(tree) -> np.ndarray:
    """Breadth-first layout with the two children of a node adjacent."""
    nodes = [tree]
    out = []
    i = 0
    while i < len(nodes):
        nd = nodes[i]
        if nd[0] == "leaf":
            out.append((nd[1], 0, 0, NODE_LEAF))
        else:
            out.append((float(nd[2]), len(nodes), nd[1], 0))
            nodes.append(nd[3])
            nodes.append(nd[4])
        i += 1
    if len(out) > 65535:
        raise ValueError("tree too large for 16-bit child indices")
    arr = np.zeros(len(out), NODE_DTYPE)
    for j, (v, left, feat, flags) in enumerate(out):
        arr[j] = (v, left, feat, flags)
    return arr


def train_forest(w: Workload, st: Stream, feats: np.ndarray, labels: np.ndarray):
    trees = []
    n = len(labels)
    for _ in range(w.n_trees):
        boot = st.integers(0, n - 1, n)
        trees.append(_layout(_grow(feats[boot], labels[boot], 0, w.max_depth, w.leaf_scale)))
    offs = np.zeros(len(trees) + 1, np.int32)
    offs[1:] = np.cumsum([len(t) for t in trees])
    return np.concatenate(trees), offs


# ---------------------------------------------------------------- instance

def warp_params(w: Workload | str, seed: int) -> np.ndarray:
    """Input-warping parameters for the workload's GPs: float32 [M][d][2] of
    Kumaraswamy (a, b), each lognormal(0, 0.4) (hyperparameters are inputs of
    the path; the tuner would fit them).  Categorical entries are drawn too
    and ignored by both sides."""
    if isinstance(w, str):
        w = WORKLOADS[w]
    st = Stream(seed, "warp")
    return np.exp(st.normal(w.n_obj * w.d * 2) * 0.4).reshape(w.n_obj, w.d, 2).astype(np.float32)


def make_instance(w: Workload | str, seed: int, n_cand: int | None = None,
                  ld_pad: int = 4) -> Instance:
    """Build one seeded instance; ``n_cand`` overrides the pool size."""
    if isinstance(w, str):
        w = WORKLOADS[w]
    return _make(w, seed, w.n_cand if n_cand is None else int(n_cand), ld_pad)


@functools.lru_cache(maxsize=8)
def _make(w: Workload, seed: int, n_cand: int, ld_pad: int) -> Instance:
    d, M, n = w.d, w.n_obj, w.n_obs
    ld = max(ld_pad, -(-n_cand // ld_pad) * ld_pad)

    cand = draw_configs(w, Stream(seed, "pool"), n_cand, ld)
    x_obs = draw_configs(w, Stream(seed, "observations"), n)
    vals = stored_values(w, x_obs)
    u = _truth_coords(w, vals)

    st = Stream(seed, "surfaces")
    wts = 0.5 + 1.5 * st.uniform(M * d).reshape(M, d)
    ctr = st.uniform(M * d).reshape(M, d)
    axis = np.zeros(d)
    for p, wt in w.budget:
        axis[p] = wt
    sg = np.asarray(w.signs, np.float64)[:, None]

    def g(uu):
        base = np.stack([np.sin(3.0 * wts[m] * uu).sum(1) + 0.5 * ((uu - ctr[m]) ** 2).sum(1)
                         for m in range(M)])
        if M == 1:
            return base
        # Conflicting objectives (the appendix on conflicting TTFT and TPOT):
        # a shared trade-off axis enters the maximised objectives with
        # alternating signs.
        trade = np.stack([sg[m, 0] * w.tradeoff[m] * (uu @ axis) for m in range(M)])
        return w.conflict_scale / np.sqrt(d) * base + trade

    z = Stream(seed, "noise").normal(n * M).reshape(M, n)
    if M > 1 and w.noise_rho != 0.0:
        corr = np.full((M, M), w.noise_rho) + (1.0 - w.noise_rho) * np.eye(M)
        z = np.linalg.cholesky(corr) @ z
    raw = g(u) + w.noise_sd * z
    obj = sg * raw
    mean, sd = obj.mean(1, keepdims=True), obj.std(1, keepdims=True)
    y = ((obj - mean) / sd).astype(np.float32)
    # Reference point: the default configuration's objectives (Section 4.5),
    # taken as a default that every observation improves on, i.e. the
    # componentwise minimum of the observed values (a lower bound of every
    # objective over the observations, as the hypervolume definition wants).
    ref = y.min(axis=1).astype(np.float32)

    hs = Stream(seed, "hyper")
    lengthscale = np.exp(0.5 * hs.normal(M * d)).reshape(M, d).astype(np.float32)
    signal_var = np.ones(M, np.float32)
    noise_var = np.maximum(1e-6, (w.noise_sd / sd[:, 0]) ** 2).astype(np.float32)

    score = sum(wt * u[:, p] for p, wt in w.budget)
    thr = np.quantile(score, 1.0 - w.infeasible_frac)
    label = (score <= thr).astype(np.float64)
    flip = Stream(seed, "label_flip").uniform(n) < w.label_flip
    label = np.where(flip, 1.0 - label, label)
    nodes, offs = train_forest(w, Stream(seed, "forest"), vals, label)

    eps = Stream(seed, "mc_base").normal(w.n_mc * M).reshape(w.n_mc, M).astype(np.float32)

    return Instance(w, seed, space_array(w), clause_array(w), cand, n_cand, x_obs, y,
                    lengthscale, signal_var, noise_var, ref, nodes, offs, eps, label)
