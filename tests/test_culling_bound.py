"""The bound the fantasy pass culls with, checked on the CPU against the oracle.

The pass (fantasy.cu) skips a candidate's Monte-Carlo EHVI (Eq. 7) when an
upper bound of it cannot reach the best exact value found so far.  The bound:
the base samples in groups of 8 by rank of their first objective; each group's
corner is its largest value per objective; since the HVI of a point is monotone
in each objective, 8 x HVI(mu + sd * corner) bounds the group's HVI sum, and
the corners' sum bounds the EHVI.  This test checks that claim with the
oracle's own HVI (the exact volume over its cell decomposition) on the
workloads' fronts and base samples, for random moments, including candidates
far above the front, far below it, and with zero variance.
"""
import numpy as np
import pytest

import oracle as O
from workloads import Stream, make_instance, seeds


def corner_groups(eps):
    """The 8-sample groups by rank of the first objective (ties by index), as the pass forms them."""
    S = len(eps)
    order = np.lexsort((np.arange(S), eps[:, 0]))
    return order.reshape(S // 8, 8)


def bound(mu, var, eps, lo, hi):
    sd = np.sqrt(np.maximum(var, 0.0))
    out = np.zeros(len(mu))
    for g in corner_groups(eps):
        corner = eps[g].max(axis=0)
        out += 8.0 / len(eps) * O.hvi_cells(mu + sd * corner[None, :], lo, hi)
    return out


@pytest.mark.parametrize("name", ["d12-fantasy", "d8-ehvi2", "d10-ehvi3"])
def test_group_corner_bound_dominates_mc_ehvi(name):
    inst = make_instance(name, seeds(name)[0], n_cand=64)
    eps = np.asarray(inst.eps, np.float64)
    assert len(eps) % 16 == 0  # the pass culls only then
    front = O.pareto_front(inst.y_obs.T, inst.ref)
    lo, hi = O.nondominated_cells(front, inst.ref)
    st = Stream(41, f"cull-{name}")
    M = inst.n_obj
    span = np.max(np.abs(front)) + 1.0 if len(front) else 3.0
    K = 160 if M == 2 else 40      # (three objectives: many more cells per HVI)
    z = K // 8
    mu = st.normal(K * M).reshape(K, M) * span
    var = st.uniform(K * M).reshape(K, M) ** 3 * 4.0
    var[:z] = 0.0                  # no uncertainty: the bound is HVI at mu itself
    mu[z:2 * z] += 3.0 * span      # far above the front: every sample improves
    mu[2 * z:3 * z] -= 3.0 * span  # far below: nothing improves
    want = O.ehvi_mc(mu, var, eps, front, inst.ref)
    ub = bound(mu, var, eps, lo, hi)
    assert np.all(ub >= want * (1 - 1e-12) - 1e-15)
    assert np.allclose(ub[:z], want[:z], rtol=1e-12, atol=1e-15)  # sd = 0: exact
    assert np.all(ub[2 * z:3 * z] == 0.0) and np.all(want[2 * z:3 * z] == 0.0)
    # the bound is informative: it is below the EHVI-free rectangle bound for most candidates
    assert np.mean(ub < 0.999 * O.hvi_cells(mu + np.sqrt(var) * eps.max(axis=0)[None, :], lo, hi) + 1e-15) > 0.5


def test_a_plausible_mistake_breaks_the_bound():
    """Corners taken as the groups' smallest values (a wrong sign of the
    bound's direction) do not bound the EHVI: the check above would fail."""
    name = "d12-fantasy"
    inst = make_instance(name, seeds(name)[0], n_cand=64)
    eps = np.asarray(inst.eps, np.float64)
    front = O.pareto_front(inst.y_obs.T, inst.ref)
    lo, hi = O.nondominated_cells(front, inst.ref)
    st = Stream(43, "cull-wrong")
    mu = st.normal(100 * inst.n_obj).reshape(100, inst.n_obj)
    var = st.uniform(100 * inst.n_obj).reshape(100, inst.n_obj) + 0.1
    want = O.ehvi_mc(mu, var, eps, front, inst.ref)
    sd = np.sqrt(var)
    wrong = np.zeros(len(mu))
    for g in corner_groups(eps):
        wrong += 8.0 / len(eps) * O.hvi_cells(mu + sd * eps[g].min(axis=0)[None, :], lo, hi)
    assert np.any(wrong < want - 1e-9)
