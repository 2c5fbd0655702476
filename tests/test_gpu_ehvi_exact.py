"""Exact EHVI over independent Gaussian objectives (the closed form of Eq. 7's
expectation) through the C ABI, against the oracle's own cell decomposition.

Bar: 1e-6 + 1e-4 |oracle| plus a derived fp32 term.  Each box factor is a
difference psi(l) - psi(u) of two fp32 evaluations, each with an error of a
few ulps of max(psi, |mu - a|, sigma); a narrow box far below mu loses the
relative accuracy of its factor to that cancellation.  The test adds, per
box and objective, 16 u (psi(l) + psi(u) + |mu - l| + sigma) times the other
factors (u = 2^-24), the first-order effect of those errors on the sum.
Values from the GPU's own posterior add the propagated posterior tolerance
as in the other acquisition tests.
"""
import numpy as np
import pytest

import oracle as O
from workloads import Stream, make_instance, seeds

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from parity_tol import ATOL, RTOL, posterior_tols, propagated_tol  # noqa: E402

U32 = 2.0 ** -24


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


def box_inputs(S, y, ref):
    lo, hi, _ = S.scoot_boxes_build(np.ascontiguousarray(y, np.float32), np.ascontiguousarray(ref, np.float32))
    grid, n_grid, corner = S.scoot_boxes_index(lo, hi)
    return lo, hi, dev(grid), n_grid, dev(corner.view(np.int32))


def rounding_tol(mu, var, lo, hi):
    """Derived fp32 term over the library's boxes (see the module docstring)."""
    mu = np.atleast_2d(mu)
    sd = np.sqrt(np.maximum(np.atleast_2d(var), 0.0))
    out = np.zeros(len(mu))
    for i in range(len(mu)):
        pl = O.expected_excess(mu[i][None, :], sd[i][None, :], lo.astype(np.float64))
        ph = O.expected_excess(mu[i][None, :], sd[i][None, :], hi.astype(np.float64))
        f = pl - ph
        e = 16 * U32 * (pl + ph + np.abs(mu[i][None, :] - lo) + sd[i][None, :])
        M = f.shape[1]
        for j in range(M):
            others = np.prod(np.delete(f, j, axis=1), axis=1)
            out[i] += np.sum(e[:, j] * others)
    return out


@pytest.mark.parametrize("M,npts", [(2, 1), (2, 40), (3, 9), (3, 30), (4, 6)])
def test_exact_ehvi_kernel_on_generated_moments(S, ctx, M, npts):
    st = Stream(500 + 13 * M + npts, "ehvix")
    ref = np.zeros(M, np.float32)
    y = (st.uniform(M * npts).reshape(M, npts) * 3.0).astype(np.float32)
    lo, hi, grid, n_grid, corner = box_inputs(S, y, ref)
    n = 3000 + 17
    mu = (st.normal(n * M).reshape(M, n) * 1.2 + 1.5).astype(np.float32)
    var = (st.uniform(n * M).reshape(M, n) ** 2 * 0.8).astype(np.float32)
    var[:, :40] = 0.0
    mask = (st.uniform(n) < 0.85).astype(np.uint8)
    acq = torch.full((n,), 7.0, device="cuda")
    S.scoot_acq_ehvi_exact(ctx, dev(mu), dev(var), n, grid, n_grid, corner, acq, dev(mask))
    ctx.check()
    g = np_(acq)
    assert np.all(g[mask == 0] == -np.inf)
    live = np.nonzero(mask)[0]
    front = O.pareto_front(y.T, ref)
    m64, v64 = mu.T[live].astype(np.float64), var.T[live].astype(np.float64)
    want = O.ehvi_analytic(m64, v64, front, ref)
    extra = rounding_tol(m64, v64, lo, hi)
    ratio = np.abs(g[live] - want) / (ATOL + RTOL * np.abs(want) + extra)
    plain = np.abs(g[live] - want) / (ATOL + RTOL * np.abs(want))
    print(f"[parity] exact EHVI M={M} P={len(front)} B={len(lo)}: max|err|/tol={ratio.max():.3f} "
          f"(stated tolerance alone: {plain.max():.3f})")
    assert ratio.max() <= 1.0
    # sigma = 0: the deterministic hypervolume improvement of mu
    z = live[live < 40]
    clo, chi = O.nondominated_cells(front, ref)
    assert np.allclose(g[z], O.hvi_cells(mu.T[z].astype(np.float64), clo, chi), rtol=1e-4, atol=1e-6)


def test_exact_ehvi_bad_corner_is_flagged(S, ctx):
    lo, hi, grid, n_grid, corner = box_inputs(S, np.array([[1.0, 2.0], [2.0, 1.0]], np.float32), np.zeros(2))
    bad = np_(corner).copy()
    bad[0, 0] = 0x7FFF0000  # upper index far beyond the grid
    mu = dev(np.ones((2, 64), np.float32))
    acq = torch.empty(64, device="cuda")
    S.scoot_acq_ehvi_exact(ctx, mu, mu, 64, grid, n_grid, dev(bad), acq)
    with pytest.raises(S.ScootError) as e:
        ctx.check()
    assert e.value.status == -4
    with pytest.raises(S.ScootError) as e:
        S.scoot_acq_ehvi_exact(ctx, mu, mu, 64, grid, np.array([400, 1], np.int32), corner, acq)
    assert e.value.status == -1


@pytest.mark.parametrize("name,k", [("tiny", 4096), ("d8-ehvi2", 1500), ("d10-ehvi3", 300)])
def test_score_ehvi_exact_parity(S, ctx, name, k):
    inst = make_instance(name, seeds(name)[1], n_cand=4096 + 61)
    n = inst.n_cand
    L = S.scoot_gp_layout_init(inst.space, inst.n_obs, inst.n_obj, 0)
    blob, _ = S.scoot_gp_prepare(inst.space, inst.x_obs, inst.y_obs, inst.lengthscale, inst.signal_var,
                                 inst.noise_var, L)
    state = dev(blob)
    cand = dev(inst.cand.view(np.int32))
    lo, hi, grid, n_grid, corner = box_inputs(S, inst.y_obs, inst.ref)
    mask = torch.empty(n, dtype=torch.uint8, device="cuda")
    S.scoot_prune(ctx, inst.space, inst.clauses, cand, n, mask)
    acq = torch.empty(n, device="cuda")
    S.scoot_score_ehvi_exact(ctx, L, state, cand, n, grid, n_grid, corner, acq, mask)
    ctx.check()
    g = np_(acq)
    known = O.prune_mask(inst.space, inst.clauses, inst.cand, n)
    assert np.array_equal(np.isfinite(g), known)
    idx = np.nonzero(known)[0]
    idx = idx[np.unique(np.linspace(0, len(idx) - 1, min(k, len(idx))).astype(int))]
    gps = [O.GP(inst.space, inst.x_obs, inst.y_obs[m], inst.lengthscale[m], inst.signal_var[m],
                inst.noise_var[m], 0) for m in range(inst.n_obj)]
    mu, var, e_mu, e_var = posterior_tols(gps, np.ascontiguousarray(inst.cand[:, idx]))
    front = O.pareto_front(inst.y_obs.T, inst.ref)
    f = lambda a, b: O.ehvi_analytic(a, b, front, inst.ref)
    want, tol = propagated_tol(f, mu, var, e_mu, e_var)
    tol = tol + rounding_tol(mu, var, lo, hi)
    ratio = np.abs(g[idx] - want) / tol
    print(f"[parity] score_ehvi_exact {name}: n={len(idx)} B={len(lo)} max|err|/tol={ratio.max():.3f}")
    assert ratio.max() <= 1.0
    # fused == posterior + acq_ehvi_exact (the posterior's product in fp32 SIMT, as in the fused
    # kernel: the same arithmetic; the tensor-core product has its own parity test)
    M = inst.n_obj
    mean = torch.empty((M, n), device="cuda")
    vv = torch.empty((M, n), device="cuda")
    S.scoot_ctx_set_tensor_cores(ctx, 0)
    try:
        S.scoot_gp_posterior(ctx, L, state, cand, n, mean, vv, mask)
    finally:
        S.scoot_ctx_set_tensor_cores(ctx, 1)
    acq2 = torch.empty(n, device="cuda")
    S.scoot_acq_ehvi_exact(ctx, mean, vv, n, grid, n_grid, corner, acq2, mask)
    g2 = np_(acq2)
    assert np.allclose(g2[known], g[known], rtol=1e-5, atol=1e-6)
