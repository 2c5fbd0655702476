"""Input warping (Section 4.3: Matérn with input warping) through the C ABI:
the posterior and the fused EI of a warped GP state against the oracle's
warped GP, with Matérn-3/2 (the paper's kernel) and Matérn-5/2.

Bars as for the unwarped posterior: variance within 1e-6 + 1e-4 |oracle|,
mean with the added 2^-22 sum_j |k_j alpha_j| term, EI with the propagated
posterior tolerance.
"""
import numpy as np
import pytest

import oracle as O
from workloads import make_instance, seeds, warp_params

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


def np_(t):
    torch.cuda.synchronize()
    return t.cpu().numpy()


def warped_state(S, inst, warp, kernel):
    L = S.scoot_gp_layout_init(inst.space, inst.n_obs, inst.n_obj, kernel)
    blob, _ = S.scoot_gp_prepare_warped(inst.space, inst.x_obs, inst.y_obs, inst.lengthscale, inst.signal_var,
                                        inst.noise_var, warp, L)
    return L, dev(blob)


def oracle_gps(inst, warp, kernel):
    return [O.GP(inst.space, inst.x_obs, inst.y_obs[m], inst.lengthscale[m], inst.signal_var[m],
                 inst.noise_var[m], kernel, warp=warp[m]) for m in range(inst.n_obj)]


@pytest.mark.parametrize("name,kernel", [("d8-ehvi2", 1), ("d10-ei", 1), ("d10-ehvi3", 0), ("tiny", 1)])
def test_warped_posterior_parity(S, ctx, name, kernel):
    n = 4096 + 37
    inst = make_instance(name, seeds(name)[1], n_cand=n)
    warp = warp_params(name, 11)
    L, state = warped_state(S, inst, warp, kernel)
    M = inst.n_obj
    mean = torch.empty((M, n), device="cuda")
    var = torch.empty((M, n), device="cuda")
    S.scoot_gp_posterior(ctx, L, state, dev(inst.cand.view(np.int32)), n, mean, var)
    gm, gv = np_(mean), np_(var)
    for m, gp in enumerate(oracle_gps(inst, warp, kernel)):
        mu, v = gp.posterior(inst.cand, n)
        cond = gp.mean_condition(inst.cand, n)
        r_mu = np.abs(gm[m] - mu) / (ATOL + RTOL * np.abs(mu) + MU_COND * cond)
        r_v = np.abs(gv[m] - v) / (ATOL + RTOL * np.abs(v))
        print(f"[parity] warped {name} k{kernel} objective {m}: mu {r_mu.max():.3f}, var {r_v.max():.3f}")
        assert r_mu.max() <= 1.0 and r_v.max() <= 1.0
        # the warp matters: the unwarped oracle is far off somewhere
        mu0, _ = O.GP(inst.space, inst.x_obs, inst.y_obs[m], inst.lengthscale[m], inst.signal_var[m],
                      inst.noise_var[m], kernel).posterior(inst.cand, n)
        assert np.abs(mu0 - mu).max() > 1e-2


@pytest.mark.parametrize("tc", [1, 0], ids=["tensor", "simt"])
def test_warped_score_ei_matern32(S, ctx, tc):
    """The paper's kernel: Matérn-3/2 with input warping, fused with EI
    (either product of L^{-1} k)."""
    name = "d10-ei"
    n = 8192 + 5
    inst = make_instance(name, seeds(name)[2], n_cand=n)
    warp = warp_params(name, 12)
    L, state = warped_state(S, inst, warp, 1)
    cand = dev(inst.cand.view(np.int32))
    mask = torch.empty(n, dtype=torch.uint8, device="cuda")
    S.scoot_prune(ctx, inst.space, inst.clauses, cand, n, mask)
    acq = torch.empty(n, device="cuda")
    S.scoot_ctx_set_tensor_cores(ctx, tc)
    try:
        S.scoot_score_ei(ctx, L, state, cand, n, 1e-4, acq, mask)
        g = np_(acq)
    finally:
        S.scoot_ctx_set_tensor_cores(ctx, 1)
    known = O.prune_mask(inst.space, inst.clauses, inst.cand, n)
    idx = np.nonzero(known)[0][::3]
    mu, var, e_mu, e_var = posterior_tols(oracle_gps(inst, warp, 1), np.ascontiguousarray(inst.cand[:, idx]))
    yb = float(inst.y_obs[0].max())
    f = lambda a, b: O.expected_improvement(a[:, 0], b[:, 0], yb, 1e-4)
    want, tol = propagated_tol(f, mu, var, e_mu, e_var)
    ratio = np.abs(g[idx] - want) / tol
    print(f"[parity] warped Matérn-3/2 score_ei tc={tc}: n={len(idx)} max|err|/tol={ratio.max():.3f}")
    assert ratio.max() <= 1.0


def test_identity_warp_equals_no_warp(S, ctx):
    name = "d8-ehvi2"
    n = 2048
    inst = make_instance(name, seeds(name)[0], n_cand=n)
    ones = np.ones((inst.n_obj, inst.d, 2), np.float32)
    L, ws = warped_state(S, inst, ones, 0)
    blob, _ = S.scoot_gp_prepare(inst.space, inst.x_obs, inst.y_obs, inst.lengthscale, inst.signal_var,
                                 inst.noise_var, L)
    cand = dev(inst.cand.view(np.int32))
    out = []
    for st in (ws, dev(blob)):
        mean = torch.empty((2, n), device="cuda")
        var = torch.empty((2, n), device="cuda")
        S.scoot_gp_posterior(ctx, L, st, cand, n, mean, var)
        out.append((np_(mean), np_(var)))
    assert np.allclose(out[0][0], out[1][0], rtol=1e-5, atol=2e-6)
    assert np.allclose(out[0][1], out[1][1], rtol=1e-5, atol=2e-6)


def test_fantasy_refuses_a_warped_state(S, ctx):
    """The fantasy downdates rebuild the covariance without warping: a warped
    GP state stops the picks on the device, reported as SCOOT_EINVAL."""
    name = "d12-fantasy"
    inst = make_instance(name, seeds(name)[0], n_cand=4096)
    L, state = warped_state(S, inst, warp_params(name, 1), 0)
    fant, box_cap = S.scoot_fantasy_prepare(inst.space, inst.x_obs, inst.y_obs, inst.lengthscale, inst.signal_var,
                                            inst.noise_var, inst.ref, 2, L)
    work = torch.empty(S.scoot_fantasy_work_bytes(L, inst.n_cand, 2, box_cap), dtype=torch.uint8, device="cuda")
    idx = torch.empty(2, dtype=torch.int64, device="cuda")
    val = torch.empty(2, device="cuda")
    cnt = torch.empty(1, dtype=torch.int32, device="cuda")
    S.scoot_suggest_fantasy(ctx, L, state, dev(fant), box_cap, dev(inst.cand.view(np.int32)), inst.n_cand,
                            dev(inst.eps), 2, work, idx, val, cnt)
    with pytest.raises(S.ScootError) as e:
        ctx.check()
    assert e.value.status == -1
    assert int(cnt.item()) == 0
