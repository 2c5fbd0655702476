"""The GP state built on the device (fp64 factorisation with L^{-1} from the
elimination of the identity), through the C ABI.

Parity: the posterior computed from the device-built state meets the same
bars against the oracle as the host-built state (variance 1e-6 + 1e-4 |o|;
mean plus 2^-22 sum_j |k_j alpha_j|), on every workload, both kernels, with
and without input warping, on both sides of the shared-memory limit of the
factorisation (n = 160 / 161) and at n = 1 and the maximum, n = 640.  Consistency: the
tables that involve no factorisation (feature map, scaled features, inverse
lengthscales, scalars, warping, categorical table) equal the host's to one
fp32 rounding of an fp64 value; alpha and L^{-1} agree with the host's to
the fp64 rounding of two different factorisation orders, amplified by the
conditioning: within 1e-6 of the largest entry (measured: identical fp32
values up to n = 160, 5e-10 at n = 1024).
"""
import numpy as np
import pytest

import oracle as O
from workloads import Stream, make_instance, seeds, warp_params

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from parity_tol import ATOL, MU_COND, RTOL  # noqa: E402


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


def device_blob(S, ctx, inst, L, warp=None, x_obs=None, y=None):
    x = inst.x_obs if x_obs is None else x_obs
    yy = inst.y_obs if y is None else y
    blob = torch.full((L.bytes,), 0xAB, dtype=torch.uint8, device="cuda")
    S.scoot_gp_prepare_device(ctx, inst.space, L, dev(np.ascontiguousarray(x).view(np.int32)),
                              dev(yy.astype(np.float32)), dev(inst.lengthscale.astype(np.float32)),
                              dev(inst.signal_var.astype(np.float32)), dev(inst.noise_var.astype(np.float32)),
                              blob, warp=None if warp is None else dev(warp.astype(np.float32)))
    ctx.check()
    return blob


def host_blob(S, inst, L, warp=None):
    if warp is None:
        b, _ = S.scoot_gp_prepare(inst.space, inst.x_obs, inst.y_obs, inst.lengthscale, inst.signal_var,
                                  inst.noise_var, L)
    else:
        b, _ = S.scoot_gp_prepare_warped(inst.space, inst.x_obs, inst.y_obs, inst.lengthscale, inst.signal_var,
                                         inst.noise_var, warp, L)
    return b


def region(blob, off, count):
    return np.frombuffer(blob, np.float32, count, off)


def compare_tables(L, hb, db, name):
    """Tables with no factorisation in them: one fp32 rounding of fp64 values."""
    M, n, d = L.n_obj, L.n, L.d
    for label, off, cnt in [("fmap", L.off_fmap, d * 4), ("xs", L.off_xs, M * n * d), ("ils", L.off_ils, M * d),
                            ("scal", L.off_scal, M * 4), ("cat", L.off_cat, M * n * L.n_pat),
                            ("warp", L.off_warp, M * d * 2)]:
        h, g = region(hb, off, cnt), region(db, off, cnt)
        err = np.abs(g.astype(np.float64) - h) / np.maximum(np.abs(h), 1e-30)
        assert np.all((g == h) | (err <= 2.0 ** -23)), f"{name} {label}: max rel {err.max():.3e}"
    # alpha and L^{-1}: the same quantities from two fp64 factorisation orders
    ah = region(hb, L.off_alpha, M * n).astype(np.float64)
    ag = region(db, L.off_alpha, M * n).astype(np.float64)
    nt = L.n_tiles * 32 * 64
    th = region(hb, L.off_linv, M * nt).astype(np.float64)
    tg = region(db, L.off_linv, M * nt).astype(np.float64)
    ea = np.abs(ag - ah).max() / max(np.abs(ah).max(), 1e-30)
    et = np.abs(tg - th).max() / max(np.abs(th).max(), 1e-30)
    print(f"[parity] {name}: alpha max rel-to-max diff {ea:.2e}, L^-1 {et:.2e}")
    assert np.array_equal(th == 0, tg == 0)  # same zero pattern (triangle and padding)
    assert ea <= 1e-6 and et <= 1e-6
    return ea, et


def posterior_check(S, ctx, inst, L, state, name, kernel=0, warp=None, n_cand=2048 + 19):
    M = inst.n_obj
    cand = dev(inst.cand.view(np.int32))
    n = min(n_cand, inst.n_cand)
    mean = torch.zeros((M, n), device="cuda")
    var = torch.zeros((M, n), device="cuda")
    S.scoot_gp_posterior(ctx, L, state, cand, n, mean, var)
    torch.cuda.synchronize()
    gm, gv = mean.cpu().numpy(), var.cpu().numpy()
    worst = 0.0
    for m in range(M):
        gp = O.GP(inst.space, inst.x_obs, inst.y_obs[m], inst.lengthscale[m], inst.signal_var[m],
                  inst.noise_var[m], kernel, warp=None if warp is None else warp[m])
        mu, v = gp.posterior(inst.cand, n)
        cond = gp.mean_condition(inst.cand, n)
        r_mu = np.abs(gm[m] - mu) / (ATOL + RTOL * np.abs(mu) + MU_COND * cond)
        r_v = np.abs(gv[m] - v) / (ATOL + RTOL * np.abs(v))
        worst = max(worst, float(r_mu.max()), float(r_v.max()))
        assert r_mu.max() <= 1.0 and r_v.max() <= 1.0, f"{name} objective {m}: mu {r_mu.max():.3f} var {r_v.max():.3f}"
    print(f"[parity] {name}: posterior from the device-built state, max |err|/tol = {worst:.3f}")


@pytest.mark.parametrize("name,kernel,warped", [("tiny", 0, False), ("d8-ehvi2", 0, False), ("d8-ehvi2", 1, True),
                                                ("d10-ei", 0, False), ("d10-ei", 1, True), ("d10-ehvi3", 0, False),
                                                ("d12-fantasy", 0, False)])
def test_device_state_matches(S, ctx, name, kernel, warped):
    inst = make_instance(name, seeds(name)[1], n_cand=4096)
    L = S.scoot_gp_layout_init(inst.space, inst.n_obs, inst.n_obj, kernel)
    warp = warp_params(name, seeds(name)[1]) if warped else None
    db = device_blob(S, ctx, inst, L, warp)
    hb = host_blob(S, inst, L, warp)
    compare_tables(L, hb, db.cpu().numpy().tobytes(), name)
    posterior_check(S, ctx, inst, L, db, f"{name} k{kernel}{' warped' if warped else ''}", kernel, warp)


@pytest.mark.parametrize("n_obs", [1, 2, 7, 63, 64, 65, 160, 161, 384, 385, 640])
def test_device_state_sizes(S, ctx, n_obs):
    """Observation counts across tile edges, the shared-memory limit of the
    factorisation (160 / 161), the cluster path's limit (384 / 385) and the maximum; the d8
    space, two objectives."""
    base = make_instance("d8-ehvi2", seeds("d8-ehvi2")[0], n_cand=4096)
    from workloads.generate import draw_configs
    w = base.workload
    st = Stream(n_obs, "gp-device-sizes")
    x = draw_configs(w, st, n_obs)
    y = st.normal(w.n_obj * n_obs).reshape(w.n_obj, n_obs).astype(np.float32)

    class Inst:
        pass
    inst = Inst()
    inst.space, inst.x_obs, inst.y_obs = base.space, x, y
    inst.lengthscale, inst.signal_var = base.lengthscale, base.signal_var
    inst.noise_var = np.maximum(base.noise_var, np.float32(1e-3))
    inst.n_obs, inst.n_obj, inst.cand, inst.n_cand = n_obs, w.n_obj, base.cand, base.n_cand
    L = S.scoot_gp_layout_init(inst.space, n_obs, inst.n_obj, 0)
    db = device_blob(S, ctx, inst, L)
    hb = host_blob(S, inst, L)
    compare_tables(L, hb, db.cpu().numpy().tobytes(), f"n={n_obs}")
    posterior_check(S, ctx, inst, L, db, f"n={n_obs}", n_cand=1024 if n_obs > 256 else 2048 + 19)


def test_device_state_rejects_bad_inputs(S, ctx):
    """A NaN observation value, a non-positive lengthscale and a singular
    matrix (two identical observations, no noise) are reported by
    scoot_ctx_check as SCOOT_EINVAL; the context stays usable."""
    inst = make_instance("d8-ehvi2", seeds("d8-ehvi2")[0], n_cand=4096)
    L = S.scoot_gp_layout_init(inst.space, inst.n_obs, inst.n_obj, 0)
    blob = torch.zeros(L.bytes, dtype=torch.uint8, device="cuda")
    args = [dev(inst.x_obs.view(np.int32)), None, dev(inst.lengthscale.astype(np.float32)),
            dev(inst.signal_var.astype(np.float32)), dev(inst.noise_var.astype(np.float32)), blob]

    def run(y=None, ls=None, x=None, tau=None):
        a = list(args)
        a[1] = dev((inst.y_obs if y is None else y).astype(np.float32))
        if ls is not None:
            a[2] = dev(ls.astype(np.float32))
        if x is not None:
            a[0] = dev(x.view(np.int32))
        if tau is not None:
            a[4] = dev(tau.astype(np.float32))
        S.scoot_gp_prepare_device(ctx, inst.space, L, *a)
        with pytest.raises(S.ScootError) as e:
            ctx.check()
        assert e.value.status == -1

    y = inst.y_obs.copy()
    y[1, 5] = np.nan
    run(y=y)
    ls = inst.lengthscale.copy()
    ls[0, 2] = 0.0
    run(ls=ls)
    x = inst.x_obs.copy()
    x[:, 1] = x[:, 0]
    run(x=x, tau=np.zeros(inst.n_obj))
    device_blob(S, ctx, inst, L)  # still usable afterwards


@pytest.mark.parametrize("name", ["d8-ehvi2", "d10-ei"])
def test_round_with_device_state(S, ctx, name):
    """A whole round whose GP state the device builds picks the same
    candidates, with the same values, as the round with the host-built
    state (the two states' L^{-1} and alpha agree to fp32 rounding)."""
    from paper_2408_04323_gb300.pipeline import RoundInputs, ScoringRound
    inst = make_instance(name, seeds(name)[0], n_cand=1 << 16)
    w = inst.workload
    inp = RoundInputs(inst.space, inst.clauses, inst.nodes, inst.tree_offset, w.leaf_scale, w.delta_num,
                      w.delta_den, inst.x_obs, inst.y_obs, inst.lengthscale, inst.signal_var, inst.noise_var,
                      inst.ref, inst.eps, w.acq, w.q)
    cand = dev(inst.cand.view(np.int32))
    out = []
    for on_dev in (False, True):
        rnd = ScoringRound(ctx, inp, inst.n_cand, gp_on_device=on_dev)
        rnd.run(cand, inst.n_cand)
        torch.cuda.synchronize()
        ctx.check()
        c = int(rnd.top_count.cpu()[0])
        out.append((rnd.top_idx.cpu().numpy()[:c], rnd.top_val.cpu().numpy()[:c]))
    (ih, vh), (id_, vd) = out
    assert len(ih) == w.q and np.array_equal(ih, id_)
    assert np.allclose(vd, vh, rtol=1e-5, atol=1e-7)


@pytest.mark.parametrize("name,warped", [("d8-ehvi2", False), ("d8-ehvi2", True), ("d12-fantasy", False)])
def test_device_state_from_host_inputs(S, ctx, name, warped):
    """The one-call path (host inputs packed into pinned memory, copied and
    built on the device) writes the same blob as scoot_gp_prepare_device fed
    the same inputs from device memory."""
    inst = make_instance(name, seeds(name)[0], n_cand=16)
    L = S.scoot_gp_layout_init(inst.space, inst.n_obs, inst.n_obj, 0)
    warp = warp_params(name, seeds(name)[0]) if warped else None
    want = device_blob(S, ctx, inst, L, warp).cpu().numpy()
    up, blob_off, work_off, total = S.scoot_gp_device_buffer_layout(L, warped)
    assert blob_off >= up and work_off >= blob_off + L.bytes and total >= work_off
    buf = torch.full((total,), 0xCD, dtype=torch.uint8, device="cuda")
    stage = torch.empty(up, dtype=torch.uint8, pin_memory=True)
    S.scoot_gp_prepare_device_from_host(ctx, inst.space, L, np.ascontiguousarray(inst.x_obs),
                                        inst.y_obs.astype(np.float32), inst.lengthscale.astype(np.float32),
                                        inst.signal_var.astype(np.float32), inst.noise_var.astype(np.float32),
                                        stage, buf, warp=None if warp is None else warp.astype(np.float32))
    torch.cuda.synchronize()
    ctx.check()
    got = buf[blob_off:blob_off + L.bytes].cpu().numpy()
    # the regions the posterior reads (padding between regions is not written)
    for off, cnt in [(L.off_fmap, L.d * 4), (L.off_xs, L.n_obj * L.n * L.d), (L.off_ils, L.n_obj * L.d),
                     (L.off_alpha, L.n_obj * L.n), (L.off_linv, L.n_obj * L.n_tiles * 32 * 64),
                     (L.off_scal, L.n_obj * 4), (L.off_cat, L.n_obj * L.n * L.n_pat), (L.off_warp, L.n_obj * L.d * 2)]:
        assert np.array_equal(got[off:off + 4 * cnt], want[off:off + 4 * cnt]), off
