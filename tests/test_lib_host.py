"""The C-ABI library without a GPU: it loads, exports what include/scoot.h
declares, and its host-side preparation agrees with the oracle."""
import ctypes as C
import os
import re

import numpy as np
import pytest

import oracle as O
from workloads import NODE_DTYPE, Stream, make_instance, seeds

from conftest import ROOT


@pytest.fixture(scope="module")
def S():
    import paper_2408_04323_gb300 as pkg
    pkg.build()
    from paper_2408_04323_gb300 import scoot
    scoot.lib()
    return scoot


def _header_functions():
    text = open(os.path.join(ROOT, "include", "scoot.h")).read()
    return sorted(set(re.findall(r"^(?:scoot_status|const char\*)\s+(scoot_\w+)\s*\(", text, re.M)))


def test_library_exports_every_declared_symbol(S):
    names = _header_functions()
    assert len(names) >= 18
    lib = S.lib()
    for name in names:
        assert hasattr(lib, name), name
    assert sorted(S.EXPORTS) == names


def test_status_strings(S):
    assert S.scoot_status_string(0) == "ok"
    assert "unsupported" in S.scoot_status_string(-6)


# ------------------------------------------------------------------ boxes

def _hvi_boxes(y, lo, hi):
    y = np.atleast_2d(y).astype(np.float64)
    ext = np.minimum(y[:, None, :], hi[None].astype(np.float64)) - lo[None].astype(np.float64)
    return np.prod(np.maximum(ext, 0), axis=2).sum(1)


@pytest.mark.parametrize("M,npts", [(2, 1), (2, 12), (3, 9), (3, 30), (4, 7)])
def test_boxes_sum_to_oracle_hvi(S, M, npts):
    st = Stream(100 + M * 7 + npts, "boxes")
    Y = (st.uniform(M * npts).reshape(M, npts) * 4.0).astype(np.float32)
    ref = np.zeros(M, np.float32)
    lo, hi, fs = S.scoot_boxes_build(Y, ref)
    front = O.pareto_front(Y.T, ref)
    assert fs == len(front)
    clo, chi = O.nondominated_cells(front, ref)
    ys = st.uniform(400 * M).reshape(400, M) * 5.0 - 0.5
    assert np.allclose(_hvi_boxes(ys, lo, hi), O.hvi_cells(ys, clo, chi), rtol=1e-12, atol=1e-12)
    # boxes are disjoint: their volumes inside a bounding box plus HV fill it
    box = np.full(M, 6.0)
    inside = np.prod(np.maximum(np.minimum(hi.astype(np.float64), box) - lo, 0), axis=1).sum()
    assert inside + O.hypervolume(front, ref) == pytest.approx(np.prod(box), rel=1e-12)
    if M == 2:
        assert len(lo) == len(front) + 1


def test_boxes_edge_cases(S):
    ref = np.array([0.5, -1.0], np.float32)
    # no point strictly above r: one box [r, +inf)^2
    Y = np.array([[0.5, 3.0], [2.0, -1.0]], np.float32)
    lo, hi, fs = S.scoot_boxes_build(Y, ref)
    assert fs == 0 and len(lo) == 1 and np.allclose(lo[0], ref) and np.all(np.isinf(hi[0]))
    # duplicates count once
    Y = np.array([[1.0, 1.0, 2.0], [1.0, 1.0, 0.0]], np.float32)
    lo, hi, fs = S.scoot_boxes_build(Y, ref)
    assert fs == 2
    # capacity too small: unsupported, count reported
    Y = (Stream(3, "cap").uniform(3 * 20).reshape(3, 20)).astype(np.float32)
    with pytest.raises(S.ScootError) as e:
        S.scoot_boxes_build(Y, np.zeros(3, np.float32), cap=2)
    assert e.value.status == -6
    with pytest.raises(S.ScootError):
        S.scoot_boxes_build(np.array([[np.nan], [1.0]], np.float32), np.zeros(2, np.float32))


def test_boxes_of_the_three_objective_workload_fit(S):
    for seed in seeds("d10-ehvi3"):
        inst = make_instance("d10-ehvi3", seed, n_cand=64)
        lo, hi, fs = S.scoot_boxes_build(inst.y_obs, inst.ref)
        assert len(lo) <= 2000 and fs <= 48


# ------------------------------------------------------------------ GP state

def _unpack_gp(S, L, blob):
    f = lambda off, n: blob[off:off + 4 * n].view(np.float32)
    n, d, M = L.n, L.d, L.n_obj
    alpha = f(L.off_alpha, M * n).reshape(M, n)
    tiles = f(L.off_linv, M * L.n_tiles * 32 * 64).reshape(M, L.n_tiles, 32, 64)
    npad = L.n_rb * 64
    linv = np.zeros((M, npad, npad), np.float32)
    for m in range(M):
        t = 0
        for rb in range(L.n_rb):
            for cj in range(2 * (rb + 1)):
                linv[m, rb * 64:(rb + 1) * 64, cj * 32:(cj + 1) * 32] = tiles[m, t].T
                t += 1
    scal = f(L.off_scal, M * 4).reshape(M, 4)
    src = f(L.off_fmap, d * 4).reshape(d, 4)[:, 3].astype(int)  # feature order -> parameter
    xs = np.zeros((M, n, d), np.float32)
    ils = np.zeros((M, d), np.float32)
    xs[:, :, src] = f(L.off_xs, M * n * d).reshape(M, n, d)
    ils[:, src] = f(L.off_ils, M * d).reshape(M, d)
    return alpha, linv[:, :n, :n], scal, xs, ils, src


@pytest.mark.parametrize("name", ["tiny", "d8-ehvi2", "d10-ei", "d10-ehvi3"])
def test_gp_prepare_matches_oracle_factor(S, name):
    inst = make_instance(name, seeds(name)[0], n_cand=64)
    M, n, d = inst.n_obj, inst.n_obs, inst.d
    L = S.scoot_gp_layout_init(inst.space, n, M)
    blob, cond = S.scoot_gp_prepare(inst.space, inst.x_obs, inst.y_obs, inst.lengthscale,
                                    inst.signal_var, inst.noise_var, L)
    alpha, linv, scal, xs, ils, src = _unpack_gp(S, L, blob)
    kinds = inst.space["kind"][src]
    assert sorted(src.tolist()) == list(range(d))
    assert np.all(np.diff((kinds == 2).astype(int)) >= 0)  # ordinal parameters come first
    for m in range(M):
        gp = O.GP(inst.space, inst.x_obs, inst.y_obs[m], inst.lengthscale[m], inst.signal_var[m], inst.noise_var[m])
        assert np.allclose(alpha[m], gp.alpha, rtol=1e-6, atol=1e-6 * np.abs(gp.alpha).max())
        Li = np.linalg.inv(gp.chol)
        assert np.allclose(linv[m], Li, rtol=1e-6, atol=1e-6 * np.abs(Li).max())
        assert np.all(np.triu(linv[m], 1) == 0)
        assert scal[m, 0] == inst.signal_var[m] and scal[m, 1] == inst.noise_var[m]
        assert scal[m, 2] == inst.y_obs[m].max()
        cat = gp.is_cat
        assert np.allclose(xs[m][:, ~cat], gp.u_obs[:, ~cat] / inst.lengthscale[m][~cat], rtol=1e-6)
        assert np.array_equal(xs[m][:, cat], gp.u_obs[:, cat])
        assert np.allclose(ils[m][cat], 1.0 / inst.lengthscale[m][cat].astype(np.float64) ** 2, rtol=1e-6)
        assert 1.0 <= cond[m] < 1e8


def test_gp_prepare_rejects_bad_inputs(S):
    inst = make_instance("tiny", 1001, n_cand=8)
    M, n, d = inst.n_obj, inst.n_obs, inst.d
    L = S.scoot_gp_layout_init(inst.space, n, M)
    args = [inst.space, inst.x_obs, inst.y_obs, inst.lengthscale, inst.signal_var, inst.noise_var]
    bad_y = inst.y_obs.copy(); bad_y[0, 3] = np.nan
    bad_l = inst.lengthscale.copy(); bad_l[1, 2] = 0.0
    for i, bad in [(2, bad_y), (3, bad_l), (4, np.array([1.0, -1.0], np.float32))]:
        a = list(args); a[i] = bad
        with pytest.raises(S.ScootError) as e:
            S.scoot_gp_prepare(*a, L)
        assert e.value.status == -1
    # duplicated observations without noise: K is singular
    x = np.ascontiguousarray(np.repeat(inst.x_obs[:, :1], n, axis=1))
    with pytest.raises(S.ScootError):
        S.scoot_gp_prepare(inst.space, x, inst.y_obs, inst.lengthscale, inst.signal_var,
                           np.zeros(M, np.float32), L)
    with pytest.raises(S.ScootError):
        S.scoot_gp_layout_init(inst.space, 2000, M)


# ------------------------------------------------------------------ forest

def test_forest_pack_roundtrip_and_validation(S):
    inst = make_instance("d8-ehvi2", seeds("d8-ehvi2")[0], n_cand=8)
    L = S.scoot_forest_layout_init(inst.nodes, inst.tree_offset, inst.d, 255)
    assert L.n_trees == inst.n_trees and L.n_nodes == len(inst.nodes) and L.n_chunks == 1
    blob = S.scoot_forest_pack(L, inst.nodes, inst.tree_offset)
    got = blob[L.off_nodes:L.off_nodes + 8 * L.n_nodes].view(NODE_DTYPE)
    for f in ("val", "feat", "flags"):
        assert np.array_equal(got[f], inst.nodes[f])
    # split nodes point at their left child counted from the chunk's first node (one chunk here)
    base = np.repeat(inst.tree_offset[:-1], np.diff(inst.tree_offset))
    split = (inst.nodes["flags"] & 1) == 0
    assert np.array_equal(got["left"][split].astype(int), (base + inst.nodes["left"].astype(int))[split])

    def bad(mutate, d=inst.d, scale=255):
        nodes = inst.nodes.copy()
        offs = inst.tree_offset.copy()
        mutate(nodes, offs)
        with pytest.raises(S.ScootError) as e:
            S.scoot_forest_layout_init(nodes, offs, d, scale)
        return e.value.status

    split = int(np.nonzero((inst.nodes["flags"] & 1) == 0)[0][0])
    leaf = int(np.nonzero(inst.nodes["flags"] & 1)[0][0])
    assert bad(lambda n, o: n.__setitem__(split, (n[split]["val"], 60000, n[split]["feat"], 0))) == -1
    assert bad(lambda n, o: n.__setitem__(split, (n[split]["val"], 0, n[split]["feat"], 0))) == -1  # cycle
    assert bad(lambda n, o: n.__setitem__(split, (n[split]["val"], n[split]["left"], 40, 0))) == -1
    assert bad(lambda n, o: n.__setitem__(leaf, (2.5, 0, 0, 1))) == -1
    assert bad(lambda n, o: n.__setitem__(leaf, (256.0, 0, 0, 1))) == -1
    assert bad(lambda n, o: n.__setitem__(split, (np.nan, n[split]["left"], n[split]["feat"], 0))) == -1


def test_forest_chunking_of_large_forests(S):
    """A forest larger than one shared-memory chunk is split at tree boundaries."""
    inst = make_instance("d12-fantasy", seeds("d12-fantasy")[0], n_cand=8)
    reps = 4
    nodes = np.concatenate([inst.nodes] * reps)
    sizes = np.diff(inst.tree_offset)
    offs = np.zeros(inst.n_trees * reps + 1, np.int32)
    offs[1:] = np.cumsum(np.tile(sizes, reps))
    L = S.scoot_forest_layout_init(nodes, offs, inst.d, 255)
    assert L.n_chunks >= 2 and L.max_chunk_nodes <= 12288
    blob = S.scoot_forest_pack(L, nodes, offs)
    ch = blob[L.off_chunks:L.off_chunks + 16 * L.n_chunks].view(np.int32).reshape(-1, 4)
    assert ch[:, 1].sum() == inst.n_trees * reps and ch[:, 3].sum() == len(nodes)
    assert np.all(ch[1:, 0] == np.cumsum(ch[:-1, 1]))


@pytest.mark.parametrize("M,npts", [(2, 1), (2, 12), (3, 9), (3, 30), (4, 7)])
def test_boxes_index_reproduces_the_boxes(S, M, npts):
    st = Stream(300 + M * 7 + npts, "boxidx")
    Y = (st.uniform(M * npts).reshape(M, npts) * 4.0).astype(np.float32)
    lo, hi, _ = S.scoot_boxes_build(Y, np.zeros(M, np.float32))
    grid, n_grid, corner = S.scoot_boxes_index(lo, hi)
    for j in range(M):
        g = grid[j, :n_grid[j]]
        assert np.all(np.diff(g) > 0)
        ext = np.concatenate([g, [np.inf]]).astype(np.float32)
        assert np.array_equal(ext[corner[:, j] & 0xFFFF], lo[:, j])
        assert np.array_equal(ext[corner[:, j] >> 16], hi[:, j])
    with pytest.raises(S.ScootError) as e:
        S.scoot_boxes_index(lo, hi, grid_cap=1)
    assert e.value.status == -6
    bad = hi.copy()
    bad[0, 0] = lo[0, 0]
    with pytest.raises(S.ScootError) as e:
        S.scoot_boxes_index(lo, bad)
    assert e.value.status == -1


def test_gp_prepare_warped_matches_oracle(S):
    from workloads import warp_params
    inst = make_instance("d10-ei", seeds("d10-ei")[0], n_cand=64)
    M, n, d = inst.n_obj, inst.n_obs, inst.d
    warp = warp_params("d10-ei", 7)
    L = S.scoot_gp_layout_init(inst.space, n, M, 1)
    blob, _ = S.scoot_gp_prepare_warped(inst.space, inst.x_obs, inst.y_obs, inst.lengthscale, inst.signal_var,
                                        inst.noise_var, warp, L)
    alpha, linv, scal, xs, ils, src = _unpack_gp(S, L, blob)
    gp = O.GP(inst.space, inst.x_obs, inst.y_obs[0], inst.lengthscale[0], inst.signal_var[0], inst.noise_var[0],
              1, warp=warp[0])
    assert np.allclose(alpha[0], gp.alpha, rtol=1e-6, atol=1e-6 * np.abs(gp.alpha).max())
    Li = np.linalg.inv(gp.chol)
    assert np.allclose(linv[0], Li, rtol=1e-6, atol=1e-6 * np.abs(Li).max())
    cat = gp.is_cat
    w = gp.warped(gp.u_obs)
    assert np.allclose(xs[0][:, ~cat], w[:, ~cat] / inst.lengthscale[0][~cat], rtol=1e-6)
    assert scal[0, 3] == 1.0
    wa = blob[L.off_warp:L.off_warp + 8 * d].view(np.float32).reshape(d, 2)
    kinds = inst.space["kind"][src]
    assert np.array_equal(wa[kinds != 2], warp[0][src][kinds != 2]) and np.all(wa[kinds == 2] == 1.0)
    plain, _ = S.scoot_gp_prepare(inst.space, inst.x_obs, inst.y_obs, inst.lengthscale, inst.signal_var,
                                  inst.noise_var, L)
    assert _unpack_gp(S, L, plain)[2][0, 3] == 0.0
    bad = warp.copy()
    bad[0, 0, 1] = 0.0
    with pytest.raises(S.ScootError) as e:
        S.scoot_gp_prepare_warped(inst.space, inst.x_obs, inst.y_obs, inst.lengthscale, inst.signal_var,
                                  inst.noise_var, bad, L)
    assert e.value.status == -1


def test_delta_controller_matches_oracle(S):
    """Algorithm 1's threshold controller in the library against the oracle's
    reading, over a seeded stream of batches."""
    st = Stream(77, "delta")
    d1 = d2 = 0.5
    c1 = c2 = 0
    for step in range(400):
        k = int(st.integers(1, 8, 1)[0])
        bad = bool(st.uniform(1)[0] < 0.3)
        d1, c1 = S.scoot_delta_update(d1, c1, k, bad)
        d2, c2 = O.delta_update(d2, c2, k, bad)
        assert (d1, c1) == (pytest.approx(d2, abs=1e-12), c2), step
        assert 0.25 <= d1 <= 0.75
    with pytest.raises(S.ScootError):
        S.scoot_delta_update(0.5, 0, -1, False)


@pytest.mark.parametrize("name,boxes,warped", [("tiny", 1, False), ("d8-ehvi2", 1, True), ("d10-ei", 0, False),
                                               ("d10-ehvi3", 2, False), ("d12-fantasy", 1, False)])
def test_round_state_build_equals_separate_calls(S, name, boxes, warped):
    """scoot_round_state_build (GP factorisation on the library's host
    threads while the caller packs the forest and builds the boxes) writes
    exactly the bytes of the separate calls, at 256-byte aligned offsets; a
    buffer that is too small is reported with the size needed; without the
    GP part (built on the device) the other parts are unchanged."""
    from workloads import warp_params
    inst = make_instance(name, seeds(name)[0], n_cand=64)
    warp = warp_params(name, seeds(name)[0]) if warped else None
    buf = np.zeros(1 << 22, np.uint8)
    st, out = S.scoot_round_state_build(inst.space, inst.x_obs, inst.y_obs, inst.lengthscale, inst.signal_var,
                                        inst.noise_var, inst.nodes, inst.tree_offset, inst.workload.leaf_scale, buf,
                                        warp=warp, boxes=boxes, h_ref=inst.ref, h_eps=inst.eps)
    L = S.scoot_gp_layout_init(inst.space, inst.n_obs, inst.n_obj, 0)
    if warp is None:
        blob, cond = S.scoot_gp_prepare(inst.space, inst.x_obs, inst.y_obs, inst.lengthscale, inst.signal_var,
                                        inst.noise_var, L)
    else:
        blob, cond = S.scoot_gp_prepare_warped(inst.space, inst.x_obs, inst.y_obs, inst.lengthscale,
                                               inst.signal_var, inst.noise_var, warp, L)
    FL = S.scoot_forest_layout_init(inst.nodes, inst.tree_offset, inst.d, inst.workload.leaf_scale)
    fb = S.scoot_forest_pack(FL, inst.nodes, inst.tree_offset)
    offs = [st.off_gp, st.off_forest] + ([st.off_box_lo, st.off_box_hi] if boxes else [])
    assert all(o % 256 == 0 for o in offs)
    assert bytes(buf[st.off_gp:st.off_gp + L.bytes]) == blob.tobytes()
    assert [st.cond[m] for m in range(inst.n_obj)] == list(cond)
    assert bytes(buf[st.off_forest:st.off_forest + FL.bytes]) == fb.tobytes()
    if boxes:
        lo, hi, fs = S.scoot_boxes_build(inst.y_obs, inst.ref)
        assert st.n_boxes == len(lo) and st.front_size == fs
        assert np.array_equal(buf[st.off_box_lo:st.off_box_lo + lo.nbytes].view(np.float32), lo.ravel())
        assert np.array_equal(buf[st.off_box_hi:st.off_box_hi + hi.nbytes].view(np.float32), hi.ravel())
        if boxes == 1:
            assert np.array_equal(buf[st.off_eps:st.off_eps + inst.eps.nbytes].view(np.float32),
                                  inst.eps.astype(np.float32).ravel())
        else:
            grid, n_grid, corner = S.scoot_boxes_index(lo, hi)
            assert list(st.n_grid[:inst.n_obj]) == list(n_grid)
            assert np.array_equal(buf[st.off_grid:st.off_grid + grid.nbytes].view(np.float32), grid.ravel())
            assert np.array_equal(buf[st.off_corner:st.off_corner + corner.nbytes].view(np.uint32), corner.ravel())
    small = np.zeros(512, np.uint8)
    none, need = S.scoot_round_state_build(inst.space, inst.x_obs, inst.y_obs, inst.lengthscale, inst.signal_var,
                                           inst.noise_var, inst.nodes, inst.tree_offset, inst.workload.leaf_scale,
                                           small, warp=warp, boxes=boxes, h_ref=inst.ref, h_eps=inst.eps)
    assert none is None and need.bytes == st.bytes
    buf2 = np.zeros(1 << 22, np.uint8)
    st2, _ = S.scoot_round_state_build(inst.space, inst.x_obs, inst.y_obs, inst.lengthscale, inst.signal_var,
                                       inst.noise_var, inst.nodes, inst.tree_offset, inst.workload.leaf_scale, buf2,
                                       warp=warp, boxes=boxes, h_ref=inst.ref, h_eps=inst.eps, gp_on_device=True)
    assert st2.off_gp == -1 and st2.off_forest == 0
    assert bytes(buf2[:FL.bytes]) == fb.tobytes()


def test_round_state_build_concurrent_callers(S):
    """Several host threads building round states at once share the
    library's thread pool (the GP objectives and the forest's packing run on
    it, nested): every result equals the single-threaded one."""
    import threading
    names = ["d8-ehvi2", "d10-ei", "tiny", "d10-ehvi3"]
    insts = [make_instance(nm, seeds(nm)[0], n_cand=16) for nm in names]
    boxes = [1, 0, 1, 2]

    def build(inst, bx):
        buf = np.zeros(1 << 21, np.uint8)
        st, _ = S.scoot_round_state_build(inst.space, inst.x_obs, inst.y_obs, inst.lengthscale, inst.signal_var,
                                          inst.noise_var, inst.nodes, inst.tree_offset, inst.workload.leaf_scale,
                                          buf, boxes=bx, h_ref=inst.ref, h_eps=inst.eps)
        return bytes(buf[:st.bytes])

    want = [build(i, b) for i, b in zip(insts, boxes)]
    errors = []

    def worker(k):
        try:
            for r in range(12):
                j = (k + r) % len(insts)
                if build(insts[j], boxes[j]) != want[j]:
                    errors.append((k, r, j))
        except Exception as e:  # reported below
            errors.append(repr(e))

    threads = [threading.Thread(target=worker, args=(k,)) for k in range(6)]
    for t in threads:
        t.start()
    for t in threads:
        t.join()
    assert not errors, errors[:5]


def test_scratch_sizes_and_buffer_layout(S):
    """Host-only sizing calls of the device builders: their documented
    formulas, 16-byte (256-byte) alignment, and rejection of bad input."""
    inst = make_instance("d8-ehvi2", seeds("d8-ehvi2")[0], n_cand=16)
    for n in (1, 64, 160, 161, 640):
        L = S.scoot_gp_layout_init(inst.space, n, 2, 0)
        tri = n * (n + 1) // 2
        want = 8 * 2 * (n * inst.d + tri * (1 if n <= 160 else 2))
        assert S.scoot_gp_device_work_bytes(L) == want
        for warped in (False, True):
            up, blob, work, total = S.scoot_gp_device_buffer_layout(L, warped)
            assert up % 256 == 0 and blob % 256 == 0 and work % 256 == 0 and total % 256 == 0
            assert up <= blob and blob + L.bytes <= work and work + want <= total
            need = 4 * inst.d * n + 4 * 2 * n + 4 * 2 * inst.d + 8 + (8 * 2 * inst.d if warped else 0)
            assert up >= need
    assert S.scoot_rf_train_work_bytes(256, 12) == 2 * 256 * 12
    assert S.scoot_rf_train_work_bytes(7, 3) == 48  # 42 rounded up to 16
    tri = 200 * 201 // 2
    base = (200 * 10 * 8 + 255) // 256 * 256
    assert S.scoot_gp_mle_work_bytes(200, 10, 3, 32) == base + 32 * 3 * 2 * tri * 8
    assert S.scoot_gp_mle_work_bytes(128, 10, 1, 64) == (128 * 10 * 8 + 255) // 256 * 256
    for bad in [(0, 10, 1, 1), (10, 0, 1, 1), (10, 10, 0, 1), (10, 10, 1, 0)]:
        with pytest.raises(S.ScootError):
            S.scoot_gp_mle_work_bytes(*bad)
    with pytest.raises(S.ScootError):
        S.scoot_rf_train_work_bytes(0, 3)


@pytest.mark.parametrize("name,q", [("d12-fantasy", 16), ("d8-ehvi2", 4), ("d10-ehvi3", 3)])
def test_fantasy_state_holds_the_fp64_factorisation(S, name, q):
    """The fantasy state: header, space, features, lengthscales, alpha and
    L^{-1} in fp64 (L L^T = K + tau^2 I of the oracle's GP), the front of the
    observations above r (the oracle's pareto_front) and the box bound
    (front + q + 1)^(M - 1); the round-state builder writes the same bytes."""
    inst = make_instance(name, seeds(name)[0], n_cand=8)
    M, n, d = inst.n_obj, inst.n_obs, inst.d
    G = S.scoot_gp_layout_init(inst.space, n, M)
    st, box_cap = S.scoot_fantasy_prepare(inst.space, inst.x_obs, inst.y_obs, inst.lengthscale, inst.signal_var,
                                          inst.noise_var, inst.ref, q, G)
    hdr = st[:64].view(np.int32)
    magic, hn, hd, hM, kern, hq, front0, front_cap, hbox = hdr[:9]
    assert magic == 0x544e4146 and (hn, hd, hM, kern, hq) == (n, d, M, 0, q)
    front = O.pareto_front(inst.y_obs.T.astype(np.float64), inst.ref.astype(np.float64))
    assert front0 == len(front) and front_cap == len(front) + q
    assert hbox == box_cap == min((len(front) + q + 1) ** (M - 1), 6144)
    offs = st[160:216].view(np.int64)
    off_space, off_u, off_ell, off_alpha, off_linv, off_front, nbytes = offs
    assert nbytes == S.scoot_fantasy_state_bytes(G, q) == len(st)
    dbl = lambda off, cnt: st[off:off + 8 * cnt].view(np.float64)
    sp = dbl(off_space, 4 * d).reshape(d, 4)
    assert np.array_equal(sp[:, 0], inst.space["kind"]) and np.array_equal(sp[:, 1], inst.space["lo"].astype(np.float64))
    fr = dbl(off_front, front0 * M).reshape(front0, M)
    assert np.array_equal(np.array(sorted(map(tuple, fr))), np.array(sorted(map(tuple, front))))
    for m in range(M):
        gp = O.GP(inst.space, inst.x_obs, inst.y_obs[m], inst.lengthscale[m], inst.signal_var[m], inst.noise_var[m])
        assert np.allclose(dbl(off_u, n * d).reshape(n, d), gp.u_obs, rtol=1e-14, atol=1e-14)
        assert np.array_equal(dbl(off_ell + 8 * m * d, d), inst.lengthscale[m].astype(np.float64))
        alpha = dbl(off_alpha + 8 * m * n, n)
        assert np.allclose(alpha, gp.alpha, rtol=1e-9, atol=1e-10 * np.abs(gp.alpha).max())
        Li = dbl(off_linv + 8 * m * n * n, n * n).reshape(n, n).T  # column-major
        assert np.allclose(np.tril(Li), Li)
        assert np.allclose(Li @ gp.chol, np.eye(n), atol=1e-8)
    # the round-state builder writes the same fantasy state from its own factorisation
    buf = np.zeros(64 << 20, np.uint8)
    out, _ = S.scoot_round_state_build(inst.space, inst.x_obs, inst.y_obs, inst.lengthscale, inst.signal_var,
                                       inst.noise_var, inst.nodes, inst.tree_offset, inst.workload.leaf_scale, buf,
                                       boxes=1, h_ref=inst.ref, h_eps=inst.eps, fantasy_q=q)
    assert out.off_fant >= 0 and out.off_fant % 256 == 0 and out.fant_box_cap == box_cap
    assert np.array_equal(buf[out.off_fant:out.off_fant + len(st)], st)


def test_ucb_beta_is_the_printed_schedule(S):
    """beta_t = 2 log(t^2 pi^2 / (6 delta)) with delta = 1/t^2 (Section 4.5)
    = 2 log(pi^2 t^4 / 6): 0.994... at t = 1, growing like 8 log t."""
    import math
    for t in (1, 2, 16, 128, 1000):
        assert S.scoot_ucb_beta(t) == pytest.approx(2.0 * math.log(math.pi ** 2 * t ** 4 / 6.0), rel=1e-14)
    assert S.scoot_ucb_beta(1) == pytest.approx(2.0 * math.log(math.pi ** 2 / 6.0), rel=1e-14)
    assert S.scoot_ucb_beta(20) - S.scoot_ucb_beta(10) == pytest.approx(8.0 * math.log(2.0), rel=1e-12)
    with pytest.raises(S.ScootError):
        S.scoot_ucb_beta(0)


def test_standardize_gives_zero_mean_unit_sd_and_a_reference_below(S):
    y = (Stream(41, "std").normal(3 * 50).reshape(3, 50) * [[3.0], [0.01], [100.0]] + [[5.0], [-2.0], [1e3]])
    y = y.astype(np.float32)
    z, ref = S.scoot_standardize(y, ref_margin=1e-3)
    assert np.allclose(z.astype(np.float64).mean(axis=1), 0.0, atol=1e-6)
    assert np.allclose(z.astype(np.float64).std(axis=1), 1.0, atol=1e-6)
    assert np.all(ref < z.min(axis=1)) and np.allclose(ref, z.min(axis=1) - 1e-3, atol=1e-7)
    # invariant to an affine change of units
    z2, _ = S.scoot_standardize((y.astype(np.float64) * 7.0 - 3.0).astype(np.float32))
    assert np.allclose(z, z2, atol=1e-4)  # up to the fp32 rounding of the rescaled inputs
    # a constant objective stays finite (the floor of the standard deviation)
    z3, _ = S.scoot_standardize(np.ones((1, 5), np.float32))
    assert np.all(z3 == 0.0)
    bad = y.copy()
    bad[1, 3] = np.nan
    with pytest.raises(S.ScootError):
        S.scoot_standardize(bad)
