"""Sequential fantasised picks (the q = 16 parallel-suggestion workload):
the GPU's rank-1 downdates against the oracle's refit of the GP with the
picked points appended, pick by pick.

Small pools are compared with the oracle's own pick sequence over the whole
pool.  Large pools (2^18, and the full 2^22 round of the benchmark) replay the
GPU's picks in the oracle (forced replay) evaluated on a seeded sample of the
live candidates plus the picks: at every step the GPU's pick value must be
the oracle's value there, and no sampled candidate may beat the pick by more
than the two values' tolerances."""
import numpy as np
import pytest

import oracle as O
from workloads import Stream, make_instance, seeds

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from parity_tol import ATOL, RTOL, posterior_tols, propagated_tol  # noqa: E402


@pytest.fixture(scope="module")
def S():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2408_04323_gb300 as pkg
    pkg.build()
    from paper_2408_04323_gb300 import scoot
    return scoot


def _round_inputs(S, inst, q):
    """Device pool, GP blob, fantasy state and base samples of an instance."""
    w = inst.workload
    G = S.scoot_gp_layout_init(inst.space, inst.n_obs, inst.n_obj)
    blob, _ = S.scoot_gp_prepare(inst.space, inst.x_obs, inst.y_obs, inst.lengthscale, inst.signal_var,
                                 inst.noise_var, G)
    fant, box_cap = S.scoot_fantasy_prepare(inst.space, inst.x_obs, inst.y_obs, inst.lengthscale, inst.signal_var,
                                            inst.noise_var, inst.ref, q, G)
    L = S.scoot_forest_layout_init(inst.nodes, inst.tree_offset, inst.d, w.leaf_scale)
    forest = torch.from_numpy(S.scoot_forest_pack(L, inst.nodes, inst.tree_offset)).cuda()
    return dict(G=G, state=torch.from_numpy(blob).cuda(), fant=torch.from_numpy(fant).cuda(), box_cap=box_cap,
                L=L, forest=forest, eps=torch.from_numpy(inst.eps).cuda(),
                cand=torch.from_numpy(inst.cand.view(np.int32)).cuda())


def _outputs(q):
    return (torch.full((q,), -7, dtype=torch.int64, device="cuda"), torch.full((q,), 7.0, device="cuda"),
            torch.full((1,), -7, dtype=torch.int32, device="cuda"))


def _gpu_round(S, ctx, inst, q, n, r, var_out=None, stream=None):
    """prune -> forest -> q fantasised picks through the C ABI."""
    w = inst.workload
    mask = torch.empty(n, dtype=torch.uint8, device="cuda")
    votes = torch.empty(n, dtype=torch.int32, device="cuda")
    S.scoot_prune(ctx, inst.space, inst.clauses, r["cand"], n, mask, stream=stream)
    S.scoot_rf_predict(ctx, r["L"], r["forest"], inst.space, r["cand"], n, w.delta_num, w.delta_den, votes, mask,
                       stream=stream)
    work = torch.empty(S.scoot_fantasy_work_bytes(r["G"], n, q, r["box_cap"]), dtype=torch.uint8, device="cuda")
    idx, val, cnt = _outputs(q)
    S.scoot_suggest_fantasy(ctx, r["G"], r["state"], r["fant"], r["box_cap"], r["cand"], n, r["eps"], q, work, idx,
                            val, cnt, mask=mask, var_out=var_out, stream=stream)
    return mask, work, idx, val, cnt


def _oracle_feasible(inst, n, idx=None):
    w = inst.workload
    words = inst.cand if idx is None else np.ascontiguousarray(inst.cand[:, idx])
    m = n if idx is None else len(idx)
    known = O.prune_mask(inst.space, inst.clauses, words, m)
    v = O.rf_votes(inst.nodes, inst.tree_offset, inst.space, words, m)
    return known & O.pof_feasible(v, inst.n_trees, w.leaf_scale, w.delta_num, w.delta_den)


def _tol_at(inst, ref, gps, j, ks):
    """The oracle's step-j EHVI at evaluated positions ks and its tolerance
    (the stated bar plus the propagated posterior tolerance)."""
    sel = ref["index"]
    _, _, e_mu, _ = posterior_tols(gps, np.ascontiguousarray(inst.cand[:, sel[ks]]))
    mu = ref["mu"][j][ks]
    var = ref["var"][j][ks]
    f = lambda a_, b_: O.ehvi_mc(a_, b_, inst.eps, ref["fronts"][j], inst.ref)
    return propagated_tol(f, mu, var, e_mu, ATOL + RTOL * var)


@pytest.mark.parametrize("seed_i,n,q,tc", [(0, 2048, 16, 1), (1, 1500, 6, 1), (0, 2048, 16, 0)],
                         ids=["2048-q16-tensor", "1500-q6-tensor", "2048-q16-simt"])
def test_fantasy_picks_follow_the_refit_oracle(S, seed_i, n, q, tc):
    """tc: the whitened posterior's L^{-1} k product on the tensor cores or in
    fp32 SIMT (both write the tiled rows of V the passes read)."""
    name = "d12-fantasy"
    inst = make_instance(name, seeds(name)[seed_i], n_cand=n)
    ctx = S.Context(0)
    S.scoot_ctx_set_tensor_cores(ctx, tc)
    try:
        r = _round_inputs(S, inst, q)
        var_out = torch.full((inst.n_obj, n), -1.0, device="cuda")
        mask, _, idx, val, cnt = _gpu_round(S, ctx, inst, q, n, r, var_out=var_out)
        ctx.check()
        feas_gpu = mask.cpu().numpy().astype(bool)
        c = int(cnt.item())
        idx = idx.cpu().numpy()[:c]
        val = val.cpu().numpy()[:c]
    finally:
        ctx.close()
    feas = _oracle_feasible(inst, n)
    assert np.array_equal(feas_gpu, feas)
    ref = O.fantasy_picks(inst, q, feas)
    assert len(idx) == len(ref["picks"]) == min(q, int(feas.sum()))
    gps = [O.GP(inst.space, inst.x_obs, inst.y_obs[m], inst.lengthscale[m], inst.signal_var[m],
                inst.noise_var[m]) for m in range(inst.n_obj)]
    same = 0
    for j, (g, o) in enumerate(zip(idx.tolist(), ref["picks"])):
        want_g, tol_g = _tol_at(inst, ref, gps, j, [g])
        print(f"[fantasy] pick {j}: gpu {g} ({val[j]:.7g}) oracle {o} ({ref['acq'][j][o]:.7g}) "
              f"|err|/tol={abs(float(val[j]) - want_g[0]) / tol_g[0]:.3f}")
        # the GPU's value at its pick is the oracle's value there, within tolerance
        assert abs(float(val[j]) - want_g[0]) <= tol_g[0]
        if g != o:
            # a different pick is only allowed on a near-tie of the oracle's values
            want_o, tol_o = _tol_at(inst, ref, gps, j, [o])
            assert want_g[0] >= want_o[0] - tol_g[0] - tol_o[0]
            break
        same += 1
    print(f"[fantasy] {same} of {len(idx)} picks identical")
    if same == len(idx) and len(idx) > 1:
        # variances after the downdates of picks 0 .. q-2, against the refit
        gv = var_out.cpu().numpy().astype(np.float64)[:, feas].T
        ov = ref["var"][-1][feas]
        err = np.abs(gv - ov) / (ATOL + RTOL * np.abs(ov))
        print(f"[fantasy] variance after {len(idx) - 1} fantasies: max|err|/tol={err.max():.3f} "
              f"max|err|={np.abs(gv - ov).max():.3e}")
        assert err.max() <= 1.0


def _forced_replay_check(inst, n, feas_sample_idx, idx, val, var_s, q, label):
    """Forced replay of the GPU's picks in the oracle at a sample of live
    candidates plus the picks; see the module docstring."""
    feas = np.zeros(n, bool)
    feas[feas_sample_idx] = True
    feas[idx] = True
    ref = O.fantasy_picks(inst, q, feas, forced=idx.tolist(), subset=feas_sample_idx)
    sel = ref["index"]
    where = {int(i): k for k, i in enumerate(sel)}
    gps = [O.GP(inst.space, inst.x_obs, inst.y_obs[m], inst.lengthscale[m], inst.signal_var[m],
                inst.noise_var[m]) for m in range(inst.n_obj)]
    worst_val = worst_beat = 0.0
    for j, g in enumerate(idx.tolist()):
        ks = np.nonzero(np.isfinite(ref["acq"][j]))[0]
        want, tol = _tol_at(inst, ref, gps, j, ks)
        kg = int(np.nonzero(ks == where[g])[0][0])
        r = abs(float(val[j]) - want[kg]) / tol[kg]
        worst_val = max(worst_val, r)
        assert r <= 1.0, (label, j, g, float(val[j]), want[kg], tol[kg])
        # no sampled candidate beats the pick by more than the two tolerances
        beat = (want - want[kg]) / (tol + tol[kg])
        worst_beat = max(worst_beat, float(beat.max()))
        assert beat.max() <= 1.0, (label, j, int(sel[ks[int(np.argmax(beat))]]))
    # variances after the q - 1 downdates at the sampled candidates
    if var_s is not None and len(idx) == q:
        ov = ref["var"][-1]
        ks = np.array([where[int(i)] for i in feas_sample_idx])
        err = np.abs(var_s.T - ov[ks]) / (ATOL + RTOL * np.abs(ov[ks]))
        print(f"[fantasy] {label}: variance after {q - 1} fantasies at {len(ks)} samples: "
              f"max|err|/tol={err.max():.3f}")
        assert err.max() <= 1.0
    print(f"[fantasy] {label}: {len(idx)} picks, max |val err|/tol={worst_val:.3f}, "
          f"max beat/tol={worst_beat:.3f} over {len(sel)} evaluated candidates")


def test_fantasy_forced_replay_at_2_18(S):
    """q = 16 picks over a 2^18 pool (several thousand tiles of the whitened
    posterior, full boxes of the workload), replayed in the oracle."""
    name, n, q = "d12-fantasy", 1 << 18, 16
    inst = make_instance(name, seeds(name)[0], n_cand=n)
    ctx = S.Context(0)
    try:
        r = _round_inputs(S, inst, q)
        var_out = torch.full((inst.n_obj, n), -1.0, device="cuda")
        mask, _, idx, val, cnt = _gpu_round(S, ctx, inst, q, n, r, var_out=var_out)
        ctx.check()
        c = int(cnt.item())
        assert c == q
        idx = idx.cpu().numpy()[:c]
        val = val.cpu().numpy()[:c]
        live = np.nonzero(mask.cpu().numpy())[0]
        st = Stream(9001, "fantasy-sample")
        samp = np.unique(live[(st.u64(1500) % np.uint64(len(live))).astype(np.int64)])
        var_s = var_out[:, torch.from_numpy(samp).cuda()].cpu().numpy().astype(np.float64)
    finally:
        ctx.close()
    # feasibility of the sample and the picks, against the oracle
    chk = np.concatenate([samp, idx])
    assert np.all(_oracle_feasible(inst, n, chk))
    _forced_replay_check(inst, n, samp, idx, val, var_s, q, "2^18")


def test_fantasy_round_at_bench_size_gate_b(S):
    """Gate B of the 2^22-candidate fantasy round in the benchmark's launch
    configuration (ScoringRound, one stream): masks bit-exact on a sample,
    the 16 picks validated by forced replay on a sample of live candidates."""
    from paper_2408_04323_gb300.pipeline import RoundInputs, ScoringRound
    name = "d12-fantasy"
    inst = make_instance(name, seeds(name)[0])
    w = inst.workload
    n = inst.n_cand
    inp = RoundInputs(inst.space, inst.clauses, inst.nodes, inst.tree_offset, w.leaf_scale, w.delta_num,
                      w.delta_den, inst.x_obs, inst.y_obs, inst.lengthscale, inst.signal_var, inst.noise_var,
                      inst.ref, inst.eps, w.acq, w.q, fantasy=True)
    ctx = S.Context(0)
    try:
        rnd = ScoringRound(ctx, inp, n)
        cand = torch.from_numpy(inst.cand.view(np.int32)).cuda()
        idx, val, cnt = rnd.run(cand, n)
        ctx.check()
        c = int(cnt.item())
        idx = idx.cpu().numpy()[:c]
        val = val.cpu().numpy()[:c]
        mask = rnd.mask.cpu().numpy().astype(bool)
    finally:
        ctx.close()
    assert c == w.q
    st = Stream(9002, "gate-b-sample")
    probe = (st.u64(1 << 15) % np.uint64(n)).astype(np.int64)
    assert np.array_equal(mask[probe], _oracle_feasible(inst, n, probe))
    assert np.array_equal(mask, O.prune_mask(inst.space, inst.clauses, inst.cand, n) & mask)
    live = np.nonzero(mask)[0]
    samp = np.unique(live[(st.u64(600) % np.uint64(len(live))).astype(np.int64)])
    _forced_replay_check(inst, n, samp, idx, val, None, w.q, "2^22 round")


def test_fantasy_call_replays_as_a_cuda_graph(S):
    """The whole call runs in stream order with no host synchronisation: it
    captures into a CUDA graph whose replays give the eager call's picks."""
    name, n, q = "d12-fantasy", 20000, 8
    inst = make_instance(name, seeds(name)[1], n_cand=n)
    ctx = S.Context(0)
    try:
        r = _round_inputs(S, inst, q)
        _, _, idx0, val0, cnt0 = _gpu_round(S, ctx, inst, q, n, r)
        torch.cuda.synchronize()
        ctx.check()
        cap = torch.cuda.Stream()
        cap.wait_stream(torch.cuda.current_stream())
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=cap):
            _, _, idx1, val1, cnt1 = _gpu_round(S, ctx, inst, q, n, r, stream=cap)
        for _ in range(2):
            idx1.fill_(-5)
            g.replay()
            torch.cuda.synchronize()
            ctx.check()
            assert torch.equal(idx1, idx0) and torch.equal(val1, val0) and torch.equal(cnt1, cnt0)
    finally:
        ctx.close()
    assert int(cnt0.item()) == q


def test_fantasy_errors_found_on_the_device(S):
    """A fantasy state prepared for fewer picks than asked, or a box capacity
    below the front's need, stops the picks and is reported by the context
    check (SCOOT_EINVAL, SCOOT_EUNSUPPORTED); the context stays usable."""
    name, n = "d12-fantasy", 4096
    inst = make_instance(name, seeds(name)[2], n_cand=n)
    ctx = S.Context(0)
    try:
        r = _round_inputs(S, inst, 4)
        mask = torch.ones(n, dtype=torch.uint8, device="cuda")
        work = torch.empty(S.scoot_fantasy_work_bytes(r["G"], n, 8, r["box_cap"]), dtype=torch.uint8, device="cuda")
        idx, val, cnt = _outputs(8)
        S.scoot_suggest_fantasy(ctx, r["G"], r["state"], r["fant"], r["box_cap"], r["cand"], n, r["eps"], 8, work,
                                idx, val, cnt, mask=mask)
        with pytest.raises(S.ScootError) as e:
            ctx.check()
        assert e.value.status == -1 and int(cnt.item()) == 0
        S.scoot_suggest_fantasy(ctx, r["G"], r["state"], r["fant"], 1, r["cand"], n, r["eps"], 4, work,
                                idx, val, cnt, mask=mask)
        with pytest.raises(S.ScootError) as e:
            ctx.check()
        assert e.value.status == -6 and int(cnt.item()) == 0
        S.scoot_suggest_fantasy(ctx, r["G"], r["state"], r["fant"], r["box_cap"], r["cand"], n, r["eps"], 4, work,
                                idx, val, cnt, mask=mask)
        ctx.check()
        assert int(cnt.item()) == 4
    finally:
        ctx.close()


def test_sharded_picks_equal_the_single_pool_call(S):
    """The phase calls over three shards of one pool (the multi-GPU
    protocol, run one shard after another on one GPU: no kernel waits on
    another shard's): after each pass the shards' records are stacked and
    every shard commits them; every shard's picks, values and count equal
    the single-pool call bit for bit, and so do its variances.  Each record
    decodes (on the host) to the shard's candidate's value, global index and
    configuration words."""
    from paper_2408_04323_gb300.shard import FANT_REC, decode_fantasy_record, selection_key, shard_range
    name, n, q = "d12-fantasy", 30011, 8
    inst = make_instance(name, seeds(name)[2], n_cand=n)
    ctx0 = S.Context(0)
    ctxs = [S.Context(0) for _ in range(3)]
    try:
        r = _round_inputs(S, inst, q)
        var0 = torch.full((inst.n_obj, n), -1.0, device="cuda")
        mask, _, idx0, val0, cnt0 = _gpu_round(S, ctx0, inst, q, n, r, var_out=var0)
        ctx0.check()
        shards = []
        for s in range(3):
            b, e = shard_range(n, s, 3)
            ld = (e - b + 3) // 4 * 4
            cand_s = torch.zeros((inst.d, ld), dtype=torch.int32, device="cuda")
            cand_s[:, :e - b] = r["cand"][:, b:e]
            mask_s = mask[b:e].contiguous()
            work = torch.empty(S.scoot_fantasy_work_bytes(r["G"], e - b, q, r["box_cap"]), dtype=torch.uint8,
                               device="cuda")
            out = _outputs(q)
            S.scoot_fantasy_begin(ctxs[s], r["G"], r["state"], r["fant"], r["box_cap"], cand_s, e - b, r["eps"], q,
                                  work, *out, mask=mask_s, index_offset=b)
            shards.append((b, e, cand_s, mask_s, work, out))
        recs = torch.zeros((3, FANT_REC), dtype=torch.int64, device="cuda")
        for j in range(q):
            for s in range(3):
                S.scoot_fantasy_local_best(ctxs[s], j, recs[s])
            if j == 0:
                for s, (b, e, cand_s, *_rest) in enumerate(shards):
                    dec = decode_fantasy_record(recs[s].cpu().numpy(), inst.d)
                    assert dec is not None and b <= dec[1] < e
                    assert np.array_equal(dec[2], inst.cand[:, dec[1]])
                    assert int(recs[s].cpu().numpy().view(np.uint64)[0]) == selection_key(dec[0], dec[1])
            for s in range(3):
                S.scoot_fantasy_commit(ctxs[s], j, recs)
        for s, (b, e, _, _, _, out) in enumerate(shards):
            var_s = torch.full((inst.n_obj, e - b), -1.0, device="cuda")
            S.scoot_fantasy_end(ctxs[s], var_s)
            ctxs[s].check()
            assert torch.equal(out[0], idx0) and torch.equal(out[1], val0) and torch.equal(out[2], cnt0), s
            assert torch.equal(var_s, var0[:, b:e]), s
    finally:
        for c in ctxs + [ctx0]:
            c.close()
    assert int(cnt0.item()) == q
