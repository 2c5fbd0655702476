"""One suggestion round through the C ABI: prune -> forest -> posterior +
acquisition -> top-q (Section 4, Algorithm 1's SUGGEST step), or, for one
objective with MACE, posterior + (UCB, PI, EI) -> random k-subset of their
Pareto front (Sections 4.5 and 4.7).

Host-side state (GP factor, box decomposition, packed forest) is prepared by
the library's own host functions (the GP state optionally by the library's
device kernels); torch only holds device memory and streams.  Nothing here
computes any step of the path itself.
"""
from __future__ import annotations

import math
from dataclasses import dataclass

import numpy as np
import torch

from . import scoot as S


@dataclass
class RoundInputs:
    """Host arrays describing one round (layouts as in include/scoot.h)."""
    space: np.ndarray          # scoot_param[d]
    clauses: np.ndarray        # scoot_clause[n_clauses]
    nodes: np.ndarray          # scoot_node[total]
    tree_offset: np.ndarray    # int32[T+1]
    leaf_scale: int
    delta_num: int
    delta_den: int
    x_obs: np.ndarray          # uint32[d][n]
    y_obs: np.ndarray          # float32[M][n]
    lengthscale: np.ndarray    # float32[M][d]
    signal_var: np.ndarray     # float32[M]
    noise_var: np.ndarray      # float32[M]
    ref: np.ndarray            # float32[M]
    eps: np.ndarray            # float32[S][M]
    acq: str                   # "ei", "ehvi", "ehvi-exact" or "mace"
    q: int
    kernel: int = S.MATERN52
    xi: float = 1e-4
    fantasy: bool = False      # q sequential picks with kriging-believer fantasies
    kappa: float | None = None  # MACE: UCB coefficient (None: mace_beta(n_obs))
    seed: int = 0               # MACE: seed of the random draw from the front
    warp: np.ndarray | None = None  # float32 [M][d][2]: Kumaraswamy input warping (None: no warping)


def mace_beta(t: int) -> float:
    """UCB coefficient for tuning iteration t (Section 4.5):
    beta_t = 2 log(t^2 pi^2 / (6 delta)) with delta = 1 / t^2, taken as the
    factor of sigma in UCB = mu + beta sigma as printed."""
    t = max(int(t), 1)
    delta = 1.0 / (t * t)
    return 2.0 * math.log(t * t * math.pi ** 2 / (6.0 * delta))


class _Staging:
    """A reused pinned host buffer for uploading a round's state in one copy.

    A new round may refill it only once the previous upload has left it (an
    event recorded after each copy is waited for before the next fill)."""

    def __init__(self):
        self.buf = None
        self.done = None

    def take(self, nbytes: int) -> torch.Tensor:
        if self.done is not None:
            self.done.synchronize()
        if self.buf is None or self.buf.numel() < nbytes:
            self.buf = torch.empty(max(nbytes, 1 << 20), dtype=torch.uint8, pin_memory=True)
        return self.buf[:nbytes]

    def sent(self, stream) -> None:
        self.done = torch.cuda.Event()
        self.done.record(stream)


_staging = _Staging()


class State:
    """Per-round state prepared by the library's host functions and uploaded
    to the device in one copy from pinned memory; gp_state, forest, box_lo,
    box_hi, eps, grid and corner are views into one device buffer.
    With ``gp_on_device`` the GP state is built by the device instead
    (scoot_gp_prepare_device, asynchronously on ``stream`` after the upload
    of its inputs), overlapping the host's preparation of the rest.
    With ``into`` (a State of the same shapes) the upload reuses that State's
    device buffer, so work captured against it (a CUDA graph) stays valid."""

    def __init__(self, inp: RoundInputs, device: torch.device, stream=None, into=None, gp_on_device=False,
                 ctx=None):
        d = len(inp.space)
        M, n = inp.y_obs.shape
        self.gp_layout = S.scoot_gp_layout_init(inp.space, n, M, inp.kernel)
        self.cond = None
        stream = torch.cuda.current_stream(device) if stream is None else stream
        parts = []
        if gp_on_device:
            if ctx is None:
                raise ValueError("gp_on_device needs a context")
            gp_in = [("gpin_obs", np.ascontiguousarray(inp.x_obs[:, :n]).view(np.int32)),
                     ("gpin_y", np.ascontiguousarray(inp.y_obs, np.float32)),
                     ("gpin_ls", np.ascontiguousarray(inp.lengthscale, np.float32)),
                     ("gpin_sf2", np.ascontiguousarray(inp.signal_var, np.float32)),
                     ("gpin_tau2", np.ascontiguousarray(inp.noise_var, np.float32))]
            if inp.warp is not None:
                gp_in.append(("gpin_warp", np.ascontiguousarray(inp.warp, np.float32)))
            parts += gp_in
        else:
            if inp.warp is None:
                blob, self.cond = S.scoot_gp_prepare(inp.space, inp.x_obs, inp.y_obs, inp.lengthscale,
                                                     inp.signal_var, inp.noise_var, self.gp_layout)
            else:
                blob, self.cond = S.scoot_gp_prepare_warped(inp.space, inp.x_obs, inp.y_obs, inp.lengthscale,
                                                            inp.signal_var, inp.noise_var, inp.warp,
                                                            self.gp_layout)
            parts.append(("gp_state", blob))
        self.forest_layout = S.scoot_forest_layout_init(inp.nodes, inp.tree_offset, d, inp.leaf_scale)
        fblob = S.scoot_forest_pack(self.forest_layout, inp.nodes, inp.tree_offset)
        parts.append(("forest", fblob))
        self.n_boxes = 0
        self.front_size = 0
        if inp.acq in ("ehvi", "ehvi-exact"):
            lo, hi, self.front_size = S.scoot_boxes_build(inp.y_obs, inp.ref)
            self.n_boxes = len(lo)
            self.h_boxes = (lo, hi)
            parts += [("box_lo", lo), ("box_hi", hi), ("eps", np.ascontiguousarray(inp.eps, np.float32))]
        if inp.acq == "ehvi-exact":
            grid, self.n_grid, corner = S.scoot_boxes_index(lo, hi)
            self.h_boxes = (lo, hi, grid, corner)
            parts += [("grid", grid), ("corner", corner.view(np.int32))]
        self.h_blobs = tuple(arr for _, arr in parts)
        # one upload: 256-byte aligned slots in a pinned staging buffer; a
        # device-built GP state takes a slot after the uploaded ones
        offs, total = [], 0
        for _, arr in parts:
            offs.append(total)
            total += (arr.nbytes + 255) // 256 * 256
        upload = total
        if gp_on_device:
            gp_off = total
            total += (self.gp_layout.bytes + 255) // 256 * 256
            work_off = total
            work_bytes = S.scoot_gp_device_work_bytes(self.gp_layout)
            total += (work_bytes + 255) // 256 * 256
        stage = _staging.take(upload)
        host = stage.numpy()
        for (_, arr), o in zip(parts, offs):
            host[o:o + arr.nbytes] = np.ascontiguousarray(arr).reshape(-1).view(np.uint8)
        if into is not None and into.buffer.numel() == total and into.offsets == offs:
            dev = into.buffer
        else:
            dev = torch.empty(total, dtype=torch.uint8, device=device)
            if stream != torch.cuda.current_stream(device):
                dev.record_stream(stream)
        with torch.cuda.stream(stream):
            dev[:upload].copy_(stage, non_blocking=True)
        _staging.sent(stream)
        self.buffer = dev
        self.offsets = offs
        self.upload_bytes = upload
        views = {}
        for (name, arr), o in zip(parts, offs):
            view = dev[o:o + arr.nbytes]
            if arr.dtype != np.uint8:
                view = view.view(torch.float32 if arr.dtype == np.float32 else torch.int32).reshape(arr.shape)
            views[name] = view
            if not name.startswith("gpin_"):
                setattr(self, name, view)
        if gp_on_device:
            self.gp_state = dev[gp_off:gp_off + self.gp_layout.bytes]
            S.scoot_gp_prepare_device(ctx, inp.space, self.gp_layout, views["gpin_obs"], views["gpin_y"],
                                      views["gpin_ls"], views["gpin_sf2"], views["gpin_tau2"], self.gp_state,
                                      work=dev[work_off:work_off + work_bytes], warp=views.get("gpin_warp"),
                                      stream=stream)


class ScoringRound:
    """Device buffers for pools of up to `capacity` candidates and the calls of one round."""

    def __init__(self, ctx: S.Context, inp: RoundInputs, capacity: int, device=None, gp_on_device=False):
        self.ctx = ctx
        self.inp = inp
        self.device = torch.device("cuda", ctx.device) if device is None else torch.device(device)
        self.gp_on_device = bool(gp_on_device)
        self.state = State(inp, self.device, gp_on_device=self.gp_on_device, ctx=ctx)
        self.capacity = int(capacity)
        dev = self.device
        self.mask = torch.empty(self.capacity, dtype=torch.uint8, device=dev)
        self.votes = torch.empty(self.capacity, dtype=torch.int32, device=dev)
        self.acq = torch.empty(self.capacity, dtype=torch.float32, device=dev)
        self.n_known = torch.zeros(1, dtype=torch.int64, device=dev)
        self.n_feasible = torch.zeros(1, dtype=torch.int64, device=dev)
        q = inp.q
        self.top_idx = torch.empty(q, dtype=torch.int64, device=dev)
        self.top_val = torch.empty(q, dtype=torch.float32, device=dev)
        self.top_count = torch.empty(1, dtype=torch.int32, device=dev)
        self.work = None
        if inp.fantasy:
            nbytes = S.scoot_fantasy_work_bytes(self.state.gp_layout, self.capacity, q)
            self.work = torch.empty(nbytes, dtype=torch.uint8, device=dev)
        self.picks = None
        self.sobol_skip = 0  # next point of the Sobol sequence for shortfall fills
        self.acq3 = self.front = None
        if inp.acq == "mace":
            if inp.y_obs.shape[0] != 1:
                raise ValueError("MACE scores one objective")
            self.acq3 = torch.empty((3, self.capacity), dtype=torch.float32, device=dev)
            self.front_cap = 4096
            self.front = torch.empty(self.front_cap, dtype=torch.int64, device=dev)
            self.top_count = torch.empty(2, dtype=torch.int32, device=dev)
            self.kappa = float(mace_beta(inp.y_obs.shape[1]) if inp.kappa is None else inp.kappa)
            self.seed = int(inp.seed)

    # number of library kernels one call of run() launches (plain top-q rounds)
    KERNELS_PER_ROUND = 7

    def kernels_per_round(self):
        """Library kernel launches of one run(): prune, compaction, forest walk, then
        either compaction + fused score + two top-q passes, or (fantasies)
        compaction + posterior + per pick EHVI, two argmax passes and a downdate
        (the last pick skips the downdate)."""
        if self.inp.acq == "mace":
            return 10  # prune, compaction, forest, compaction, score, five Pareto kernels
        if not self.inp.fantasy:
            return 7
        return 3 + 2 + 4 * self.inp.q - 1

    def fill_shortfall(self, batch: int = 4096, stream=None):
        """Section 4.6: when a round yields fewer than q suggestions, the rest
        are Sobol points.  Reading: the first q - count points of the sequence
        (continuing from self.sobol_skip) that satisfy the known constraints.
        Returns host words [d][m] (m <= q - count, fewer only if a batch of
        points holds too few feasible ones) and advances the sequence past
        the last point used.  Synchronises with the round's count."""
        count = int(self.top_count[0].item())
        need = self.inp.q - count
        if need <= 0:
            return np.zeros((len(self.inp.space), 0), np.uint32)
        batch = (int(batch) + 3) // 4 * 4
        dev = self.device
        words = torch.empty((len(self.inp.space), batch), dtype=torch.int32, device=dev)
        mask = torch.empty(batch, dtype=torch.uint8, device=dev)
        idx = torch.empty(need, dtype=torch.int64, device=dev)
        cnt = torch.empty(1, dtype=torch.int32, device=dev)
        S.scoot_sobol_configs(self.ctx, self.inp.space, self.sobol_skip, batch, words, stream)
        S.scoot_prune(self.ctx, self.inp.space, self.inp.clauses, words, batch, mask, None, stream)
        S.scoot_first_feasible(self.ctx, mask, batch, need, idx, cnt, stream)
        got = int(cnt.item())
        pos = idx[:got].cpu().numpy()
        self.sobol_skip += int(pos[-1]) + 1 if got == need else batch
        return words.cpu().numpy().view(np.uint32)[:, pos]

    def run(self, cand: torch.Tensor, n: int, stream=None):
        """prune -> rf -> score -> top-q on a resident pool cand (int32 [d][ld]).

        Returns (idx, val, count).  With MACE, idx holds the random picks from
        the front, count is (picks, front size), val is not written and the
        front itself is in self.front (first front_cap members)."""
        if n > self.capacity:
            raise ValueError("pool larger than the round's capacity")
        inp, st = self.inp, self.state
        S.scoot_prune(self.ctx, inp.space, inp.clauses, cand, n, self.mask, self.n_known, stream)
        S.scoot_rf_predict(self.ctx, st.forest_layout, st.forest, inp.space, cand, n, inp.delta_num,
                           inp.delta_den, self.votes, self.mask, self.n_feasible, stream)
        if inp.fantasy:
            idx, val = S.scoot_suggest_fantasy(self.ctx, st.gp_layout, st.gp_state, inp.space, inp.x_obs, inp.y_obs,
                                               inp.lengthscale, inp.signal_var, inp.noise_var, cand, n, inp.ref,
                                               st.eps, inp.q, self.work, mask=self.mask, stream=stream)
            self.picks = (idx, val)
            k = len(idx)
            self.top_idx[:k].copy_(torch.from_numpy(idx))
            self.top_val[:k].copy_(torch.from_numpy(val))
            self.top_count.fill_(k)
            return self.top_idx, self.top_val, self.top_count
        if inp.acq == "mace":
            S.scoot_score_mace(self.ctx, st.gp_layout, st.gp_state, cand, n, inp.xi, self.kappa, self.acq3,
                               self.mask, stream)
            S.scoot_select_pareto(self.ctx, self.acq3, n, inp.q, self.seed, self.top_idx, self.top_count,
                                  self.mask, self.front, stream)
            return self.top_idx, self.top_val, self.top_count
        if inp.acq == "ei":
            S.scoot_score_ei(self.ctx, st.gp_layout, st.gp_state, cand, n, inp.xi, self.acq, self.mask, stream)
        elif inp.acq == "ehvi-exact":
            S.scoot_score_ehvi_exact(self.ctx, st.gp_layout, st.gp_state, cand, n, st.grid, st.n_grid, st.corner,
                                     self.acq, self.mask, stream)
        else:
            S.scoot_score_ehvi(self.ctx, st.gp_layout, st.gp_state, cand, n, st.box_lo, st.box_hi, st.eps,
                               self.acq, self.mask, stream)
        S.scoot_select_topq(self.ctx, self.acq, n, inp.q, self.top_idx, self.top_val, self.top_count,
                            self.mask, stream)
        return self.top_idx, self.top_val, self.top_count
