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
    """UCB coefficient for tuning iteration t (Section 4.5), from the library
    (scoot_ucb_beta); t < 1 counts as 1."""
    return S.scoot_ucb_beta(max(int(t), 1))


class _Staging:
    """A reused pinned host buffer for uploading a round's state in one copy.

    A new round may refill it only once the previous upload has left it (an
    event recorded after each copy is waited for before the next fill)."""

    def __init__(self):
        self.buf = None
        self.done = None

    def capacity(self) -> int:
        return 1 << 20 if self.buf is None else self.buf.numel()

    def take(self, nbytes: int, keep: int = 0) -> torch.Tensor:
        """The buffer, at least nbytes long; when it has to grow, its first
        `keep` bytes are carried over."""
        if self.done is not None:
            self.done.synchronize()
        if self.buf is None or self.buf.numel() < nbytes:
            old = self.buf
            self.buf = torch.empty(max(nbytes, 1 << 20), dtype=torch.uint8, pin_memory=True)
            if old is not None and keep:
                self.buf[:keep].copy_(old[:keep])
        return self.buf

    def sent(self, stream) -> None:
        self.done = torch.cuda.Event()
        self.done.record(stream)


_staging = _Staging()
_staging_gp = _Staging()  # the GP inputs, uploaded before the rest when the device builds the GP state


class State:
    """Per-round state built by the library's host call
    scoot_round_state_build (GP state, packed forest, boxes with eps or with
    their grid index) straight into a pinned staging buffer and uploaded in
    one copy; gp_state, forest, box_lo, box_hi, eps, grid and corner are
    views into device buffers.  With ``gp_on_device`` the GP state is built
    by the device (scoot_gp_prepare_device): its inputs are uploaded and its
    kernels launched on ``stream`` first, so that the device factorises
    while the host packs the forest and builds the boxes.  With ``into`` (a
    State of the same shapes) the uploads reuse that State's device buffers
    and views, so work captured against them (a CUDA graph) stays valid."""

    def __init__(self, inp: RoundInputs, device: torch.device, stream=None, into=None, gp_on_device=False,
                 ctx=None):
        M, n = inp.y_obs.shape
        stream = torch.cuda.current_stream(device) if stream is None else stream
        if gp_on_device and ctx is None:
            raise ValueError("gp_on_device needs a context")
        self.gp_buffer = None
        if gp_on_device:
            self._gp_on_device(inp, device, stream, into, ctx)
        boxes = {"ehvi": 1, "ehvi-exact": 2}.get(inp.acq, 0)
        stage = _staging.take(_staging.capacity())
        while True:
            built, out = S.scoot_round_state_build(inp.space, inp.x_obs, inp.y_obs, inp.lengthscale,
                                                   inp.signal_var, inp.noise_var, inp.nodes, inp.tree_offset,
                                                   inp.leaf_scale, stage.numpy(), kernel=inp.kernel, warp=inp.warp,
                                                   boxes=boxes, h_ref=inp.ref, h_eps=inp.eps,
                                                   gp_on_device=gp_on_device,
                                                   fantasy_q=inp.q if inp.fantasy else 0)
            if built is not None:
                break
            stage = _staging.take(int(out.bytes))
        self.gp_layout = out.gp
        self.forest_layout = out.forest
        self.cond = [out.cond[m] for m in range(M)] if not gp_on_device else None
        self.n_boxes = int(out.n_boxes)
        self.front_size = int(out.front_size)
        if boxes == 2:
            self.n_grid = np.array(out.n_grid[:M], np.int32)
        total = int(out.bytes)
        offsets = (int(out.off_gp), int(out.off_forest), int(out.off_box_lo), int(out.off_box_hi), int(out.off_eps),
                   int(out.off_grid), int(out.off_corner), int(out.off_fant), total)
        self.fant_box_cap = int(out.fant_box_cap)
        reuse = into is not None and into.buffer.numel() == total and into.offsets == offsets
        if reuse:
            dev = into.buffer
        else:
            dev = torch.empty(total, dtype=torch.uint8, device=device)
            if stream != torch.cuda.current_stream(device):
                dev.record_stream(stream)
        with torch.cuda.stream(stream):
            dev.copy_(stage[:total], non_blocking=True)
        _staging.sent(stream)
        self.buffer = dev
        self.offsets = offsets
        self.upload_bytes = total + (self.gp_upload_bytes if gp_on_device else 0)
        if reuse:  # same offsets: the views of `into` are views of this buffer
            for name in ("forest", "box_lo", "box_hi", "eps", "grid", "corner", "fant_state") + \
                    (() if gp_on_device else ("gp_state",)):
                if hasattr(into, name):
                    setattr(self, name, getattr(into, name))
            return

        def view(off, nbytes, dtype=None, shape=None):
            v = dev[off:off + nbytes]
            return v if dtype is None else v.view(dtype).reshape(shape)
        if not gp_on_device:
            self.gp_state = view(out.off_gp, self.gp_layout.bytes)
        self.forest = view(out.off_forest, self.forest_layout.bytes)
        if inp.fantasy:
            self.fant_state = view(out.off_fant, S.scoot_fantasy_state_bytes(self.gp_layout, inp.q))
        B = self.n_boxes
        if boxes:
            self.box_lo = view(out.off_box_lo, B * M * 4, torch.float32, (B, M))
            self.box_hi = view(out.off_box_hi, B * M * 4, torch.float32, (B, M))
        if boxes == 1:
            self.eps = view(out.off_eps, inp.eps.shape[0] * M * 4, torch.float32, (inp.eps.shape[0], M))
        if boxes == 2:
            self.grid = view(out.off_grid, M * out.grid_cap * 4, torch.float32, (M, out.grid_cap))
            self.corner = view(out.off_corner, B * M * 4, torch.int32, (B, M))

    def _gp_on_device(self, inp, device, stream, into, ctx):
        """Upload the GP inputs and launch the device build of the GP state
        (one library call)."""
        M, n = inp.y_obs.shape
        layout = S.scoot_gp_layout_init(inp.space, n, M, inp.kernel)
        up, blob_off, _, total = S.scoot_gp_device_buffer_layout(layout, inp.warp is not None)
        if into is not None and into.gp_buffer is not None and into.gp_buffer.numel() == total:
            dev = into.gp_buffer
            self.gp_state = into.gp_state
        else:
            dev = torch.empty(total, dtype=torch.uint8, device=device)
            if stream != torch.cuda.current_stream(device):
                dev.record_stream(stream)
            self.gp_state = dev[blob_off:blob_off + layout.bytes]
        stage = _staging_gp.take(up)
        S.scoot_gp_prepare_device_from_host(ctx, inp.space, layout, inp.x_obs, inp.y_obs, inp.lengthscale,
                                            inp.signal_var, inp.noise_var, stage, dev, warp=inp.warp, stream=stream)
        _staging_gp.sent(stream)
        self.gp_buffer = dev
        self.gp_upload_bytes = up


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
            nbytes = S.scoot_fantasy_work_bytes(self.state.gp_layout, self.capacity, q, self.state.fant_box_cap)
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
        compaction + posterior + the front's boxes + per pick a pass (downdate,
        EHVI, block argmax) and the pick's terms."""
        if self.inp.acq == "mace":
            return 10  # prune, compaction, forest, compaction, score, five Pareto kernels
        if not self.inp.fantasy:
            return 7
        return 3 + 3 + 2 * self.inp.q

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
            S.scoot_suggest_fantasy(self.ctx, st.gp_layout, st.gp_state, st.fant_state, st.fant_box_cap, cand, n,
                                    st.eps, inp.q, self.work, self.top_idx, self.top_val, self.top_count,
                                    mask=self.mask, stream=stream)
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
