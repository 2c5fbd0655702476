"""Algorithm 1's tuning loop around the suggestion round, on the library's
calls: a Sobol initial design (Section 4.6), then per iteration the forest
retrained on the crash labels (device CART), the GP hyperparameters fitted
by maximum likelihood (device, from several starts), a candidate pool of
Sobol points scored by the round (prune, forest POF >= Delta, posterior and
acquisition, top-q), a shortfall filled with further Sobol points, and
Delta updated from the evaluated suggestions by the controller.

The caller evaluates the suggestions (the paper's stress tests of the
engine) and reports them with observe().  Nothing here computes a step of
the path: every step is a library call, this module only keeps the history
and marshals it.
"""
from __future__ import annotations

import math

import numpy as np
import torch

from . import scoot as S
from .pipeline import RoundInputs, ScoringRound


class TuningLoop:
    """One tuner: a space, its known-constraint clauses and the settings of
    the round (acquisition, q, forest size, MC samples)."""

    def __init__(self, ctx: S.Context, space, clauses, n_obj: int, q: int, acq: str | None = None,
                 n_trees: int = 100, max_depth: int = 10, leaf_scale: int = 255, n_mc: int = 64,
                 pool: int = 1 << 16, mle_starts: int = 8, mle_steps: int = 60, seed: int = 0):
        self.ctx = ctx
        self.space = np.asarray(space)
        self.clauses = np.asarray(clauses)
        self.d = len(self.space)
        self.M = int(n_obj)
        self.q = int(q)
        self.acq = acq or ("ei" if self.M == 1 else "ehvi")
        self.n_trees, self.max_depth, self.leaf_scale = int(n_trees), int(max_depth), int(leaf_scale)
        self.pool = (int(pool) + 3) // 4 * 4
        self.mle_starts, self.mle_steps = int(mle_starts), int(mle_steps)
        self.rng = np.random.default_rng(seed)
        self.eps = self.rng.standard_normal((int(n_mc), self.M)).astype(np.float32)
        self.device = torch.device("cuda", ctx.device)
        self.x = np.zeros((self.d, 0), np.uint32)       # evaluated configurations (words)
        self.y = np.zeros((self.M, 0), np.float64)      # their objectives (maximised), NaN if crashed
        self.ok = np.zeros(0, bool)                      # ran without crashing
        self.delta, self.delta_count = 0.5, 0             # Algorithm 1's threshold and its counter
        self.sobol_skip = 0
        self.theta = None                                 # [M][d + 2] fitted log hyperparameters

    # ------------------------------------------------------------------ sampling
    def initial_design(self, n: int) -> np.ndarray:
        """The first n Sobol points that satisfy the known constraints."""
        out = np.zeros((self.d, 0), np.uint32)
        batch = max(4096, (4 * n + 3) // 4 * 4)
        while out.shape[1] < n:
            words = torch.empty((self.d, batch), dtype=torch.int32, device=self.device)
            mask = torch.empty(batch, dtype=torch.uint8, device=self.device)
            S.scoot_sobol_configs(self.ctx, self.space, self.sobol_skip, batch, words)
            S.scoot_prune(self.ctx, self.space, self.clauses, words, batch, mask)
            m = mask.cpu().numpy().astype(bool)
            w = words.cpu().numpy().view(np.uint32)[:, m]
            out = np.concatenate([out, w[:, :n - out.shape[1]]], axis=1)
            self.sobol_skip += batch
        return out

    # ------------------------------------------------------------------ history
    def observe(self, words: np.ndarray, y: np.ndarray, ok: np.ndarray) -> None:
        """Evaluated configurations words [d][k], objectives y [M][k]
        (maximised; ignored where ok is False) and whether each ran.  The
        threshold controller sees the batch (any crash raises Delta)."""
        words = np.asarray(words, np.uint32).reshape(self.d, -1)
        ok = np.asarray(ok, bool).reshape(-1)
        y = np.where(ok[None, :], np.asarray(y, np.float64).reshape(self.M, -1), np.nan)
        self.x = np.concatenate([self.x, words], axis=1)
        self.y = np.concatenate([self.y, y], axis=1)
        self.ok = np.concatenate([self.ok, ok])
        self.delta, self.delta_count = S.scoot_delta_update(self.delta, self.delta_count, int(ok.sum()),
                                                            bool((~ok).any()))

    # ------------------------------------------------------------------ model fitting
    def _forest(self):
        """CART forest on bootstraps of all observations, labels = ran."""
        n = self.x.shape[1]
        boot = self.rng.integers(0, n, size=(self.n_trees, n)).astype(np.int32)
        nodes = torch.empty((self.n_trees, 2 * n - 1), dtype=torch.int64, device=self.device)
        counts = torch.empty(self.n_trees, dtype=torch.int32, device=self.device)
        obs = torch.from_numpy(np.ascontiguousarray(self.x).view(np.int32)).to(self.device)
        S.scoot_rf_train(self.ctx, self.space, obs, n, torch.from_numpy(self.ok.astype(np.uint8)).to(self.device),
                         torch.from_numpy(boot).to(self.device), self.max_depth, self.leaf_scale, nodes, counts)
        self.ctx.check()
        return S.compact_forest(nodes.cpu().numpy(), counts.cpu().numpy())

    def _gp(self, words, y_std):
        """Maximum-likelihood hyperparameters per objective from mle_starts
        starts (the previous fit and random ones); returns lengthscales,
        signal and noise variances as float32."""
        n, P = words.shape[1], self.d + 2
        lo = np.array([math.log(0.02)] * self.d + [math.log(0.05), math.log(1e-4)])
        hi = np.array([math.log(20.0)] * self.d + [math.log(20.0), math.log(1.0)])
        base = self.theta if self.theta is not None else np.tile(np.array([0.0] * self.d + [0.0, math.log(0.01)]),
                                                                 (self.M, 1))
        starts = base[None] + self.rng.standard_normal((self.mle_starts, self.M, P)) * 0.5
        starts[0] = base
        starts = np.clip(starts, lo, hi)
        dev = self.device
        th = torch.zeros(starts.shape, dtype=torch.float64, device=dev)
        lml = torch.zeros((self.mle_starts, self.M), dtype=torch.float64, device=dev)
        S.scoot_gp_mle(self.ctx, self.space, torch.from_numpy(np.ascontiguousarray(words).view(np.int32)).to(dev), n,
                       torch.from_numpy(np.ascontiguousarray(y_std, np.float32)).to(dev),
                       torch.from_numpy(np.ascontiguousarray(starts)).to(dev), lo, hi,
                       (1 << P) - 1, self.mle_steps, 0.05, th, lml)
        self.ctx.check()
        th, lml = th.cpu().numpy(), lml.cpu().numpy()
        best = np.nanargmax(np.where(np.isfinite(lml), lml, -np.inf), axis=0)
        self.theta = np.stack([th[best[m], m] for m in range(self.M)])
        ls = np.exp(self.theta[:, :self.d]).astype(np.float32)
        return ls, np.exp(self.theta[:, self.d]).astype(np.float32), np.exp(self.theta[:, self.d + 1]).astype(np.float32)

    # ------------------------------------------------------------------ suggestion
    def suggest(self) -> np.ndarray:
        """q configurations (words [d][q]) for the next evaluations."""
        good = self.ok
        if good.sum() < 2:
            return self.initial_design(self.q)
        words = np.ascontiguousarray(self.x[:, good])
        y_std, ref = S.scoot_standardize(self.y[:, good], ref_margin=1e-3)
        nodes, offs = self._forest()
        ls, sf2, tau2 = self._gp(words, y_std)
        inp = RoundInputs(self.space, self.clauses, nodes, offs, self.leaf_scale, int(round(self.delta * 20)), 20,
                          words, np.ascontiguousarray(y_std, np.float32), ls, sf2, tau2, ref, self.eps, self.acq,
                          self.q)
        rnd = ScoringRound(self.ctx, inp, self.pool, self.device)
        rnd.sobol_skip = self.sobol_skip
        cand = torch.empty((self.d, self.pool), dtype=torch.int32, device=self.device)
        S.scoot_sobol_configs(self.ctx, self.space, self.sobol_skip, self.pool, cand)
        self.sobol_skip += self.pool
        rnd.sobol_skip = self.sobol_skip
        idx, _, count = rnd.run(cand, self.pool)
        k = int(count[0].item())
        picks = cand.cpu().numpy().view(np.uint32)[:, idx[:k].cpu().numpy()]
        fill = rnd.fill_shortfall()
        self.sobol_skip = rnd.sobol_skip
        self.ctx.check()
        return np.concatenate([picks, fill], axis=1)
