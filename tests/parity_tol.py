"""Tolerances shared by the GPU parity tests.

Stated bound: |gpu - oracle| <= 1e-6 + 1e-4 |oracle|.  Derived terms (both
computed by the oracle): the posterior mean adds 2^-22 * sum_j |k_j alpha_j|,
the rounding scale of an fp32 dot product mu = k . alpha; a value computed
from the GPU's own posterior adds the first-order change of the oracle's
value when mu and sigma^2 move by their own tolerances."""
import numpy as np

ATOL, RTOL = 1e-6, 1e-4
MU_COND = 2.0 ** -22


def posterior_tols(gps, words):
    """Oracle mu, var [K][M] and the tolerances of the GPU's mu and var."""
    mv = [gp.posterior(words) for gp in gps]
    mu = np.stack([a for a, _ in mv], 1)
    var = np.stack([b for _, b in mv], 1)
    cond = np.stack([gp.mean_condition(words) for gp in gps], 1)
    e_mu = ATOL + RTOL * np.abs(mu) + MU_COND * cond
    e_var = ATOL + RTOL * var
    return mu, var, e_mu, e_var


def propagated_tol(f, mu, var, e_mu, e_var):
    """f(mu, var), and 1e-6 + 1e-4 |f| plus the half-differences of f when
    each mu_m and var_m moves by its tolerance."""
    base = f(mu, var)
    tol = ATOL + RTOL * np.abs(base)
    for m in range(mu.shape[1]):
        d = np.zeros_like(mu); d[:, m] = e_mu[:, m]
        tol = tol + 0.5 * np.abs(f(mu + d, var) - f(mu - d, var))
        d = np.zeros_like(var); d[:, m] = e_var[:, m]
        tol = tol + 0.5 * np.abs(f(mu, var + d) - f(mu, np.maximum(var - d, 0.0)))
    return base, tol
