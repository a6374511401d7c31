"""Measured per-head distortion tables and the exact DP over them (App. E, "Exact DP over
measured distortion"; Table c2-measured).  Test infrastructure: only tests/, the smoke entry
point and the benchmark's CPU baseline may use this module.

The allocator's surrogate D(r, b) = sum_{i>r} w_i + q(b) sum_{i<=r} w_i (Eq. drb-preview)
assumes the Bennett high-resolution quantizer model q(b) = 2^{-2b}/12.  App. E replaces it by
the distortion measured when the head's calibration activations go through the deployed
quantizer once per candidate (r, b), and re-runs the same exact DP on those tables.

Definition followed (the paper states the procedure, not a formula; this is its plain
reading in the allocator's own units):
  D_meas(r, b) = (1/N) sum_t sum_i omega_i (u_i . (x_t - x^_t))^2
where x^_t is the token reconstructed from its codes by the deployed quantizer at (r, b)
(W = U_r H_r^T, Delta and mu as stored: calibrate.head_params; codes: compress.compress;
reconstruction: attention.reconstruct), u_i are the head's basis vectors in the allocator's
order and omega_i the per-direction error weight that makes the surrogate's units: 1 for the
MSE objective (w_i = lambda_i) and sigma_Q,i^2 for the attention-KL objective
(w_i = sigma_Q,i^2 lambda_i).  With these units D_meas(0, b) = sum_i w_i exactly (the basis
diagonalises the population covariance of the same tokens), the r = 0 case of the surrogate.
"""
from __future__ import annotations

import math

import numpy as np

from . import attention, calibrate, compress
from .allocator import Opts, rank_grid


def error_weights(cal, q_cal=None):
    """omega_i in the allocator's basis order: 1 for MSE, sigma_Q,i^2 for KL (the calibration
    queries of the head's group, as in calibrate.calibrate_head)."""
    d = cal["U"].shape[0]
    if q_cal is None:
        return np.ones(d)
    return calibrate.query_variance(cal["U"], q_cal)


def measured_distortion(x_cal, cal, omega, signs, r: int, b: int) -> float:
    """D_meas(r, b) of one head (module docstring), fp64."""
    x = np.asarray(x_cal, dtype=np.float64)
    p = calibrate.head_params(cal, r, b if r else 1, signs)
    if r == 0:
        xh = attention.reconstruct(np.zeros((x.shape[0], 0), np.int64), p["W"], 0.0, 1, p["mu"])
    else:
        _, codes = compress.compress(x, p["W"], p["mu"], p["delta"], b)
        xh = attention.reconstruct(codes, p["W"], p["delta"], b, p["mu"])
    e = (x - xh) @ np.asarray(cal["U"], dtype=np.float64)  # u_i . (x - x^), all i
    return float(np.mean((e * e) @ np.asarray(omega, dtype=np.float64)))


def measured_table(x_cal, cal, omega, signs, r_grid, b_grid) -> np.ndarray:
    """D[i][j] = D_meas(r_grid[i], b_grid[j]); the r = 0 row repeats one value."""
    D = np.zeros((len(r_grid), len(b_grid)))
    for i, r in enumerate(r_grid):
        for j, b in enumerate(b_grid):
            if r == 0 and j > 0:
                D[i, j] = D[i, 0]
            else:
                D[i, j] = measured_distortion(x_cal, cal, omega, signs, int(r), int(b))
    return D


def table_options(table, r_grid, b_grid):
    """All (rate, D, r, b) choices of one head from its table, one per distinct rate (the
    smallest D; on a tie the first in r-ascending, b-ascending order), sorted by rate: the
    same option set allocator.head_options builds from the surrogate."""
    best = {}
    for i, r in enumerate(r_grid):
        bs = [(0, 0)] if r == 0 else list(enumerate(b_grid))
        for j, b in bs:
            rate = int(r) * int(b)
            D = float(table[i][j])
            if rate not in best or D < best[rate][0]:
                best[rate] = (D, int(r), int(b))
    return [(rate, *best[rate]) for rate in sorted(best)]


def exact_dp_tables(tables, r_grid, b_grid, B_tot: float):
    """App. E's exact separable-knapsack DP on per-head tables: minimise sum_h D_h subject to
    sum_h r_h b_h <= B_tot (dp over integer rates; strict '<' keeps the lowest-rate option on
    ties; the final pick is the smallest total D, then the fewest bits).  Returns
    (r, b, D per head, total D)."""
    n = len(tables)
    cap = int(math.floor(B_tot + 1e-9))
    dp = np.full(cap + 1, math.inf)
    dp[0] = 0.0
    choice = np.zeros((n, cap + 1), dtype=np.int32)
    opts = [table_options(t, r_grid, b_grid) for t in tables]
    for h in range(n):
        new = np.full(cap + 1, math.inf)
        ch = np.full(cap + 1, -1, dtype=np.int32)
        for k, (rate, D, _, _) in enumerate(opts[h]):
            if rate > cap:
                break
            cand = np.full(cap + 1, math.inf)
            cand[rate:] = dp[:cap + 1 - rate] + D
            better = cand < new
            new[better] = cand[better]
            ch[better] = k
        dp = new
        choice[h] = ch
    beta = int(np.argmin(dp))
    r, b, D = [0] * n, [0] * n, [0.0] * n
    for h in range(n - 1, -1, -1):
        rate, Dh, rr, bb = opts[h][int(choice[h][beta])]
        r[h], b[h], D[h] = rr, bb, Dh
        beta -= rate
    return r, b, D, float(dp.min())


def default_grids(d: int = 128, o: Opts | None = None):
    """The allocator's candidate grid: r in {0, 2, ..., d}, b in [b_min, b_max]."""
    o = o or Opts()
    return rank_grid(d, o), list(range(o.b_min, o.b_max + 1))
