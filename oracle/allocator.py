"""Per-head (rank, bit-width) allocation: C1, C2 damped update ("water-filling"), exact DP.

Paper: head distortion D(r, b) of Eq. (drb-preview) / Lemma head-dist; the global problem
Eq. (global); C1 (Sec. 3.2, Prop. c1-kkt and its solver paragraph); C2 (Sec. 3.3, App. D,
Eq. c2-update); exact DP (App. E, Table c2-dp); the calibration loop of Table alg:kvrobin
steps 3-4.

Readings (the paper is silent or inconsistent):
  * C1 feasibility: the paper's b = round(B/r) can give r*b > B.  Here every feasible (r, b)
    with r*b <= B is enumerated; for fixed r, D decreases in b, so the best b is
    min(b_max, floor(B/r)), and r is skipped when that is below b_min.  r = 0 (no codes,
    D = sum w) is a candidate when allow_r0.  Ties: smaller D, then smaller r*b, then
    larger r.  This is the brute-force optimum over the integer feasible set.
  * grid: b in [b_min, b_max] = [1, 8], r in {0, 2, 4, ..., d}.
  * C2: B_min = 0 when allow_r0, else r_step*b_min; C1 runs on the real-valued budgets;
    after the update the budgets are renormalised to sum to B_tot and clamped at B_min once;
    if mean D is 0 the loop stops; exactly `rounds` rounds, then a final C1.
  * completion: after the final C1, bits left unused by the floor (B_tot - sum r*b) are
    spent greedily on the single upgrade (r', b') of some head with the largest distortion
    drop per added bit that still fits, until no upgrade fits.  Total rate then equals the
    budget whenever the remaining slack can buy anything.
  * exact DP: minimises sum D_h over per-head choices subject to sum r_h b_h <= B_tot (the
    separable knapsack of App. E over rates instead of budgets; same optimum).
All sums run sequentially in head / index order so that any other implementation that
follows the same order reproduces the floating-point values bit for bit.
"""
from __future__ import annotations

import itertools
import math
from dataclasses import dataclass

import numpy as np

from .quantizer import q

MODE_DAMPED, MODE_EXACT, MODE_UNIFORM = 0, 1, 2


@dataclass
class Opts:
    mode: int = MODE_DAMPED
    rounds: int = 5
    eta: float = 0.3
    b_min: int = 1
    b_max: int = 8
    r_step: int = 2
    allow_r0: bool = True
    B_min: float | None = None
    complete: bool = True

    def bmin_budget(self) -> float:
        if self.B_min is not None:
            return self.B_min
        return 0.0 if self.allow_r0 else float(self.r_step * self.b_min)


def prefix_sums(w) -> list[float]:
    """pre[k] = w_0 + ... + w_{k-1}, summed left to right."""
    pre = [0.0]
    s = 0.0
    for x in w:
        s = s + float(x)
        pre.append(s)
    return pre


def distortion(pre, r: int, b: int) -> float:
    """D(r, b) = sum_{i>r} w_i + q(b) sum_{i<=r} w_i  (Eq. drb-preview), from prefix sums.
    r = 0 means nothing is kept: D = sum w."""
    d = len(pre) - 1
    if r == 0:
        return pre[d]
    return (pre[d] - pre[r]) + q(b) * pre[r]


def rank_grid(d: int, o: Opts) -> list[int]:
    g = list(range(o.r_step, d + 1, o.r_step))
    return ([0] if o.allow_r0 else []) + g


def c1(pre, B: float, o: Opts):
    """C1 (Sec. 3.2): best (r, b) for one head under r*b <= B.  Returns (r, b, D)."""
    d = len(pre) - 1
    best = None
    for r in rank_grid(d, o):
        if r == 0:
            b = 0
        else:
            b = min(o.b_max, math.floor(B / r))
            if b < o.b_min:
                continue
        D = distortion(pre, r, b)
        key = (D, r * b, -r)
        if best is None or key < best[0]:
            best = (key, r, b, D)
    if best is None:
        raise ValueError("budget admits no (r, b) and r = 0 is not allowed")
    return best[1], best[2], best[3]


def c1_bruteforce(pre, B: float, o: Opts):
    """Every (r, b) on the grid with r*b <= B, smallest D (for pinning c1)."""
    d = len(pre) - 1
    best = None
    for r in rank_grid(d, o):
        bs = [0] if r == 0 else range(o.b_min, o.b_max + 1)
        for b in bs:
            if r * b > B:
                continue
            D = distortion(pre, r, b)
            if best is None or D < best[2]:
                best = (r, b, D)
    return best


def _upgrades(pre, r0: int, b0: int, D0: float, slack: int, o: Opts):
    """Best single upgrade for one head: (gain per bit, extra bits, r, b, D) or None."""
    d = len(pre) - 1
    best = None
    for r in rank_grid(d, o):
        if r == 0:
            continue
        for b in range(o.b_min, o.b_max + 1):
            extra = r * b - r0 * b0
            if extra <= 0 or extra > slack:
                continue
            D = distortion(pre, r, b)
            if not D < D0:
                continue
            gain = (D0 - D) / extra
            if best is None or gain > best[0]:
                best = (gain, extra, r, b, D)
    return best


def complete(pres, r, b, D, B_tot: float, o: Opts):
    """Spend the bits the floor left unused (reading 'completion' above).  In place."""
    slack = int(math.floor(B_tot + 1e-9)) - sum(ri * bi for ri, bi in zip(r, b))
    cache = [None] * len(r)
    while slack > 0:
        best_h = -1
        best = None
        for h in range(len(r)):
            if cache[h] is None or cache[h][1] > slack:
                cache[h] = _upgrades(pres[h], r[h], b[h], D[h], slack, o) or (-1.0, 0, 0, 0, 0.0)
            cand = cache[h]
            if cand[0] <= 0:
                continue
            if best is None or cand[0] > best[0]:
                best, best_h = cand, h
        if best is None:
            break
        _, extra, rr, bb, DD = best
        r[best_h], b[best_h], D[best_h] = rr, bb, DD
        slack -= extra
        cache[best_h] = None
    return slack


def c2_damped(pres, bpd: float, o: Opts, trace=None):
    """C2 damped proportional update (App. D, Eq. c2-update) around C1, Table alg:kvrobin
    steps 3-4: B_h <- bpd*d; `rounds` times: C1 per head, then
    B_h <- max(B_min, B_h + eta * Bbar * (sqrt(D_h / Dbar) - 1)), renormalise to B_tot."""
    n = len(pres)
    d = len(pres[0]) - 1
    B_tot = n * d * bpd
    Bbar = B_tot / n
    Bmin = o.bmin_budget()
    B = [bpd * d] * n
    for _ in range(o.rounds):
        Ds = [c1(pres[h], B[h], o)[2] for h in range(n)]
        s = 0.0
        for x in Ds:
            s = s + x
        Dbar = s / n
        if trace is not None:
            trace.append((list(B), list(Ds)))
        if Dbar == 0.0:
            break
        newB = [max(Bmin, B[h] + o.eta * Bbar * (math.sqrt(Ds[h] / Dbar) - 1.0)) for h in range(n)]
        s = 0.0
        for x in newB:
            s = s + x
        f = B_tot / s
        B = [max(Bmin, x * f) for x in newB]
    res = [c1(pres[h], B[h], o) for h in range(n)]
    return B, [x[0] for x in res], [x[1] for x in res], [x[2] for x in res]


def head_options(pre, o: Opts):
    """All (rate, D, r, b) choices of one head, one per distinct rate (the smallest D; on a
    tie the first in r-ascending, b-ascending order), sorted by rate."""
    d = len(pre) - 1
    best = {}
    for r in rank_grid(d, o):
        bs = [0] if r == 0 else range(o.b_min, o.b_max + 1)
        for b in bs:
            rate = r * b
            D = distortion(pre, r, b)
            if rate not in best or D < best[rate][0]:
                best[rate] = (D, r, b)
    return [(rate, *best[rate]) for rate in sorted(best)]


def exact_dp(pres, B_tot: float, o: Opts):
    """Exact separable-knapsack DP (App. E): minimise sum_h D_h subject to
    sum_h r_h b_h <= B_tot.  dp over integer rates; strict '<' keeps the lowest-rate option on
    ties; the final pick is the smallest total D, then the fewest bits."""
    n = len(pres)
    cap = int(math.floor(B_tot + 1e-9))
    INF = math.inf
    dp = np.full(cap + 1, INF)
    dp[0] = 0.0
    choice = np.zeros((n, cap + 1), dtype=np.int32)
    opts = [head_options(p, o) for p in pres]
    for h in range(n):
        new = np.full(cap + 1, INF)
        ch = np.full(cap + 1, -1, dtype=np.int32)
        for k, (rate, D, _, _) in enumerate(opts[h]):
            if rate > cap:
                break
            cand = np.full(cap + 1, INF)
            cand[rate:] = dp[:cap + 1 - rate] + D
            better = cand < new
            new[better] = cand[better]
            ch[better] = k
        dp = new
        choice[h] = ch
    beta = int(np.argmin(dp))  # first index of the minimum -> fewest bits on ties
    r, b, D = [0] * n, [0] * n, [0.0] * n
    for h in range(n - 1, -1, -1):
        k = int(choice[h][beta])
        rate, Dh, rr, bb = opts[h][k]
        r[h], b[h], D[h] = rr, bb, Dh
        beta -= rate
    return r, b, D, float(dp.min())


def brute_force_joint(pres, B_tot: float, o: Opts):
    """Enumerate every combination of per-head (r, b) (tiny heads only).  Returns the
    minimum total D and one minimiser."""
    d = len(pres[0]) - 1
    per = []
    for p in pres:
        c = []
        for r in rank_grid(d, o):
            for b in ([0] if r == 0 else range(o.b_min, o.b_max + 1)):
                c.append((r * b, distortion(p, r, b), r, b))
        per.append(c)
    best = None
    for combo in itertools.product(*per):
        rate = sum(x[0] for x in combo)
        if rate > B_tot:
            continue
        tot = 0.0
        for x in combo:
            tot = tot + x[1]
        if best is None or tot < best[0]:
            best = (tot, combo)
    return best[0], [(x[2], x[3]) for x in best[1]]


def allocate(weights, bpd: float, o: Opts | None = None):
    """Top level: weights (n_heads x d, each row sorted descending), target bpd.
    Returns dict(r, b, budget, dist, rate_bits, B_tot, slack)."""
    o = o or Opts()
    w = np.asarray(weights, dtype=np.float64)
    n, d = w.shape
    pres = [prefix_sums(w[h]) for h in range(n)]
    B_tot = n * d * bpd
    if o.mode == MODE_EXACT:
        r, b, D, _ = exact_dp(pres, B_tot, o)
        B = [float(ri * bi) for ri, bi in zip(r, b)]
    elif o.mode == MODE_UNIFORM:
        B = [bpd * d] * n
        res = [c1(pres[h], B[h], o) for h in range(n)]
        r, b, D = [x[0] for x in res], [x[1] for x in res], [x[2] for x in res]
    else:
        B, r, b, D = c2_damped(pres, bpd, o)
    slack = int(math.floor(B_tot + 1e-9)) - sum(ri * bi for ri, bi in zip(r, b))
    if o.complete and o.mode != MODE_EXACT:
        slack = complete(pres, r, b, D, B_tot, o)
    return dict(r=np.array(r), b=np.array(b), budget=np.array(B), dist=np.array(D),
                rate_bits=int(sum(ri * bi for ri, bi in zip(r, b))), B_tot=B_tot, slack=slack)
