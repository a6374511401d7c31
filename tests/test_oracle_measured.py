"""Pins of the oracle's measured-distortion tables and the exact DP over them (App. E,
"Exact DP over measured distortion"), checked against what the definitions and the
mathematics fix rather than against the oracle itself:
  * r = 0 keeps nothing: D = sum_i w_i exactly (the basis diagonalises the tokens' own
    population covariance), for the MSE and the attention-KL weights;
  * the reconstruction-based table equals an independent evaluation in the eigen coordinates
    (truncated energy plus the rotated-back quantisation error of y = H_r c_r);
  * with Gaussian tokens the quantisation error of each Hadamard block is the closed-form
    Gaussian MSE of the clamped uniform quantizer at that block's loading (quantizer
    .gaussian_mse), within the sampling error of 4096 tokens;
  * the table DP reproduces the surrogate DP when fed the surrogate's own tables, and equals a
    brute-force search over every combination of per-head choices on random tables."""
import itertools
import math

import numpy as np
import pytest

from oracle import allocator as oal
from oracle import calibrate as ocal
from oracle import hadamard as ohad
from oracle import measured as om
from oracle import quantizer as oq
from paper_2609_24298_gb300 import synth


def head(cfg=2, layer=3, h=1, side=1, kl=False, n=512):
    spec = synth.CONFIGS[cfg]
    src = synth.HeadSource(cfg, layer, h, side, spec["alpha"])
    x = src.calibration(n)
    qc = synth.calibration_queries(cfg, layer, h, 4, 512, spec["alpha"]) if kl else None
    cal = ocal.calibrate_head(x, qc)
    return x, cal, om.error_weights(cal, qc), synth.hadamard_signs(*src.key)


@pytest.mark.parametrize("kl", [False, True])
def test_rank_zero_is_total_weight(kl):
    x, cal, omega, signs = head(kl=kl)
    D = om.measured_distortion(x, cal, omega, signs, 0, 1)
    assert D == pytest.approx(float(np.sum(cal["w"])), rel=1e-9)


@pytest.mark.parametrize("kl", [False, True])
@pytest.mark.parametrize("r,b", [(2, 1), (18, 2), (64, 3), (100, 4), (128, 8)])
def test_eigen_coordinate_evaluation(kl, r, b):
    x, cal, omega, signs = head(kl=kl)
    D = om.measured_distortion(x, cal, omega, signs, r, b)
    # independent evaluation: c = U^T (x - mu); y = H_r c_r; the error in the eigen basis is
    # c_i for i > r and (H_r^T (y - y^))_i for i <= r
    c = (np.asarray(x, np.float64) - cal["mu"][None, :]) @ cal["U"]
    H = ohad.hadamard(r, signs)
    y = c[:, :r] @ H.T
    delta = float(np.float32(oq.step_size(cal["lam"][:r], b)))
    code = np.clip(np.floor(y / delta + 2 ** (b - 1)), 0, 2 ** b - 1)
    eps = y - delta * (code - 2 ** (b - 1) + 0.5)
    e = np.concatenate([eps @ H, c[:, r:]], axis=1)
    D2 = float(np.mean((e * e) @ omega))
    assert D == pytest.approx(D2, rel=1e-4)


@pytest.mark.parametrize("r", [32, 100, 128])
@pytest.mark.parametrize("b", [1, 2, 3, 4])
def test_block_error_matches_gaussian_closed_form(r, b):
    # MSE weights: block beta of H_r mixes channels of mean variance v_beta, so every rotated
    # channel of the block is N(0, v_beta); with the common step Delta = 2 L_b sigma_bar / 2^b
    # its error is v_beta * gaussian_mse(L_b sigma_bar / sqrt(v_beta), b).  4096 tokens: the
    # channels of a block are strongly correlated (the leading eigen-direction dominates), so
    # the overload part of the error needs many tokens to settle (512 tokens under-sample the
    # tails by up to 15% at b = 4; 4096 by 3%)
    x, cal, omega, signs = head(kl=False, n=4096)
    D = om.measured_distortion(x, cal, omega, signs, r, b)
    lam = cal["lam"]
    sigma = math.sqrt(float(np.mean(lam[:r])))
    L = oq.loading_factor(b)
    pred, o = float(np.sum(lam[r:])), 0
    for n in ohad.block_sizes(r):
        v = float(np.mean(lam[o:o + n]))
        pred += n * v * oq.gaussian_mse(L * sigma / math.sqrt(v), b)
        o += n
    kept = D - float(np.sum(lam[r:]))
    kept_pred = pred - float(np.sum(lam[r:]))
    assert kept == pytest.approx(kept_pred, rel=0.05)


def test_table_layout_and_monotone_truncation():
    x, cal, omega, signs = head(kl=True)
    rg, bg = [0, 2, 8, 32], [1, 2, 3]
    T = om.measured_table(x, cal, omega, signs, rg, bg)
    assert T.shape == (4, 3)
    assert np.all(T[0] == T[0, 0])
    for i, r in enumerate(rg):
        # what is dropped is exactly the energy past r; the kept part only adds
        assert np.all(T[i] >= float(np.sum(cal["w"][r:])) * (1 - 1e-12))


def test_table_dp_reproduces_surrogate_dp():
    rng = np.random.default_rng(3)
    d = 8
    o = oal.Opts(mode=oal.MODE_EXACT, b_min=1, b_max=8, r_step=2, allow_r0=True)
    rg, bg = oal.rank_grid(d, o), list(range(1, 9))
    W = np.sort(rng.gamma(1.0, 1.0, (5, d)), axis=1)[:, ::-1]
    pres = [oal.prefix_sums(w) for w in W]
    tables = [np.array([[oal.distortion(p, r, b if r else 0) for b in bg] for r in rg]) for p in pres]
    for B in (5.0, 17.0, 40.0):
        r1, b1, D1, t1 = oal.exact_dp(pres, B, o)
        r2, b2, D2, t2 = om.exact_dp_tables(tables, rg, bg, B)
        assert (r1, b1) == (r2, b2) and t1 == t2


def test_table_dp_equals_brute_force():
    rng = np.random.default_rng(11)
    rg, bg = [0, 2, 4], [1, 2, 3]
    for trial in range(20):
        tables = [np.sort(rng.random((3, 3)), axis=None)[::-1].reshape(3, 3) for _ in range(3)]
        for t in tables:
            t[0, :] = t[0, 0] + 1.0  # r = 0: the largest distortion, any b
        B = float(rng.integers(0, 25))
        _, _, _, tot = om.exact_dp_tables(tables, rg, bg, B)
        best = math.inf
        per = [[(0, t[0, 0])] + [(r * b, t[i, j]) for i, r in enumerate(rg) if r for j, b in enumerate(bg)]
               for t in tables]
        for combo in itertools.product(*per):
            if sum(c[0] for c in combo) <= B:
                best = min(best, sum(c[1] for c in combo))
        assert tot == pytest.approx(best, rel=0, abs=1e-12)
