"""The static per-head uniform scalar quantizer and its distortion model.

Paper: Eq. (q) q(b) = 2^{-2b}/12 (Sec. 3 "Distortion model"; App. A.1, Eq. q-normalized);
the quantizer of App. A.1: inputs clipped to [-L sigma, L sigma], step
Delta = 2 L sigma / 2^b, one static step per head (no per-token scale, App. "effective
bpd": rotation methods carry zero per-token overhead).

Readings (the paper leaves these open):
  * cells: 2^b cells of width Delta tile [-L sigma, L sigma] (the paper says "mid-tread",
    but 2^b cells of width 2 L sigma / 2^b is the mid-rise geometry; a mid-tread grid with
    2^b levels would be asymmetric and degenerate at b = 1).  code = clamp(floor(y/Delta
    + 2^{b-1}), 0, 2^b - 1), reconstruction at the cell centre Delta (code - 2^{b-1} + 1/2);
    an input exactly on a cell boundary belongs to the upper cell.
  * sigma: the common per-channel standard deviation after the rotation,
    sigma_bar^2 = (1/r) sum_{i<=r} lambda_i (App. A.1, Lemma head-dist step 4).
  * loading factor L_b: never given (absorbed into alpha).  Taken as the L minimising the
    exact mean-squared error of this quantizer on N(0, 1) (golden-section search).
"""
from __future__ import annotations

import math

import numpy as np


def q(b: int) -> float:
    """Bennett leading-order distortion per unit variance, Eq. (q): 2^{-2b} / 12."""
    return math.ldexp(1.0, -2 * b) / 12.0


def _phi(x: float) -> float:
    if math.isinf(x):
        return 0.0
    return math.exp(-0.5 * x * x) / math.sqrt(2.0 * math.pi)


def _Phi(x: float) -> float:
    if x == math.inf:
        return 1.0
    if x == -math.inf:
        return 0.0
    return 0.5 * math.erfc(-x / math.sqrt(2.0))


def _cell_mse(a: float, b: float, c: float) -> float:
    """int_a^b (x - c)^2 phi(x) dx for the standard normal density (closed form from
    int x^2 phi = Phi - x phi and int x phi = -phi)."""
    ta = 0.0 if math.isinf(a) else a * _phi(a)
    tb = 0.0 if math.isinf(b) else b * _phi(b)
    return (1.0 + c * c) * (_Phi(b) - _Phi(a)) - (tb - ta) + 2.0 * c * (_phi(b) - _phi(a))


def gaussian_mse(L: float, b: int) -> float:
    """Exact MSE of the 2^b-cell clamped uniform quantizer on [-L, L] for X ~ N(0, 1)."""
    n = 1 << b
    step = 2.0 * L / n
    total = 0.0
    for k in range(n):
        lo = -math.inf if k == 0 else -L + k * step
        hi = math.inf if k == n - 1 else -L + (k + 1) * step
        centre = -L + (k + 0.5) * step
        total += _cell_mse(lo, hi, centre)
    return total


def loading_factor(b: int, lo: float = 0.5, hi: float = 8.0, tol: float = 1e-12) -> float:
    """MSE-optimal loading factor L_b for N(0,1) (golden-section search on [lo, hi])."""
    gr = (math.sqrt(5.0) - 1.0) / 2.0
    a, c = lo, hi
    x1 = c - gr * (c - a)
    x2 = a + gr * (c - a)
    f1, f2 = gaussian_mse(x1, b), gaussian_mse(x2, b)
    while c - a > tol:
        if f1 <= f2:
            c, x2, f2 = x2, x1, f1
            x1 = c - gr * (c - a)
            f1 = gaussian_mse(x1, b)
        else:
            a, x1, f1 = x1, x2, f2
            x2 = a + gr * (c - a)
            f2 = gaussian_mse(x2, b)
    return 0.5 * (a + c)


def step_size(lam_retained, b: int, L: float | None = None) -> float:
    """Delta = 2 L_b sigma_bar / 2^b with sigma_bar^2 = mean of the retained eigenvalues."""
    lam = np.asarray(lam_retained, dtype=np.float64)
    if lam.size == 0:
        return 0.0
    if L is None:
        L = loading_factor(b)
    sigma = math.sqrt(float(lam.mean()))
    return 2.0 * L * sigma / (1 << b)


def pre_round(y, delta: float, b: int) -> np.ndarray:
    """u = y / Delta + 2^{b-1}: the value the quantizer floors."""
    return np.asarray(y, dtype=np.float64) / float(delta) + float(1 << (b - 1))


def quantize(y, delta: float, b: int) -> np.ndarray:
    """code = clamp(floor(y/Delta + 2^{b-1}), 0, 2^b - 1) (int64)."""
    u = pre_round(y, delta, b)
    return np.clip(np.floor(u), 0, (1 << b) - 1).astype(np.int64)


def dequantize(code, delta: float, b: int) -> np.ndarray:
    """Cell centre Delta (code - 2^{b-1} + 1/2)."""
    return float(delta) * (np.asarray(code, dtype=np.float64) - (1 << (b - 1)) + 0.5)
