"""Pins for oracle.quantizer: Eq. (q), the granular bound of App. A.1 (cell width Delta),
Bennett's Delta^2/12 for inputs uniform within cells, and the published optimum uniform
quantizer steps for a Gaussian source (tests/golden/max1960_uniform_gaussian.txt)."""
import math
import os

import numpy as np
import pytest

from oracle import quantizer as qz

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "max1960_uniform_gaussian.txt")


def test_q_values():
    assert qz.q(1) == 1.0 / 48.0
    assert qz.q(2) == 1.0 / 192.0
    assert qz.q(8) == 2.0 ** -16 / 12.0


def test_one_bit_loading_factor_closed_form():
    # two cells split at 0; the optimum puts each centre at E[X | X > 0] = sqrt(2/pi),
    # i.e. L = 2 sqrt(2/pi); the MSE there is 1 - 2/pi.
    # the MSE is quadratic around its minimum, so a search on MSE values resolves L only to
    # about sqrt(machine epsilon)
    L = qz.loading_factor(1)
    assert abs(L - 2.0 * math.sqrt(2.0 / math.pi)) < 1e-7
    assert abs(qz.gaussian_mse(L, 1) - (1.0 - 2.0 / math.pi)) < 1e-12


def test_golden_max_table():
    rows = [l.split() for l in open(GOLDEN) if l.strip() and not l.startswith("#")]
    for levels, step in rows:
        b = int(levels).bit_length() - 1
        got = 2.0 * qz.loading_factor(b) / (1 << b)
        assert abs(got - float(step)) / float(step) < 1e-3, (levels, got, step)


@pytest.mark.parametrize("b", [1, 2, 3, 5, 8])
def test_gaussian_mse_matches_monte_carlo(b):
    L = qz.loading_factor(b)
    x = np.random.default_rng(b).standard_normal(2_000_000)
    delta = 2 * L / (1 << b)
    xh = qz.dequantize(qz.quantize(x, delta, b), delta, b)
    mc = np.mean((x - xh) ** 2)
    assert abs(mc - qz.gaussian_mse(L, b)) / qz.gaussian_mse(L, b) < 0.01


@pytest.mark.parametrize("b", [1, 2, 4, 7, 8])
def test_granular_error_bound_and_clamp(b):
    delta = 0.37
    lim = delta * (1 << (b - 1))
    y = np.random.default_rng(3).uniform(-3 * lim, 3 * lim, 100000)
    c = qz.quantize(y, delta, b)
    assert c.min() >= 0 and c.max() <= (1 << b) - 1
    yh = qz.dequantize(c, delta, b)
    inside = np.abs(y) < lim
    assert np.all(np.abs(y[inside] - yh[inside]) <= delta / 2 + 1e-15)
    assert np.all(c[y >= lim] == (1 << b) - 1)
    assert np.all(c[y < -lim] == 0)


def test_boundary_goes_to_upper_cell():
    delta, b = 0.5, 3
    # y = 0 is the boundary between codes 3 and 4
    assert qz.quantize(np.array([0.0]), delta, b)[0] == 4
    assert qz.quantize(np.array([-0.5]), delta, b)[0] == 3
    assert qz.dequantize(np.array([4]), delta, b)[0] == 0.25


def test_bennett_uniform_within_cells():
    """Inputs uniform inside the cells give exactly Delta^2/12 (Bennett's granular term)."""
    b, delta = 4, 0.1
    rng = np.random.default_rng(11)
    codes = rng.integers(0, 1 << b, 1_000_000)
    y = qz.dequantize(codes, delta, b) + rng.uniform(-delta / 2, delta / 2, codes.size)
    err = y - qz.dequantize(qz.quantize(y, delta, b), delta, b)
    assert abs(np.mean(err ** 2) / (delta ** 2 / 12) - 1) < 0.01


def test_step_size_uses_mean_retained_variance():
    lam = np.array([4.0, 2.0, 1.0, 1.0])
    b = 2
    d = qz.step_size(lam, b)
    assert abs(d - 2 * qz.loading_factor(b) * math.sqrt(2.0) / 4) < 1e-15
