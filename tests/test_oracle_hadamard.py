"""Pins for oracle.hadamard against the definition of a scaled Walsh-Hadamard matrix and the
variance-equalisation property the paper states (App. A.1; Lemma head-dist, step 4)."""
import numpy as np
import pytest

from oracle import hadamard


def test_sylvester_textbook_orders():
    assert np.array_equal(hadamard.sylvester(2), np.array([[1, 1], [1, -1]]))
    h4 = np.array([[1, 1, 1, 1], [1, -1, 1, -1], [1, 1, -1, -1], [1, -1, -1, 1]])
    assert np.array_equal(hadamard.sylvester(4), h4)


def test_block_sizes():
    assert hadamard.block_sizes(18) == [16, 2]
    assert hadamard.block_sizes(128) == [128]
    assert hadamard.block_sizes(100) == [64, 32, 4]
    assert sum(hadamard.block_sizes(126)) == 126


@pytest.mark.parametrize("r", [2, 4, 6, 8, 18, 24, 64, 100, 126, 128])
def test_orthogonal(r):
    s = np.where(np.random.default_rng(r).integers(0, 2, r) == 1, 1, -1)
    H = hadamard.hadamard(r, s)
    assert np.abs(H @ H.T - np.eye(r)).max() < 1e-14
    assert np.abs(H.T @ H - np.eye(r)).max() < 1e-14


@pytest.mark.parametrize("r", [2, 8, 64, 128])
def test_power_of_two_entries_and_equalisation(r):
    """Rows of the scaled Walsh-Hadamard matrix have squared entries 1/r, so every rotated
    channel of diag(lambda) has variance mean(lambda)."""
    s = np.where(np.random.default_rng(7).integers(0, 2, r) == 1, 1, -1)
    H = hadamard.hadamard(r, s)
    assert np.allclose(H * H, 1.0 / r, atol=1e-15, rtol=0)
    lam = np.sort(np.random.default_rng(1).exponential(size=r))[::-1]
    C = H @ np.diag(lam) @ H.T
    assert np.allclose(np.diag(C), lam.mean(), rtol=1e-13, atol=0)


def test_block_equalisation_non_power_of_two():
    r = 18
    s = np.ones(r)
    H = hadamard.hadamard(r, s)
    lam = np.arange(r, 0, -1).astype(float)
    d = np.diag(H @ np.diag(lam) @ H.T)
    assert np.allclose(d[:16], lam[:16].mean(), rtol=1e-13)
    assert np.allclose(d[16:], lam[16:].mean(), rtol=1e-13)


def test_sign_flip_applies_to_columns():
    r = 4
    s = np.array([1, -1, 1, -1])
    H = hadamard.hadamard(r, s)
    assert np.allclose(H, hadamard.sylvester(4) / 2 * s[None, :])
