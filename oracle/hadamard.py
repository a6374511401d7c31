"""Hadamard rotation fused into the retained basis (Sec. 3.4 "Per-channel equalization via
Hadamard rotation"; App. A.1; Lemma "head-level reconstruction MSE", step 4).

The paper uses the r x r Walsh-Hadamard matrix H_r, scaled so that H_r H_r^T = I, with a
random sign flip drawn once at calibration.  A Walsh-Hadamard matrix exists only for r a
power of two, while the C1 rank grid has step 2 (r = 18, 24, 100, ...).

Reading taken for other r: H_r = blockdiag(H_{2^k1}, H_{2^k2}, ...) . diag(s), one
normalised Sylvester block per binary digit of r, largest block first, s the +-1 sign
vector.  For power-of-two r this is exactly the scaled Walsh-Hadamard matrix with the sign
flip; for other r it is still orthogonal and equalises variance inside each block.
"""
from __future__ import annotations

import numpy as np


def sylvester(n: int) -> np.ndarray:
    """Unnormalised Sylvester-Hadamard matrix of order n (n a power of two), entries +-1:
    H_1 = [1], H_2n = [[H_n, H_n], [H_n, -H_n]]."""
    if n < 1 or (n & (n - 1)) != 0:
        raise ValueError("order must be a power of two")
    h = np.ones((1, 1))
    while h.shape[0] < n:
        h = np.block([[h, h], [h, -h]])
    return h


def block_sizes(r: int) -> list[int]:
    """Binary digits of r as block orders, largest first (r = 18 -> [16, 2])."""
    sizes = []
    bit = 1 << max(r.bit_length() - 1, 0)
    while bit:
        if r & bit:
            sizes.append(bit)
        bit >>= 1
    return sizes


def hadamard(r: int, signs) -> np.ndarray:
    """H_r (r x r, fp64) with H_r H_r^T = I: normalised Sylvester blocks times diag(signs[:r])."""
    h = np.zeros((r, r))
    o = 0
    for n in block_sizes(r):
        h[o:o + n, o:o + n] = sylvester(n) / np.sqrt(n)
        o += n
    s = np.asarray(signs[:r], dtype=np.float64)
    return h * s[None, :]
