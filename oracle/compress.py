"""Per-token compression, Table alg:kvrobin step 7: z_t = quantize(V^T K_t, b*), with the
projection and the Hadamard rotation applied as one multiply by the fused basis W = U_r H_r^T
(Sec. 3.4 "zero latency").  The calibration mean is removed first (the covariances of
step 1 are centred), so y = W^T (x - mu).  fp64 throughout; W, mu and Delta are the stored
fp32 values and x the bf16 input values.
"""
from __future__ import annotations

import numpy as np

from . import quantizer


def project(x, W, mu):
    """y = (x - mu) W  for token vectors x [T, d]; W [d, r]."""
    x = np.asarray(x, dtype=np.float64)
    return (x - np.asarray(mu, dtype=np.float64)[None, :]) @ np.asarray(W, dtype=np.float64)


def compress(x, W, mu, delta, b):
    """Returns (u, codes): the pre-rounding values u = y/Delta + 2^{b-1} and the codes."""
    r = np.asarray(W).shape[1]
    if r == 0:
        T = np.asarray(x).shape[0]
        return np.zeros((T, 0)), np.zeros((T, 0), dtype=np.int64)
    y = project(x, W, mu)
    u = quantizer.pre_round(y, float(delta), b)
    return u, np.clip(np.floor(u), 0, (1 << b) - 1).astype(np.int64)
