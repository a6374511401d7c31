"""Dequantise-on-read decode attention (Table alg:kvrobin step 8; App. G "Wall-clock at the
primitive level": dequantisation and the inverse rotation fused in one pass).

Plain definition (what the oracle checks the kernels against): reconstruct every cached
key and value from its codes, K_t = mu_K + W_K Delta_K (c_t - 2^{b-1} + 1/2) (likewise V),
then o_g = softmax(q_g . K / sqrt(d)) V for each query head g of the group (logits
s_t = <Q, K_t>/sqrt(d) as in Sec. 4).  fp64, max-subtracted softmax.

`rank_space` restates the same quantity the way the kernels evaluate it: scores from the
projected query q~ = (Delta_K / sqrt d) W_K^T q against the raw codes (the dropped terms are
constant in t, so softmax ignores them), values accumulated in rank space and mapped back
once by W_V.  It exists to pin that algebra against the plain definition.
"""
from __future__ import annotations

import math

import numpy as np

from . import quantizer


def reconstruct(codes, W, delta, b, mu):
    """X_t = mu + W Delta (c_t - 2^{b-1} + 1/2): [T, d] (fp64).  r = 0 gives mu."""
    codes = np.asarray(codes)
    T = codes.shape[0]
    mu = np.asarray(mu, dtype=np.float64)
    W = np.asarray(W, dtype=np.float64)
    if W.shape[1] == 0:
        return np.repeat(mu[None, :], T, axis=0)
    z = quantizer.dequantize(codes, float(delta), b)
    return mu[None, :] + z @ W.T


def softmax_attend(q, K, V):
    """o_g = softmax(q_g K^T / sqrt(d)) V for q [G, d], K/V [T, d]."""
    q = np.asarray(q, dtype=np.float64)
    d = q.shape[-1]
    s = (q @ np.asarray(K, dtype=np.float64).T) / math.sqrt(d)
    s = s - s.max(axis=1, keepdims=True)
    p = np.exp(s)
    p = p / p.sum(axis=1, keepdims=True)
    return p @ np.asarray(V, dtype=np.float64)


def decode(q, k_codes, v_codes, pk, pv):
    """Plain-definition decode for one KV head: q [G, d]; codes [T, r]; pk/pv hold W, delta,
    b, mu (the stored per-head parameters)."""
    K = reconstruct(k_codes, pk["W"], pk["delta"], pk["b"], pk["mu"])
    V = reconstruct(v_codes, pv["W"], pv["delta"], pv["b"], pv["mu"])
    return softmax_attend(q, K, V)


def rank_space(q, k_codes, v_codes, pk, pv):
    """The same output computed in rank space (see module docstring)."""
    q = np.asarray(q, dtype=np.float64)
    d = q.shape[-1]
    WK = np.asarray(pk["W"], dtype=np.float64)
    WV = np.asarray(pv["W"], dtype=np.float64)
    T = np.asarray(k_codes).shape[0]
    if WK.shape[1] == 0:
        s = np.zeros((q.shape[0], T))
    else:
        qt = (float(pk["delta"]) / math.sqrt(d)) * (q @ WK)
        s = qt @ np.asarray(k_codes, dtype=np.float64).T
    s = s - s.max(axis=1, keepdims=True)
    p = np.exp(s)
    ell = p.sum(axis=1, keepdims=True)
    mu = np.asarray(pv["mu"], dtype=np.float64)
    if WV.shape[1] == 0:
        return np.repeat(mu[None, :], q.shape[0], axis=0)
    acc = p @ np.asarray(v_codes, dtype=np.float64)
    zbar = float(pv["delta"]) * (acc / ell - ((1 << (pv["b"] - 1)) - 0.5))
    return mu[None, :] + zbar @ WV.T
