"""Decode attention with the rotary position embedding applied after reconstruction.

TEST INFRASTRUCTURE ONLY (see the package docstring).

The paper compresses K *before* the rotary embedding (Sec. 5, "Scope"; App. "Post-RoPE
experiments": after the rotation the per-head covariance depends on the position, so a
static basis fits it poorly).  A RoPE model then attends with the rotation applied to each
reconstructed key at its own position and to the query at its position:

    o_g = softmax_t( R(p) q_g . R(t) K^_t / sqrt(d) ) V^,
    K^_t = mu_K + W_K Delta_K (c_t - 2^{b-1} + 1/2)   (as attention.reconstruct)

Reading (the paper prints no rotation formula): the rotate-half form used by the models the
paper evaluates (Llama-3, Mistral, Qwen): channel j pairs with channel j + d/2, and pair j
turns by the angle pos * omega_j, omega_j = theta^(-2j/d) (theta = 500000 for Llama-3-8B).
Key t sits at position t (its index in the sequence); the query's position is an input.
Angles are taken in fp64 from exact integer positions.
"""
from __future__ import annotations

import numpy as np

from . import attention


def frequencies(d, theta):
    """omega_j = theta^(-2j/d), j = 0 .. d/2 - 1 (fp64)."""
    return np.power(float(theta), -2.0 * np.arange(d // 2, dtype=np.float64) / d)


def rotate(x, pos, theta):
    """R(pos) x for x [..., d] at positions pos (broadcast against x's leading axes):
    x cos + rotate_half(x) sin, rotate_half(x) = (-x[d/2:], x[:d/2]), with the angles
    pos * omega_j repeated over both halves."""
    x = np.asarray(x, dtype=np.float64)
    d = x.shape[-1]
    h = d // 2
    ang = np.asarray(pos, dtype=np.float64)[..., None] * frequencies(d, theta)
    c = np.concatenate([np.cos(ang), np.cos(ang)], axis=-1)
    s = np.concatenate([np.sin(ang), np.sin(ang)], axis=-1)
    rh = np.concatenate([-x[..., h:], x[..., :h]], axis=-1)
    return x * c + rh * s


def decode(q, k_codes, v_codes, pk, pv, q_pos, theta, k_pos=None):
    """RoPE decode for one KV head: q [G, d] at position q_pos, codes [T, r] of the keys at
    positions k_pos (default 0 .. T-1); pk / pv as for attention.decode."""
    K = attention.reconstruct(k_codes, pk["W"], pk["delta"], pk["b"], pk["mu"])
    V = attention.reconstruct(v_codes, pv["W"], pv["delta"], pv["b"], pv["mu"])
    T = K.shape[0]
    kp = np.arange(T) if k_pos is None else np.asarray(k_pos)
    return attention.softmax_attend(rotate(q, q_pos, theta), rotate(K, kp, theta), V)
