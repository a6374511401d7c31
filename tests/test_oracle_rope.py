"""Pins for oracle.rope (decode with the rotary embedding applied after reconstruction; the
paper compresses K before it, Sec. 5 "Scope") against what the mathematics fixes: the
complex-multiplication form of the rotation, closed forms in two and four dimensions, the
frequency ladder's end points, the direction of the turn, norm preservation and composition,
dependence on relative position only, a brute-force loop with explicit 2 x 2 rotations, and
the special cases position 0, T = 1 and a zero key."""
import math

import numpy as np
import pytest

from oracle import attention, rope

from .test_oracle_attention import setup_decode


def test_zero_position_is_the_identity():
    g = np.random.default_rng(1)
    x = g.standard_normal((7, 128))
    assert np.array_equal(rope.rotate(x, 0, 500000.0), x)
    q, ck, cv, pk, pv, _, _ = setup_decode(90, 32, 3, 48, 2)
    a = rope.decode(q, ck, cv, pk, pv, 0, 500000.0, k_pos=np.zeros(90))
    assert np.array_equal(a, attention.decode(q, ck, cv, pk, pv))


def test_complex_multiplication_form():
    """Pair j = (x_j, x_{j+d/2}) read as x_j + i x_{j+d/2} is multiplied by exp(i pos omega_j)."""
    g = np.random.default_rng(2)
    x = g.standard_normal((5, 128))
    pos = np.array([0, 1, 17, 4095, 32767])
    theta = 500000.0
    om = theta ** (-np.arange(64) / 64.0)
    z = (x[:, :64] + 1j * x[:, 64:]) * np.exp(1j * pos[:, None] * om[None, :])
    want = np.concatenate([z.real, z.imag], axis=1)
    assert np.abs(rope.rotate(x, pos, theta) - want).max() < 1e-12


def test_closed_forms_in_two_and_four_dimensions():
    # d = 2: one pair at omega_0 = 1 turns by pos radians
    c3, s3 = -0.9899924966004454, 0.1411200080598672  # cos 3, sin 3
    assert np.allclose(rope.rotate(np.array([1.0, 0.0]), 3, 10.0), [c3, s3], rtol=0, atol=1e-15)
    assert np.allclose(rope.rotate(np.array([0.0, 1.0]), 3, 10.0), [-s3, c3], rtol=0, atol=1e-15)
    # d = 4, theta = 100: omega = (1, 1/10); e_1 is the first half of pair 1 -> dims 1 and 3
    c5, s5 = 0.8775825618903728, 0.479425538604203  # cos 0.5, sin 0.5
    assert np.allclose(rope.rotate(np.array([0.0, 1.0, 0.0, 0.0]), 5, 100.0), [0.0, c5, 0.0, s5], rtol=0, atol=1e-15)


def test_frequency_ladder():
    om = rope.frequencies(128, 10000.0)
    assert om[0] == 1.0
    assert abs(om[32] - 0.01) < 1e-17  # theta^(-1/2) at j = d/4
    assert abs(om[63] - 10000.0 ** (-126 / 128)) < 1e-18
    assert np.all(np.diff(om) < 0)


@pytest.mark.parametrize("j", [0, 5, 63])
def test_direction_of_the_turn(j):
    """<R(p) e_j, R(t) e_j> = cos(omega_j (t - p)) and <R(p) e_{j+64}, R(t) e_j> = sin(omega_j (t - p))."""
    theta, p, t = 500000.0, 700, 1234
    om = rope.frequencies(128, theta)[j]
    e = np.eye(128)
    kt = rope.rotate(e[j], t, theta)
    assert abs(rope.rotate(e[j], p, theta) @ kt - math.cos(om * (t - p))) < 1e-12
    assert abs(rope.rotate(e[j + 64], p, theta) @ kt - math.sin(om * (t - p))) < 1e-12


def test_norm_and_composition():
    g = np.random.default_rng(3)
    x = g.standard_normal((4, 128))
    a, b, theta = 1000, 23, 500000.0
    ra = rope.rotate(x, a, theta)
    assert np.allclose(np.linalg.norm(ra, axis=1), np.linalg.norm(x, axis=1), rtol=1e-14)
    assert np.abs(rope.rotate(rope.rotate(x, b, theta), a, theta) - rope.rotate(x, a + b, theta)).max() < 1e-11


def test_only_relative_positions_matter():
    q, ck, cv, pk, pv, _, _ = setup_decode(200, 64, 2, 32, 3)
    theta = 500000.0
    a = rope.decode(q, ck, cv, pk, pv, 199, theta)
    b = rope.decode(q, ck, cv, pk, pv, 199 + 5000, theta, k_pos=np.arange(200) + 5000)
    assert np.abs(a - b).max() < 1e-9 * np.abs(a).max()
    # and the rotation does change the result
    assert np.abs(a - attention.decode(q, ck, cv, pk, pv)).max() > 1e-3 * np.abs(a).max()


def test_brute_force_loops_on_a_tiny_head():
    """Explicit 2 x 2 rotations of every pair, scores, softmax and weighted sum in Python loops."""
    g = np.random.default_rng(4)
    d, T, G, theta, p = 8, 5, 2, 50.0, 9
    q, K, V = g.standard_normal((G, d)), g.standard_normal((T, d)), g.standard_normal((T, d))
    h = d // 2

    def turn(x, pos):
        out = list(x)
        for j in range(h):
            ang = pos * theta ** (-2.0 * j / d)
            c, s = math.cos(ang), math.sin(ang)
            out[j] = c * x[j] - s * x[j + h]
            out[j + h] = s * x[j] + c * x[j + h]
        return out

    want = np.zeros((G, d))
    for gi in range(G):
        qr = turn(q[gi], p)
        sc = [sum(a * b for a, b in zip(qr, turn(K[t], t))) / math.sqrt(d) for t in range(T)]
        m = max(sc)
        w = [math.exp(s - m) for s in sc]
        for t in range(T):
            for i in range(d):
                want[gi, i] += w[t] / sum(w) * V[t, i]
    got = attention.softmax_attend(rope.rotate(q, p, theta), rope.rotate(K, np.arange(T), theta), V)
    assert np.abs(got - want).max() < 1e-13


def test_single_token_and_zero_key():
    q, ck, cv, pk, pv, _, _ = setup_decode(1, 32, 3, 32, 3)
    o = rope.decode(q, ck, cv, pk, pv, 41, 500000.0)
    v0 = attention.reconstruct(cv, pv["W"], pv["delta"], 3, pv["mu"])[0]
    assert np.abs(o - v0[None, :]).max() < 1e-12
    # r_K = 0 with mu_K = 0: every rotated key is zero, so attention is uniform
    q, ck, cv, pk, pv, _, _ = setup_decode(77, 0, 0, 32, 3)
    pk = dict(pk, mu=np.zeros_like(pk["mu"]))
    o = rope.decode(q, ck, cv, pk, pv, 76, 500000.0)
    V = attention.reconstruct(cv, pv["W"], pv["delta"], 3, pv["mu"])
    assert np.abs(o - V.mean(0)[None, :]).max() < 1e-12
