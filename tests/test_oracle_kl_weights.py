"""Pin for the attention-KL weights of oracle.calibrate (Sec. 4, Prop. kl-bound and
"Reordering and plug-in"), independent of the formula the oracle uses.

The proposition's weight for direction u_i comes from the variance of the logit error
Delta s_t = Q . E_t / sqrt(d) when the key error E_t has variance sigma_K,i^2 along u_i:
the expected softmax KL is then proportional to E[(Q . u_i)^2] * sigma_K,i^2.  This test
measures that KL directly.  The clean keys are zero, so the clean attention is uniform for
every query and the second-order term is exact:

    E[KL(p || p~)] = (T - 1) / (2 T) * eps^2 / d * E_Q[(Q . u_i)^2] * lambda_i

for E_t = eps * eta_t * sqrt(lambda_i) * u_i with eta_t ~ N(0, 1) independent over tokens.
The KL is summed over the G query heads that share the kv head, so the query moment is the
uncentred second moment pooled over all of the group's calibration queries.

A tiny head (d = 8, G = 2) with query means far from zero and two query heads of very
different scale makes the alternative readings fail: a centred variance, or the moment of
one query head alone, misses the measured KL by far more than the tolerance (checked below,
so the test keeps its power).
"""
import numpy as np
import pytest
from scipy.special import logsumexp

from oracle import calibrate

D = 8
G = 2
N_Q = 3000        # calibration queries per query head
T = 64            # tokens of the synthetic cache
EPS = 1e-3        # key-error scale: logit errors stay ~1e-2, so the quartic term is ~1e-4


def _setup():
    rng = np.random.default_rng(24298)
    # keys: distinct eigenvalues, rotated
    lam = np.array([9.0, 6.0, 4.0, 2.5, 1.6, 1.0, 0.6, 0.3])
    R, _ = np.linalg.qr(rng.standard_normal((D, D)))
    x_cal = (rng.standard_normal((20000, D)) * np.sqrt(lam)) @ R.T + 0.2
    # queries: large means along a few key directions, and two heads of different scale
    m0 = 3.0 * R[:, 6] - 2.0 * R[:, 1]
    m1 = 1.5 * R[:, 3]
    q0 = m0 + rng.standard_normal((N_Q, D)) * np.array([0.3, 1.0, 0.5, 0.2, 0.8, 0.4, 0.6, 0.3])
    q1 = m1 + 2.5 * rng.standard_normal((N_Q, D)) @ np.diag([1.0, 0.2, 0.7, 0.3, 1.2, 0.5, 0.1, 0.9])
    q_cal = np.stack([q0, q1])  # (G, n, d)
    return rng, x_cal, q_cal


def _measured_kl(rng, q_pooled, u, lam_i):
    """Monte-Carlo E[KL(uniform || softmax(Delta s))] over the pooled queries, one error draw
    per query, and the second-order prediction's query factor recovered from it."""
    proj = q_pooled @ u                                   # (n,)
    eta = rng.standard_normal((q_pooled.shape[0], T))     # (n, T)
    ds = (EPS * np.sqrt(lam_i) / np.sqrt(D)) * proj[:, None] * eta
    # KL(p || p~) with p uniform: log-sum-exp(ds) - log T - mean(ds)
    kl = logsumexp(ds, axis=1) - np.log(T) - ds.mean(axis=1)
    # E[KL] / ((T - 1)/(2T) eps^2 / d) estimates E[(Q . u)^2] * lambda_i
    return kl.mean() / ((T - 1) / (2 * T) * EPS ** 2 / D)


def test_kl_weights_match_measured_attention_kl():
    rng, x_cal, q_cal = _setup()
    cal = calibrate.calibrate_head(x_cal, q_cal)
    U, lam, w = cal["U"], cal["lam"], cal["w"]
    q_pooled = q_cal.reshape(-1, D)
    measured = np.array([_measured_kl(rng, q_pooled, U[:, j], lam[j]) for j in range(D)])

    # the oracle's weights follow the measured KL direction by direction (Monte-Carlo
    # noise ~ sqrt(2 / (T - 1)) / sqrt(G * N_Q) ~ 0.3 %)
    rel = np.abs(w / measured - 1.0)
    assert rel.max() < 0.03, (w, measured)
    # the reorder is by measured importance: every pair of directions whose weights differ
    # by more than 10 % is in the measured order
    for i in range(D):
        for j in range(i + 1, D):
            if w[i] > 1.1 * w[j]:
                assert measured[i] > measured[j]

    # the alternative readings are far off, so the check above has power
    proj = q_cal @ U                                       # (G, n, d)
    centred = proj.reshape(-1, D).var(axis=0) * lam
    head0 = (proj[0] ** 2).mean(axis=0) * lam
    assert np.abs(centred / measured - 1.0).max() > 0.3
    assert np.abs(head0 / measured - 1.0).max() > 0.3


@pytest.mark.parametrize("g_only", [0, 1])
def test_one_query_head_group(g_only):
    """With a single query head the pooled moment is that head's moment."""
    rng, x_cal, q_cal = _setup()
    q1 = q_cal[g_only]
    cal = calibrate.calibrate_head(x_cal, q1)
    measured = np.array([_measured_kl(rng, q1, cal["U"][:, j], cal["lam"][j]) for j in range(D)])
    assert np.abs(cal["w"] / measured - 1.0).max() < 0.04
