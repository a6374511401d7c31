"""One-time per-head calibration (Table alg:kvrobin steps 1, 2, 5, 6; App. F "Calibration").

  step 1  centred covariance of the head's calibration vectors -> eigenvalues lambda
          (descending) and eigenbasis U; query variance sigma_Q,i^2 in that basis.
  step 2  attention-KL weights w_i = sigma_Q,i^2 * lambda_i (Prop. kl-bound, Sec. 4
          "Reordering and plug-in") and reordering of the basis by w descending; the MSE
          objective uses w_i = lambda_i and keeps the eigen order.
  step 5  basis fusion W = U_r H_r^T (d x r), so that y = W^T x = H_r U_r^T x
          (App. A.1 "Y = H_r U_r^T X"; the step-5 formula in the table is read this way
          because r x r times d x r does not conform).
  step 6  stored per head: W (fp32), Delta (fp32), mu (fp32), r, b.

Readings: the covariance is the population (1/N) centred covariance; each eigenvector's
sign is fixed so that its largest-magnitude component is positive (first such index on a
tie); sigma_Q,i^2 = E[(u_i . q)^2] is the uncentred second moment over the calibration
queries of all G query heads sharing the KV head (mean over G); reordering is a stable sort
of -w; Delta uses the mean of the retained eigenvalues (see quantizer.step_size).
"""
from __future__ import annotations

import numpy as np

from . import hadamard, quantizer


def centred_covariance(x):
    x = np.asarray(x, dtype=np.float64)
    mu = x.mean(axis=0)
    xc = x - mu[None, :]
    return mu, (xc.T @ xc) / x.shape[0]


def eigenbasis(cov):
    """Eigenvalues descending and matching unit eigenvectors (columns) with the sign rule."""
    lam, U = np.linalg.eigh(cov)
    order = np.argsort(-lam, kind="stable")
    lam, U = lam[order], U[:, order].copy()
    for j in range(U.shape[1]):
        k = int(np.argmax(np.abs(U[:, j])))
        if U[k, j] < 0:
            U[:, j] = -U[:, j]
    return lam, U


def query_variance(U, q_cal):
    """sigma_Q,i^2 = mean over calibration queries of (u_i . q)^2; q_cal is (n, d) or
    (G, n, d) (pooled over the G query heads)."""
    qs = np.asarray(q_cal, dtype=np.float64).reshape(-1, U.shape[0])
    proj = qs @ U
    return (proj * proj).mean(axis=0)


def calibrate_head(x_cal, q_cal=None):
    """Steps 1-2 for one head.  Returns dict(mu, lam, U, w) with U's columns (and lam)
    in the order used by the allocator (w descending for KL, eigen order for MSE)."""
    mu, cov = centred_covariance(x_cal)
    lam, U = eigenbasis(cov)
    if q_cal is None:
        w = lam.copy()
        return dict(mu=mu, lam=lam, U=U, w=w, cov=cov)
    sq = query_variance(U, q_cal)
    w = sq * lam
    order = np.argsort(-w, kind="stable")
    return dict(mu=mu, lam=lam[order], U=U[:, order], w=w[order], cov=cov)


def fuse_basis(U, r: int, signs):
    """W = U_r H_r^T (d x r, fp64)."""
    if r == 0:
        return np.zeros((U.shape[0], 0))
    H = hadamard.hadamard(r, signs)
    return U[:, :r] @ H.T


def head_params(cal, r: int, b: int, signs):
    """Step 5-6: the stored per-head parameters (fp32 W, Delta, mu)."""
    W = fuse_basis(cal["U"], r, signs)
    delta = quantizer.step_size(cal["lam"][:r], b) if r > 0 else 0.0
    return dict(r=int(r), b=int(b), W=W.astype(np.float32), delta=np.float32(delta),
                mu=np.asarray(cal["mu"], dtype=np.float32))
