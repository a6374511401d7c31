"""Seeded synthetic inputs shaped like the KV-cache workloads of the paper.

This module only draws random data: spectra, rotations, key/value/query vectors, sign
vectors, sequence lengths and page tables.  It holds none of the method's arithmetic
(no covariance, eigen-decomposition, Hadamard fusion, allocation, quantisation or
packing), so it may feed both the CUDA path and the fp64 oracle.

Generator (per head):
  * spectrum  lambda_i = i**(-alpha), i = 1..d, rescaled so that sum(lambda) = d, with
    alpha ~ U[alpha_lo, alpha_hi] drawn per (layer, head, side);
  * rotation  R Haar-distributed (QR of a Gaussian matrix, column signs fixed by the sign of
    diag(R_qr));
  * outliers  4 distinct original coordinates are multiplied by 8;
  * vectors   x = S R diag(sqrt(lambda)) g with g ~ N(0, I), rounded to bf16.
Calibration tokens use their own stream; decode queries are N(0, I) bf16 (optionally
scaled); KL calibration queries use the same power-law generator with their own alpha.

Seeds: every stream is a numpy SeedSequence built from (2609, config, layer, head, side,
stream) so that any slice of a large workload can be regenerated independently.
"""
from __future__ import annotations

import numpy as np

BASE_SEED = 2609
D_HEAD = 128
N_OUTLIERS = 4
OUTLIER_SCALE = 8.0

# stream ids
S_SPECTRUM, S_ROTATION, S_OUTLIER, S_TOKENS, S_CALIB, S_QUERY, S_QCALIB, S_SIGNS, S_MISC = range(9)


def rng(config: int, layer: int, head: int, side: int, stream: int, extra: int = 0) -> np.random.Generator:
    """Independent numpy generator for one (config, layer, head, side, stream) tuple."""
    ss = np.random.SeedSequence([BASE_SEED, config, layer, head, side, stream, extra])
    return np.random.Generator(np.random.PCG64(ss))


def to_bf16(x: np.ndarray) -> np.ndarray:
    """Round float32/float64 values to the nearest bf16 (ties to even); returns float32
    values that are exactly representable in bf16."""
    f = np.ascontiguousarray(x, dtype=np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    bias = ((u >> 16) & 1) + 0x7FFF
    u = ((u + bias) & 0xFFFF0000).astype(np.uint32)
    return u.view(np.float32).reshape(f.shape)


def bf16_bits(x_bf16_valued: np.ndarray) -> np.ndarray:
    """uint16 bit patterns of float32 values that are exactly bf16."""
    f = np.ascontiguousarray(x_bf16_valued, dtype=np.float32)
    return (f.view(np.uint32) >> 16).astype(np.uint16)


def power_law_spectrum(alpha: float, d: int = D_HEAD) -> np.ndarray:
    lam = np.arange(1, d + 1, dtype=np.float64) ** (-alpha)
    return lam * (d / lam.sum())


def haar_orthogonal(g: np.random.Generator, d: int = D_HEAD) -> np.ndarray:
    a = g.standard_normal((d, d))
    q, r = np.linalg.qr(a)
    return q * np.sign(np.diag(r))[None, :]


class HeadSource:
    """The distribution of one head's K (or V) vectors: x = S R diag(sqrt(lambda)) g."""

    def __init__(self, config: int, layer: int, head: int, side: int, alpha_range, d: int = D_HEAD,
                 n_outliers: int = N_OUTLIERS):
        self.key = (config, layer, head, side)
        self.d = d
        a_lo, a_hi = alpha_range
        self.alpha = float(rng(config, layer, head, side, S_SPECTRUM).uniform(a_lo, a_hi))
        self.lam = power_law_spectrum(self.alpha, d)
        self.R = haar_orthogonal(rng(config, layer, head, side, S_ROTATION), d)
        scale = np.ones(d)
        idx = rng(config, layer, head, side, S_OUTLIER).choice(d, size=n_outliers, replace=False)
        scale[idx] = OUTLIER_SCALE
        self.outliers = np.sort(idx)
        # mixing matrix A so that x = A g
        self.A = (scale[:, None] * self.R) * np.sqrt(self.lam)[None, :]

    def sample(self, n: int, stream: int, extra: int = 0) -> np.ndarray:
        """n vectors (n x d), float32 values exactly representable in bf16."""
        g = rng(*self.key, stream, extra).standard_normal((n, self.d))
        return to_bf16(g @ self.A.T)

    def tokens(self, n: int, seq: int = 0) -> np.ndarray:
        return self.sample(n, S_TOKENS, seq)

    def calibration(self, n: int = 512) -> np.ndarray:
        return self.sample(n, S_CALIB)


def decode_queries(config: int, layer: int, kv_head: int, n_seqs: int, group: int, d: int = D_HEAD,
                   scale: float = 1.0) -> np.ndarray:
    """Decode queries for the `group` query heads that share one KV head: (n_seqs, group, d),
    N(0, scale^2 I) rounded to bf16."""
    g = rng(config, layer, kv_head, 0, S_QUERY).standard_normal((n_seqs, group, d)) * scale
    return to_bf16(g)


def calibration_queries(config: int, layer: int, kv_head: int, group: int, n: int, alpha_range,
                        d: int = D_HEAD) -> np.ndarray:
    """Calibration queries for the KL weights: (group, n, d), drawn per query head from the
    same power-law generator with their own alpha."""
    out = np.empty((group, n, d), dtype=np.float32)
    for gq in range(group):
        src = HeadSource(config, layer, 1000 + kv_head * group + gq, 2, alpha_range, d)
        out[gq] = src.sample(n, S_QCALIB)
    return out


def hadamard_signs(config: int, layer: int, head: int, side: int, d: int = D_HEAD) -> np.ndarray:
    """The random sign flip drawn once per head at calibration (+1/-1, int8, length d; the
    first r entries are used)."""
    g = rng(config, layer, head, side, S_SIGNS)
    return np.where(g.integers(0, 2, size=d) == 1, 1, -1).astype(np.int8)


def ragged_lengths(config: int, n_seqs: int, lo: int, hi: int) -> np.ndarray:
    """Sequence lengths uniform on the integers [lo, hi]."""
    return rng(config, 0, 0, 0, S_MISC, 1).integers(lo, hi + 1, size=n_seqs).astype(np.int32)


def shuffled_pages(config: int, n_pages: int) -> np.ndarray:
    """A seeded permutation of physical page ids 0..n_pages-1."""
    return rng(config, 0, 0, 0, S_MISC, 2).permutation(n_pages).astype(np.int32)


# The five workloads.  Each entry gives shapes, alpha ranges and the allocation recipe.
CONFIGS = {
    1: dict(name="tiny", layers=1, kv_heads=8, q_heads=32, seqs=1, tokens=2048,
            alpha=(0.5, 2.0), bpd=2.0, joint=False),
    2: dict(name="llama3-8b", layers=32, kv_heads=8, q_heads=32, seqs=8, tokens=32768,
            alpha=(0.3, 2.5), bpd=1.0, joint=False),
    3: dict(name="llama3-70b-joint", layers=80, kv_heads=8, q_heads=64, seqs=1, tokens=131072,
            alpha=(0.3, 2.5), bpd=0.5, joint=True),
    4: dict(name="prefill-compress", layers=32, kv_heads=8, q_heads=32, seqs=64, tokens=4096,
            alpha=(0.5, 2.0), bpd=4.0, joint=False),
    5: dict(name="ragged-sweep", layers=32, kv_heads=8, q_heads=32, seqs=32, tokens=(1024, 65536),
            alpha=(0.3, 2.5), bpd=(0.5, 1.0, 2.0, 3.0, 4.0), joint=False, page_tokens=256),
}
