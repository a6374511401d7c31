"""GPU parity of the device calibration (Table alg:kvrobin steps 1-2; cobra_calibrate_heads)
against the oracle's (oracle/calibrate.py: numpy's symmetric eigen-solver) and the library's
host calibration, on the Llama-3-8B model's heads: K heads with the attention-KL weights
(their group's calibration queries), V heads with the MSE weights.

Both sides work in fp64.  The eigenvalues agree to 1e-10 of the largest, the weights to 1e-9
relative, the directions (after the sign rule) to 1e-7 per component: an eigenvector moves by
about (rounding x |A|) / (gap to its neighbours), and the synthetic spectra keep relative gaps
above ~1e-3 down to the 128th eigenvalue.  The allocator's order of the directions must be the
same permutation."""
import numpy as np
import pytest
import torch

from oracle import calibrate as ocal
from paper_2609_24298_gb300 import cobra, pipeline, synth

from .gpu_util import DEV

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    cobra.lib()


def heads(cfg=2, layers=(0, 17), n_kv=8):
    spec = synth.CONFIGS[cfg]
    G = spec["q_heads"] // spec["kv_heads"]
    srcs, xs, qs = [], [], []
    for side in (0, 1):
        for l in layers:
            for h in range(n_kv):
                s = synth.HeadSource(cfg, l, h, side, spec["alpha"])
                srcs.append(s)
                xs.append(s.calibration(512))
                qs.append(synth.calibration_queries(cfg, l, h, G, 512, spec["alpha"]) if side == 0 else None)
    return srcs, xs, qs


def check(got, want):
    lmax = float(np.max(want["lam"]))
    np.testing.assert_allclose(got["mu"], want["mu"], rtol=0, atol=1e-12 * max(1.0, float(np.max(np.abs(want["mu"])))))
    np.testing.assert_allclose(got["lam"], want["lam"], rtol=0, atol=1e-10 * lmax)
    np.testing.assert_allclose(got["w"], want["w"], rtol=1e-9, atol=1e-12 * float(np.max(want["w"])))
    np.testing.assert_allclose(got["U"], want["U"], rtol=0, atol=1e-7)


def test_device_calibration_matches_oracle_and_host():
    srcs, xs, qs = heads()
    dev = pipeline.calibrate_heads_device(xs, qs, device=DEV)
    host = pipeline.calibrate_heads(xs, qs)
    for d, hcal, x, q in zip(dev, host, xs, qs):
        want = ocal.calibrate_head(np.asarray(x, np.float64), q)
        check(d, want)
        check(d, hcal)


def test_device_calibration_feeds_the_same_allocation():
    srcs, xs, qs = heads(layers=(3,))
    dev = pipeline.calibrate_heads_device(xs, qs, device=DEV)
    host = pipeline.calibrate_heads(xs, qs)
    n = len(xs) // 2
    for part in (slice(0, n), slice(n, 2 * n)):
        a = cobra.cobra_allocate(np.stack([c["w"] for c in dev[part]]), 1.0)
        b = cobra.cobra_allocate(np.stack([c["w"] for c in host[part]]), 1.0)
        assert np.array_equal(a["r"], b["r"]) and np.array_equal(a["b"], b["b"])
