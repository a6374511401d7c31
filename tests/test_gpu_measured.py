"""GPU parity of the measured distortion tables (App. E, "Exact DP over measured distortion"):
cobra_measure_distortion against the oracle's tables (oracle/measured.py) on the same
calibration tokens and per-head calibration, for the MSE and attention-KL weights, over the
allocator's whole candidate grid, and the exact DP on the device tables against the DP on the
oracle's tables.

Tolerance: the device works in fp32 (eigen coordinates by an fp32 GEMM, the Hadamard by fp32
butterflies) where the oracle works in fp64 from the stored fp32 basis: each entry agrees to a
relative 1e-4 (sums of 512 x 128 squared errors whose terms carry ~1e-6 relative rounding),
plus what a few codes flipping at a cell boundary can move it.  A flip turns one rotated
error eps_j = +Delta/2 into -Delta/2, so e = H_r^T eps moves by Delta along a unit vector and
the token's weighted error by at most 2 Delta |e|_w sqrt(max w) + Delta^2 max w, with
|e|_w <= sqrt(r max w) Delta (each |eps_j| <= Delta/2 inside the clip range); divided by the
512 tokens and allowed 4 times."""
import numpy as np
import pytest
import torch

from oracle import calibrate as ocal
from oracle import measured as om
from oracle import quantizer as oq
from paper_2609_24298_gb300 import cobra, synth

from .gpu_util import DEV

pytestmark = pytest.mark.gpu
RTOL = 1e-4


@pytest.fixture(scope="module", autouse=True)
def need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    cobra.lib()


def heads(cfg, n, kl):
    spec = synth.CONFIGS[cfg]
    out = []
    for h in range(n):
        src = synth.HeadSource(cfg, 1, h, 0 if kl else 1, spec["alpha"])
        x = src.calibration(512)
        qc = synth.calibration_queries(cfg, 1, h, 4, 512, spec["alpha"]) if kl else None
        cal = ocal.calibrate_head(x, qc)
        out.append((x, cal, om.error_weights(cal, qc), synth.hadamard_signs(*src.key)))
    return out


def tolerance(hs, rg, bg, want):
    """Per-entry tolerance (module docstring)."""
    tol = np.zeros_like(want)
    for h, (x, cal, omega, _) in enumerate(hs):
        wmax = float(np.max(omega))
        for i, r in enumerate(rg):
            for j, b in enumerate(bg):
                if r == 0:
                    tol[h, i, j] = RTOL * want[h, i, j]
                    continue
                dl = float(np.float32(oq.step_size(cal["lam"][:r], b)))
                flip = 2 * dl * np.sqrt(r) * dl * wmax + dl * dl * wmax
                tol[h, i, j] = RTOL * want[h, i, j] + 4 * flip / x.shape[0]
    return tol


def assert_tables(got, want, tol):
    bad = np.abs(got - want) > tol
    assert not bad.any(), [(tuple(i), got[tuple(i)], want[tuple(i)], tol[tuple(i)]) for i in np.argwhere(bad)[:5]]


def device_tables(hs, rg, bg):
    f32 = lambda a: torch.tensor(np.stack(a), dtype=torch.float32, device=DEV).contiguous()
    x = f32([h[0] for h in hs])
    U = f32([h[1]["U"].T.reshape(-1) for h in hs])  # row k of U^T = column k of U
    f64 = lambda a: torch.tensor(np.stack(a), dtype=torch.float64, device=DEV).contiguous()
    lam = f64([h[1]["lam"] for h in hs])
    w = f64([h[1]["w"] for h in hs])
    mu = f32([h[1]["mu"] for h in hs])
    signs = torch.tensor(np.stack([h[3] for h in hs]), dtype=torch.int8, device=DEV).contiguous()
    coords = torch.empty((len(hs), x.shape[1], 128), dtype=torch.float32, device=DEV)
    D = torch.full((len(hs), len(rg), len(bg)), float("nan"), dtype=torch.float64, device=DEV)
    cobra.cobra_measure_distortion(x, U, lam, w, mu, signs, rg, bg, coords, D)
    torch.cuda.synchronize()
    return D.cpu().numpy()


@pytest.mark.parametrize("kl", [False, True])
def test_tables_match_oracle_on_a_grid(kl):
    hs = heads(2, 4, kl)
    rg, bg = [0, 2, 18, 32, 64, 100, 126, 128], [1, 2, 3, 5, 8]
    got = device_tables(hs, rg, bg)
    want = np.stack([om.measured_table(x, c, w, s, rg, bg) for x, c, w, s in hs])
    assert_tables(got, want, tolerance(hs, rg, bg, want))


def test_full_candidate_grid_and_dp():
    hs = heads(1, 2, True)
    rg, bg = om.default_grids()
    got = device_tables(hs, rg, bg)
    want = np.stack([om.measured_table(x, c, w, s, rg, bg) for x, c, w, s in hs])
    assert_tables(got, want, tolerance(hs, rg, bg, want))
    for bpd in (0.5, 1.0, 2.0):
        a = cobra.cobra_allocate_tables(got, rg, bg, bpd)
        r, b, _, tot = om.exact_dp_tables(list(want), rg, bg, len(hs) * 128 * bpd)
        if list(a["r"]) != r or list(a["b"]) != b:
            # a near-tie decided the other way: the device's choice must be as good on the
            # oracle's tables up to the tolerance
            alt = sum(want[h][rg.index(int(a["r"][h]))][bg.index(int(a["b"][h])) if a["r"][h] else 0]
                      for h in range(len(hs)))
            assert alt <= tot * (1 + 1e-3)


def test_measured_allocation_end_to_end():
    """App. E's allocator on the tiny model (1 layer x 8 kv heads, K with attention-KL weights,
    V with MSE weights, 2 bpd): the library's calibration, device tables and table DP give the
    oracle's allocation from the oracle's calibration and tables (or an equally good
    near-tie), and a cache built with that allocation decodes within the decode tolerance."""
    from paper_2609_24298_gb300 import pipeline

    from .gpu_util import oracle_calibrations
    from .test_gpu_fullsize import run_workload

    cfg, bpd = 1, 2.0
    cals, srcs = oracle_calibrations(cfg, 1)
    spec = synth.CONFIGS[cfg]
    qs = [synth.calibration_queries(cfg, s.key[1], s.key[2], spec["q_heads"] // spec["kv_heads"], 512, spec["alpha"])
          if s.key[3] == 0 else None for s in srcs]
    lib_cals = pipeline.calibrate_heads([s.calibration(512) for s in srcs], qs)
    r, b = pipeline.measured_allocation(lib_cals, srcs, bpd, device=DEV)
    rg, bg = om.default_grids()
    n = len(cals) // 2
    for side in (0, 1):
        part = slice(side * n, (side + 1) * n)
        tabs = [om.measured_table(s.calibration(512), c, om.error_weights(c, q), synth.hadamard_signs(*s.key), rg, bg)
                for c, s, q in zip(cals[part], srcs[part], qs[part])]
        ro, bo, _, tot = om.exact_dp_tables(tabs, rg, bg, n * 128 * bpd)
        if list(r[part]) != ro or list(b[part]) != bo:
            alt = sum(t[rg.index(int(rr))][bg.index(int(bb)) if rr else 0] for t, rr, bb in zip(tabs, r[part], b[part]))
            assert alt <= tot * (1 + 1e-3)
    params = [ocal.head_params(c, int(rr), int(bb) if rr else 1, synth.hadamard_signs(*s.key))
              for c, s, rr, bb in zip(cals, srcs, r, b)]
    run_workload(cfg, 1, params, srcs, [2048], [(0, h, 0) for h in range(8)])
