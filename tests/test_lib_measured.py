"""CPU tests of the library's exact DP over explicit distortion tables (App. E, "Exact DP over
measured distortion"): it makes the oracle's choices exactly, on random tables and on the
oracle's measured tables of real synthetic heads, and rejects malformed input."""
import os

import numpy as np
import pytest

from oracle import calibrate as ocal
from oracle import measured as om
from paper_2609_24298_gb300 import cobra, synth


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not os.path.exists(cobra.LIB_PATH):
        from paper_2609_24298_gb300 import build

        build.build()
    cobra.lib()


def check_same(tables, rg, bg, bpd, d):
    got = cobra.cobra_allocate_tables(tables, rg, bg, bpd, d)
    r, b, D, tot = om.exact_dp_tables(list(tables), rg, bg, len(tables) * d * bpd)
    assert list(got["r"]) == r and list(got["b"]) == b
    assert list(got["dist"]) == D
    assert got["rate_bits"] == sum(x * y for x, y in zip(r, b))


def test_random_tables_match_oracle():
    rng = np.random.default_rng(5)
    rg, bg = [0, 2, 4, 6, 8], list(range(1, 9))
    for trial in range(10):
        n = int(rng.integers(1, 7))
        t = rng.random((n, len(rg), len(bg)))
        # fewer bits never help: distortion falls along r * b, with ties planted
        t = np.sort(t.reshape(n, -1), axis=1)[:, ::-1].reshape(n, len(rg), len(bg)).copy()
        t[:, :, 3] = t[:, :, 2]
        for bpd in (0.0, 0.3, 1.0, 2.5, 8.0):
            check_same(t, rg, bg, bpd, 8)


def test_measured_tables_of_synthetic_heads_match_oracle():
    spec = synth.CONFIGS[1]
    rg, bg = [0, 2, 4, 8, 16, 32], [1, 2, 3, 4]
    tables = []
    for h in range(4):
        src = synth.HeadSource(1, 0, h, 1, spec["alpha"])
        x = src.calibration(256)
        cal = ocal.calibrate_head(x)
        tables.append(om.measured_table(x, cal, om.error_weights(cal), synth.hadamard_signs(*src.key), rg, bg))
    for bpd in (0.25, 0.5, 1.0, 2.0):
        check_same(np.stack(tables), rg, bg, bpd, 128)


def test_table_argument_checks():
    t = np.ones((1, 2, 2))
    with pytest.raises(cobra.CobraError) as e:
        cobra.cobra_allocate_tables(t, [2, 0], [1, 2], 1.0, 8)  # r not ascending
    assert e.value.status == cobra.COBRA_EINVAL
    with pytest.raises(cobra.CobraError) as e:
        cobra.cobra_allocate_tables(t, [0, 2], [2, 2], 1.0, 8)  # b not strictly ascending
    assert e.value.status == cobra.COBRA_EINVAL
    bad = t.copy()
    bad[0, 1, 1] = np.nan
    with pytest.raises(cobra.CobraError) as e:
        cobra.cobra_allocate_tables(bad, [0, 2], [1, 2], 1.0, 8)
    assert e.value.status == cobra.COBRA_EINVAL
    with pytest.raises(cobra.CobraError) as e:
        cobra.cobra_allocate_tables(t, [0, 9], [1, 2], 1.0, 8)  # r > d
    assert e.value.status == cobra.COBRA_EINVAL


def test_device_entry_points_check_arguments_before_the_gpu():
    # cobra_measure_distortion and cobra_calibrate_heads validate sizes, lists and alignment on
    # the host and return before any launch (fake device addresses are never touched)
    L = cobra.lib()
    import ctypes

    def measure(n_heads=1, n_tok=4, r=(0, 2), b=(1, 2), x=256, D=256):
        rl = (ctypes.c_int * len(r))(*r)
        bl = (ctypes.c_int * len(b))(*b)
        return L.cobra_measure_distortion(n_heads, n_tok, x, 256, 256, 256, 256, 256, len(r), rl, len(b), bl, 256, D,
                                          None)

    assert measure(r=()) == cobra.COBRA_EINVAL
    assert measure(r=tuple(range(0, 132, 2))) == cobra.COBRA_EINVAL  # 66 ranks
    assert measure(r=(4, 2)) == cobra.COBRA_EINVAL  # not ascending
    assert measure(r=(0, 130)) == cobra.COBRA_EINVAL  # r > 128
    assert measure(b=(0,)) == cobra.COBRA_EINVAL
    assert measure(b=(9,)) == cobra.COBRA_EINVAL
    assert measure(n_tok=0) == cobra.COBRA_EINVAL
    assert measure(x=258) == cobra.COBRA_EALIGN
    assert measure(D=260) == cobra.COBRA_EALIGN

    def calib(n_heads=1, n_tok=4, n_q=0, q=None, x=256, mu=256):
        return L.cobra_calibrate_heads(n_heads, n_tok, x, n_q, q, mu, 256, 256, 256, None)

    assert calib(n_tok=0) == cobra.COBRA_EINVAL
    assert calib(n_heads=0) == cobra.COBRA_EINVAL
    assert calib(n_q=3, q=None) == cobra.COBRA_EINVAL
    assert calib(x=258) == cobra.COBRA_EALIGN
    assert calib(mu=260) == cobra.COBRA_EALIGN
