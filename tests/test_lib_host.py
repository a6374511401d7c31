"""CPU tests of libcobra: the library loads and exports every symbol include/cobra.h
declares; its host-side allocator reproduces the oracle's integer allocation exactly; its
calibration, Hadamard, loading factor, fusion and layout agree with the oracle; argument
checks reject bad input without touching a GPU."""
import ctypes
import os
import re

import numpy as np
import pytest

from oracle import allocator as oal
from oracle import calibrate as ocal
from oracle import hadamard as ohad
from oracle import layout as olay
from oracle import quantizer as oq
from paper_2609_24298_gb300 import cobra, synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def L():
    if not os.path.exists(cobra.LIB_PATH):
        from paper_2609_24298_gb300 import build

        build.build()
    return cobra.lib()


def header_functions():
    src = open(os.path.join(ROOT, "include", "cobra.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(cobra_[a-z0-9_]+)\s*\(", src)))


def test_every_declared_symbol_is_exported(L):
    names = header_functions()
    assert len(names) >= 18
    for n in names:
        assert hasattr(L, n), n
        assert n in cobra.SIGNATURES, n


def test_version_and_strings(L):
    assert cobra.cobra_version() == 1
    assert cobra.status_string(cobra.COBRA_ETIMEOUT) == "device wait timed out"


def spectra(n, d, seed, lo=0.3, hi=2.5):
    g = np.random.default_rng(seed)
    out = []
    for _ in range(n):
        a = g.uniform(lo, hi)
        lam = np.arange(1, d + 1) ** (-a)
        out.append(lam * d / lam.sum())
    return np.array(out)


@pytest.mark.parametrize("bpd,seed", [(0.5, 0), (1.0, 1), (2.0, 2), (3.0, 3), (4.0, 4)])
def test_damped_allocation_matches_oracle_bit_for_bit(L, bpd, seed):
    W = spectra(96, 128, seed)
    got = cobra.cobra_allocate(W, bpd)
    want = oal.allocate(W, bpd)
    assert np.array_equal(got["r"], want["r"])
    assert np.array_equal(got["b"], want["b"])
    assert np.array_equal(got["budget"], want["budget"])
    assert np.array_equal(got["dist"], want["dist"])
    assert got["rate_bits"] == want["rate_bits"]


@pytest.mark.parametrize("mode", [oal.MODE_UNIFORM, oal.MODE_EXACT])
def test_other_modes_match_oracle(L, mode):
    W = spectra(6, 16, 9, 0.2, 3.0)
    for bpd in (0.5, 1.0, 2.5):
        got = cobra.cobra_allocate(W, bpd, cobra.alloc_opts(mode=mode))
        want = oal.allocate(W, bpd, oal.Opts(mode=mode))
        assert np.array_equal(got["r"], want["r"]) and np.array_equal(got["b"], want["b"])
        assert np.array_equal(got["dist"], want["dist"])


def test_paper_grid_options_match_oracle(L):
    W = spectra(32, 128, 12)
    got = cobra.cobra_allocate(W, 1.0, cobra.alloc_opts(b_min=2, allow_r0=0, complete=0))
    want = oal.allocate(W, 1.0, oal.Opts(b_min=2, allow_r0=False, complete=False))
    assert np.array_equal(got["r"], want["r"]) and np.array_equal(got["b"], want["b"])


def test_allocation_on_calibrated_config1(L):
    spec = synth.CONFIGS[1]
    ws = []
    for h in range(8):
        src = synth.HeadSource(1, 0, h, 0, spec["alpha"])
        ws.append(ocal.calibrate_head(src.calibration(512), synth.calibration_queries(1, 0, h, 4, 512, spec["alpha"]))["w"])
    W = np.stack(ws)
    got = cobra.cobra_allocate(W, 2.0)
    want = oal.allocate(W, 2.0)
    assert np.array_equal(got["r"], want["r"]) and np.array_equal(got["b"], want["b"])


def test_loading_factor_and_hadamard_match_oracle(L):
    for b in range(1, 9):
        assert abs(cobra.cobra_loading_factor(b) - oq.loading_factor(b)) < 1e-12
    for r in (2, 6, 18, 64, 100, 128):
        s = synth.hadamard_signs(1, 0, r, 0)[:r]
        assert np.abs(cobra.cobra_hadamard(r, s) - ohad.hadamard(r, s)).max() < 1e-15


@pytest.mark.parametrize("kl", [False, True])
def test_calibration_matches_oracle(L, kl):
    src = synth.HeadSource(1, 0, 3, 0, (0.5, 2.0))
    x = src.calibration(512)
    q = synth.calibration_queries(1, 0, 3, 4, 512, (0.5, 2.0)) if kl else None
    got = cobra.cobra_calibrate_head(x, q)
    want = ocal.calibrate_head(x, q)
    scale = want["lam"].max()
    assert np.abs(got["mu"] - want["mu"]).max() < 1e-12
    assert np.abs(got["lam"] - want["lam"]).max() < 1e-10 * scale
    assert np.abs(got["w"] - want["w"]).max() < 1e-9 * want["w"].max()
    # eigenvectors of well-separated eigenvalues agree (same sign rule)
    gap = np.abs(np.diff(np.sort(want["lam"])))
    for j in range(16):
        assert np.abs(got["U"][:, j] - want["U"][:, j]).max() < 1e-7
    s = synth.hadamard_signs(*src.key)
    for r, b in ((32, 3), (64, 2), (128, 1), (18, 5)):
        Wg, dg = cobra.cobra_fuse_basis(got["U"], got["lam"], r, b, s)
        pw = ocal.head_params(want, r, b, s)
        assert abs(float(dg) - float(pw["delta"])) <= 1e-6 * float(pw["delta"])
        assert np.abs(Wg[:, :16] - pw["W"][:, :16]).max() < 1e-6


def test_layout_plan_matches_oracle(L):
    r = np.array([128, 0, 2, 18, 64], np.int32)
    b = np.array([1, 3, 1, 3, 8], np.int32)
    offs, tot = cobra.cobra_plan_layout(r, b, 7)
    o2, t2 = olay.plan_regions(r, b, 7)
    assert list(offs) == list(o2) and tot == t2
    for rr, bb in zip(r, b):
        assert cobra.cobra_row_bytes(int(rr), int(bb)) == (olay.row_bytes(int(rr), int(bb)) if rr else 0)


def test_argument_checks_reject_bad_input(L):
    with pytest.raises(cobra.CobraError) as e:
        cobra.cobra_allocate(np.full((2, 8), np.nan), 1.0)
    assert e.value.status == cobra.COBRA_EINVAL
    with pytest.raises(cobra.CobraError):
        cobra.cobra_allocate(np.ones((2, 8)), 1.0, cobra.alloc_opts(b_min=5, b_max=2))
    with pytest.raises(cobra.CobraError) as e:
        cobra.cobra_plan_layout(np.array([3], np.int32), np.array([2], np.int32), 4)  # odd rank
    assert e.value.status == cobra.COBRA_EINVAL
    with pytest.raises(cobra.CobraError):
        cobra.cobra_loading_factor(9)
    # device entry points check arguments before touching the GPU
    d = cobra.compress_desc(head0=0, layer_stride=1, n_layers=1, n_kv_heads=1, side=0, n_seqs=1, rows_per_seq=1)
    with pytest.raises(cobra.CobraError) as e:
        cobra.cobra_compress(256, d, 256, 64, 10, 256)  # t0 not a multiple of 128
    assert e.value.status == cobra.COBRA_EINVAL
    with pytest.raises(cobra.CobraError) as e:
        cobra.cobra_compress(256, d, 258, 0, 10, 256)  # x not 16-byte aligned
    assert e.value.status == cobra.COBRA_EALIGN
    with pytest.raises(cobra.CobraError) as e:
        cobra.cobra_compress(256, d, 256, 0, 300, 256)  # more rows than rows_per_seq
    assert e.value.status == cobra.COBRA_EINVAL
    dd = cobra.decode_desc(k_head0=0, v_head0=1, layer_stride=1, n_layers=1, n_kv_heads=1, group=3, n_seqs=1,
                           rows_per_seq=1)
    with pytest.raises(cobra.CobraError):
        cobra.cobra_decode_workspace_size(dd, np.array([2, 2]), np.array([1, 1]), np.array([10]))
    # the decode step's append descriptors must describe the decode descriptor's K and V heads
    d4 = cobra.decode_desc(k_head0=0, v_head0=1, layer_stride=1, n_layers=1, n_kv_heads=1, group=4, n_seqs=1,
                           rows_per_seq=1)
    info = cobra.DecodeInfo(1, 1, 16, 0)
    kd = cobra.compress_desc(head0=0, layer_stride=1, n_layers=1, n_kv_heads=1, side=0, n_seqs=1, rows_per_seq=1)
    vd = cobra.compress_desc(head0=1, layer_stride=1, n_layers=1, n_kv_heads=1, side=1, n_seqs=1, rows_per_seq=1)
    kd_other = cobra.compress_desc(head0=1, layer_stride=1, n_layers=1, n_kv_heads=1, side=0, n_seqs=1,
                                   rows_per_seq=1)
    for k_, v_ in ((vd, vd), (kd, kd), (kd_other, vd)):
        with pytest.raises(cobra.CobraError) as e:
            cobra.cobra_decode_step(256, d4, info, k_, v_, 256, 256, 256, 256, 256, 256, None, 256, 256, 1 << 20)
        assert e.value.status == cobra.COBRA_EINVAL
    with pytest.raises(cobra.CobraError) as e:
        cobra.cobra_decode_qproj_append(256, d4, info, 256, vd, 256, 256, 256, None, 256, 1 << 20)
    assert e.value.status == cobra.COBRA_EINVAL


def test_decode_plan_sizes(L):
    dd = cobra.decode_desc(k_head0=0, v_head0=2, layer_stride=2, n_layers=1, n_kv_heads=2, group=4, n_seqs=3,
                           rows_per_seq=300)
    r = np.array([128, 64, 32, 0], np.int32)
    b = np.array([2, 3, 8, 0], np.int32)
    n = cobra.cobra_decode_workspace_size(dd, r, b, np.array([32768, 1, 0], np.int32))
    assert n > 0 and n % 256 == 0


def test_binding_rejects_non_contiguous_buffers():
    import torch
    x = torch.zeros((4, 6))
    assert cobra._ptr(x) == x.data_ptr()
    with pytest.raises(ValueError):
        cobra._ptr(x.t())
    with pytest.raises(ValueError):
        cobra._ptr(x[:, ::2])


def test_selftest_wait_limits_checked_before_launch():
    # limits outside (0, 100 ms] are refused on the host, before any device work
    for bad in (0, 100_000_001):
        with pytest.raises(Exception):
            cobra.cobra_selftest_wait_timeout(bad)


def test_rope_entry_points_check_arguments_before_the_gpu(L):
    # table: 16 fine rows + one row per 16 positions, 128 floats each
    assert cobra.cobra_rope_table_bytes(1) == 17 * 128 * 4
    assert cobra.cobra_rope_table_bytes(32768) == (16 + 2048) * 128 * 4
    assert cobra.cobra_rope_table_bytes(33) == (16 + 3) * 128 * 4
    for bad in (0, (1 << 22) + 1):
        with pytest.raises(cobra.CobraError) as e:
            cobra.cobra_rope_table_bytes(bad)
        assert e.value.status == cobra.COBRA_EINVAL
    need = cobra.cobra_rope_table_bytes(100)
    for theta, table, nbytes, status in ((0.0, 256, need, cobra.COBRA_EINVAL), (float("nan"), 256, need, cobra.COBRA_EINVAL),
                                         (1e4, None, need, cobra.COBRA_EINVAL), (1e4, 264, need, cobra.COBRA_EALIGN),
                                         (1e4, 256, need - 16, cobra.COBRA_ESPACE)):
        with pytest.raises(cobra.CobraError) as e:
            cobra.cobra_rope_table(theta, 100, table, nbytes)
        assert e.value.status == status
    d4 = cobra.decode_desc(k_head0=0, v_head0=1, layer_stride=1, n_layers=1, n_kv_heads=1, group=4, n_seqs=1,
                           rows_per_seq=1)
    d3 = cobra.decode_desc(k_head0=0, v_head0=1, layer_stride=1, n_layers=1, n_kv_heads=1, group=3, n_seqs=1,
                           rows_per_seq=1)
    info = cobra.DecodeInfo(1, 1, 16, 0)
    cases = [(d4, None, 256, 256, 10, cobra.COBRA_EINVAL),  # no query
             (d4, 256, 256, 264, 10, cobra.COBRA_EALIGN),   # table not 16-byte aligned
             (d4, 256, 258, 256, 10, cobra.COBRA_EALIGN),   # q_pos not 4-byte aligned
             (d4, 256, 256, 256, 0, cobra.COBRA_EINVAL),    # no positions
             (d3, 256, 256, 256, 10, cobra.COBRA_EINVAL)]   # group of 3
    for desc, q, qpos, table, max_pos, status in cases:
        with pytest.raises(cobra.CobraError) as e:
            cobra.cobra_decode_rope_attn(256, desc, info, q, qpos, table, max_pos, 256, 256, None, 256, 256, 1 << 20)
        assert e.value.status == status
