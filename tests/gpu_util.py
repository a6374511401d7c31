"""Helpers for the GPU parity tests: per-head parameters computed by the oracle (calibration,
allocation, fusion), uploaded through the C ABI, and comparisons against the oracle."""
from __future__ import annotations

import numpy as np
import torch

from oracle import allocator as oal
from oracle import attention as oatt
from oracle import calibrate as ocal
from oracle import compress as ocomp
from oracle import layout as olay
from paper_2609_24298_gb300 import cobra, synth

DEV = "cuda:0"


def oracle_head(src, r, b, q_cal=None):
    cal = ocal.calibrate_head(src.calibration(512), q_cal)
    return ocal.head_params(cal, r, b, synth.hadamard_signs(*src.key)) | {"w": cal["w"]}


def oracle_calibrations(cfg, layers, joint=False):
    """Oracle calibration of every (side, layer, kv head) of a config, in library head order
    [K heads..., V heads...]; KL weights with the config's calibration queries for separate
    K allocation, MSE weights otherwise.  Returns (calibrations, sources)."""
    spec = synth.CONFIGS[cfg]
    H = spec["kv_heads"]
    G = spec["q_heads"] // H
    srcs = [synth.HeadSource(cfg, l, h, side, spec["alpha"]) for side in (0, 1) for l in range(layers) for h in range(H)]
    cals = []
    for i, s in enumerate(srcs):
        side, rem = divmod(i, layers * H)
        l, h = divmod(rem, H)
        q = synth.calibration_queries(cfg, l, h, G, 512, spec["alpha"]) if (side == 0 and not joint) else None
        cals.append(ocal.calibrate_head(s.calibration(512), q))
    return cals, srcs


def oracle_allocated_params(cals, srcs, bpd, joint=False):
    """Oracle allocation at `bpd` (K and V separately, or jointly) and basis fusion."""
    w = np.stack([c["w"] for c in cals])
    n = len(cals) // 2
    if joint:
        res = oal.allocate(w, bpd)
        r, b = res["r"], res["b"]
    else:
        a, c = oal.allocate(w[:n], bpd), oal.allocate(w[n:], bpd)
        r, b = np.concatenate([a["r"], c["r"]]), np.concatenate([a["b"], c["b"]])
    return [ocal.head_params(c, int(rr), int(bb) if rr else 1, synth.hadamard_signs(*s.key))
            for c, s, rr, bb in zip(cals, srcs, r, b)]


def oracle_heads_allocated(cfg, layers, bpd, joint=False):
    """Oracle calibration + allocation + fusion for every (side, layer, kv head) of a config.
    Returns (params list in library head order [K heads..., V heads...], sources)."""
    cals, srcs = oracle_calibrations(cfg, layers, joint)
    return oracle_allocated_params(cals, srcs, bpd, joint), srcs


def upload(params, n_slots):
    r = np.array([p["r"] for p in params], np.int32)
    b = np.array([p["b"] if p["r"] else 1 for p in params], np.int32)
    delta = np.array([p["delta"] if p["r"] else 0.0 for p in params], np.float32)
    offs, total = cobra.cobra_plan_layout(r, b, n_slots)
    nbytes = cobra.cobra_params_bytes(r)
    block = torch.empty(nbytes, dtype=torch.uint8, device=DEV)
    mu = np.stack([p["mu"] for p in params]).astype(np.float32)
    cobra.cobra_params_build(block, nbytes, r, b, delta, offs, [p["W"] for p in params], mu.reshape(-1))
    return block, offs, total, r, b


def codes_ok(got, u, want):
    """Codes equal, or differ by one where the oracle's pre-rounding value is within 1e-4 of
    an integer (a cell boundary)."""
    near = np.abs(u - np.round(u)) < 1e-4
    return np.all((got == want) | ((np.abs(got - want) == 1) & near))


def read_head_codes(host_cache, off, side, r, b, T, rows_slot0=0, page_table=None, seq=0, rows_per_seq=None):
    """Codes [T, r] of one (head, seq) from a host copy of the cache."""
    rbytes = olay.row_bytes(r, b)
    nrows = -(-T // 128)
    rows = []
    for row in range(nrows):
        addr = olay.row_address(int(off), r, b, seq, row, rows_per_seq or nrows, page_table)
        rows.append(host_cache[addr:addr + rbytes])
    return olay.unpack_tokens(np.stack(rows), side, r, b, T) if nrows else np.zeros((0, r), np.int64)


def oracle_decode(q, kc, vc, pk, pv):
    if kc.shape[0] == 0:
        return np.zeros((q.shape[0], q.shape[1]))
    return oatt.decode(q, kc, vc, pk, pv)


def rel_err(o, ref):
    """max over query heads of ||o - ref||_inf / ||ref||_inf."""
    den = np.maximum(np.abs(ref).max(axis=-1), 1e-30)
    return float((np.abs(o - ref).max(axis=-1) / den).max())


def oracle_head_params(params):
    """The oracle's per-head parameters in the product's HeadParams form (for DeviceParams)."""
    from paper_2609_24298_gb300 import pipeline
    r = np.array([p["r"] for p in params], np.int32)
    b = np.array([p["b"] if p["r"] else 1 for p in params], np.int32)
    delta = np.array([p["delta"] if p["r"] else 0.0 for p in params], np.float32)
    mu = np.stack([p["mu"] for p in params]).astype(np.float32)
    return pipeline.HeadParams(r, b, delta, [p["W"] for p in params], mu)

