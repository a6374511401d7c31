"""Assembling a compressed KV cache through libcobra (product path).

Calibration, allocation and basis fusion run in the library's host code, compression and
decode in its CUDA kernels; this module only generates the synthetic inputs (synth), moves
buffers (torch) and calls the C ABI.  Head numbering inside the parameter block: K heads
first (index layer * H + kv), then V heads (index L * H + layer * H + kv).
"""
from __future__ import annotations

import os
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass, field

import numpy as np
import torch

from . import cobra, synth

D = cobra.D_HEAD


def _threads():
    return max(1, min(32, os.cpu_count() or 1))


def calibrate_heads(xs, qs=None):
    """Product calibration (Table alg:kvrobin steps 1-2) of many heads in parallel threads."""
    qs = qs if qs is not None else [None] * len(xs)
    with ThreadPoolExecutor(_threads()) as ex:
        return list(ex.map(lambda a: cobra.cobra_calibrate_head(a[0], a[1]), zip(xs, qs)))


@dataclass
class HeadParams:
    r: np.ndarray
    b: np.ndarray
    delta: np.ndarray
    W: list
    mu: np.ndarray
    alloc: dict = field(default_factory=dict)


def fuse_heads(cals, r, b, signs) -> HeadParams:
    Ws, deltas = [], []
    for cal, rr, bb, s in zip(cals, r, b, signs):
        W, dl = cobra.cobra_fuse_basis(cal["U"], cal["lam"], int(rr), int(bb) if rr else 1, s)
        Ws.append(W)
        deltas.append(dl)
    mu = np.stack([np.asarray(c["mu"], np.float32) for c in cals])
    return HeadParams(np.asarray(r, np.int32), np.asarray(b, np.int32), np.asarray(deltas, np.float32), Ws, mu)


class DeviceParams:
    """Parameter block + cache regions on the device."""

    def __init__(self, hp: HeadParams, n_slots: int, device="cuda"):
        self.hp = hp
        self.n_slots = int(n_slots)
        self.offsets, self.cache_bytes = cobra.cobra_plan_layout(hp.r, hp.b, self.n_slots)
        nbytes = cobra.cobra_params_bytes(hp.r)
        self.block = torch.empty(nbytes, dtype=torch.uint8, device=device)
        cobra.cobra_params_build(self.block, nbytes, hp.r, hp.b, hp.delta, self.offsets, hp.W, hp.mu.reshape(-1))
        self.cache = torch.zeros(max(self.cache_bytes, 256), dtype=torch.uint8, device=device)

    def head_rb(self):
        return self.hp.r, np.where(self.hp.r > 0, self.hp.b, 0)


@dataclass
class Workload:
    cfg: int
    layers: int
    kv: int
    group: int
    seqs: int
    tokens: np.ndarray  # per-sequence lengths
    bpd: float
    joint: bool
    dev: DeviceParams = None
    rows_per_seq: int = 0
    pages_per_seq: int = 0
    page_table: torch.Tensor = None

    @property
    def n_heads_side(self):
        return self.layers * self.kv


def build_params(cfg: int, layers: int, bpd: float, joint: bool, kl_queries: bool = True, alloc_opts=None,
                 v_bpd: float | None = None, v_opts=None):
    """Calibrate every (layer, kv head, side) of a config on 512 calibration tokens, allocate
    (K and V separately, or jointly over both sides with MSE weights), fuse the bases.  With
    v_bpd the V side gets its own rate (the K+V split of Sec. 5, "Joint K+V compression") and
    v_opts its own allocator options (e.g. the uniform per-head budget of App. vside)."""
    spec = synth.CONFIGS[cfg]
    H = spec["kv_heads"]
    G = spec["q_heads"] // H
    srcs = [synth.HeadSource(cfg, l, h, side, spec["alpha"]) for side in (0, 1) for l in range(layers) for h in range(H)]
    xs = [s.calibration(512) for s in srcs]
    qs = []
    for side in (0, 1):
        for l in range(layers):
            for h in range(H):
                use_q = side == 0 and kl_queries and not joint
                qs.append(synth.calibration_queries(cfg, l, h, G, 512, spec["alpha"]) if use_q else None)
    cals = calibrate_heads(xs, qs)
    n = layers * H
    w = np.stack([c["w"] for c in cals])
    if joint:
        res = cobra.cobra_allocate(w, bpd, alloc_opts)
        r, b = res["r"], res["b"]
        allocs = [res]
    else:
        rk = cobra.cobra_allocate(w[:n], bpd, alloc_opts)
        rv = cobra.cobra_allocate(w[n:], bpd if v_bpd is None else v_bpd, alloc_opts if v_opts is None else v_opts)
        r, b = np.concatenate([rk["r"], rv["r"]]), np.concatenate([rk["b"], rv["b"]])
        allocs = [rk, rv]
    signs = [synth.hadamard_signs(*s.key) for s in srcs]
    hp = fuse_heads(cals, r, b, signs)
    hp.alloc = dict(parts=allocs, w=w)
    hp.cals = cals
    return hp, srcs


def calibrate_heads_device(xs, qs=None, device="cuda"):
    """Steps 1-2 for many heads on the device (cobra_calibrate_heads): the heads with
    calibration queries (attention-KL weights) in one launch, the others (MSE) in another.
    Returns the same dicts as calibrate_heads (U[:, j] = direction j)."""
    qs = qs if qs is not None else [None] * len(xs)
    out = [None] * len(xs)
    for kl in (True, False):
        idx = [i for i, q in enumerate(qs) if (q is not None) == kl]
        if not idx:
            continue
        x = torch.tensor(np.stack([np.asarray(xs[i], np.float32) for i in idx]), device=device).contiguous()
        q = None
        if kl:
            q = torch.tensor(np.stack([np.asarray(qs[i], np.float32).reshape(-1, D) for i in idx]),
                             device=device).contiguous()
        n = len(idx)
        f64 = lambda *shape: torch.empty(shape, dtype=torch.float64, device=device)
        mu, lam, U, w = f64(n, D), f64(n, D), f64(n, D * D), f64(n, D)
        cobra.cobra_calibrate_heads(x, q, mu, lam, U, w)
        torch.cuda.synchronize()
        mu, lam, U, w = mu.cpu().numpy(), lam.cpu().numpy(), U.cpu().numpy(), w.cpu().numpy()
        for k, i in enumerate(idx):
            out[i] = dict(mu=mu[k], lam=lam[k], U=U[k].reshape(D, D).T.copy(), w=w[k])
    return out


def measured_tables(cals, srcs, r_list, b_list, device="cuda", n_tok: int = 512, stream=None) -> np.ndarray:
    """App. E: every head's calibration tokens through the deployed quantizer at every
    candidate (r, b), on the device (cobra_measure_distortion).  Returns D [n][len(r)][len(b)]."""
    f32 = lambda a: torch.tensor(np.asarray(a, np.float32), device=device).contiguous()
    x = f32(np.stack([s.calibration(n_tok) for s in srcs]))
    U = f32(np.stack([c["U"].T.reshape(-1) for c in cals]))  # column k of U = row k of U^T
    f64 = lambda a: torch.tensor(np.asarray(a, np.float64), device=device).contiguous()
    lam = f64(np.stack([c["lam"] for c in cals]))
    w = f64(np.stack([c["w"] for c in cals]))
    mu = f32(np.stack([c["mu"] for c in cals]))
    signs = torch.tensor(np.stack([synth.hadamard_signs(*s.key) for s in srcs]), dtype=torch.int8,
                         device=device).contiguous()
    coords = torch.empty((len(cals), n_tok, D), dtype=torch.float32, device=device)
    out = torch.empty((len(cals), len(r_list), len(b_list)), dtype=torch.float64, device=device)
    cobra.cobra_measure_distortion(x, U, lam, w, mu, signs, r_list, b_list, coords, out, stream)
    torch.cuda.synchronize()
    return out.cpu().numpy()


def measured_allocation(cals, srcs, bpd: float, joint: bool = False, device="cuda"):
    """App. E's allocator: the exact DP on measured tables over the allocator's grid
    (r in {0, 2, ..., 128}, b in 1..8), K and V separately (or jointly).  Returns (r, b)."""
    r_list, b_list = list(range(0, D + 1, 2)), list(range(1, 9))
    T = measured_tables(cals, srcs, r_list, b_list, device)
    n = len(cals) // 2
    parts = [T] if joint else [T[:n], T[n:]]
    res = [cobra.cobra_allocate_tables(t, r_list, b_list, bpd, D) for t in parts]
    return np.concatenate([x["r"] for x in res]), np.concatenate([x["b"] for x in res])


def device_tokens(src_list, n_seqs: int, n_tok: int, seed: int, device="cuda", t_offset: int = 0):
    """Synthetic bf16 K or V for one layer and side, generated on the device:
    [n_seqs, n_tok, H, 128] with x = A g per head (A from the head's HeadSource)."""
    A = torch.tensor(np.stack([s.A for s in src_list]), dtype=torch.float32, device=device)  # [H, d, d]
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    g = torch.randn((n_seqs, n_tok, len(src_list), D), generator=gen, device=device, dtype=torch.float32)
    x = torch.einsum("sthd,hed->sthe", g, A)  # einsum may return a permuted layout
    return x.to(torch.bfloat16).contiguous()


def fill_cache(wl: Workload, srcs, device="cuda", stream=None, keep_layers=()):
    """Compress every layer's synthetic K and V (all tokens of all sequences) into the cache
    with cobra_compress.  Returns the device tensors of the layers listed in keep_layers."""
    H, L = wl.kv, wl.layers
    n_tok = int(wl.tokens.max())
    kept = {}
    for l in range(L):
        for side in (0, 1):
            src_list = [srcs[side * L * H + l * H + h] for h in range(H)]
            x = device_tokens(src_list, wl.seqs, n_tok, seed=(wl.cfg * 1000003 + l * 2 + side), device=device)
            desc = cobra.compress_desc(head0=side * L * H + l * H, layer_stride=H, n_layers=1, n_kv_heads=H, side=side,
                                       n_seqs=wl.seqs, rows_per_seq=wl.rows_per_seq, pages_per_seq=wl.pages_per_seq,
                                       x_stride_layer=0, x_stride_seq=n_tok * H * D, x_stride_tok=H * D,
                                       x_stride_head=D)
            cobra.cobra_compress(wl.dev.block, desc, x, 0, n_tok, wl.dev.cache, wl.page_table, stream)
            if l in keep_layers:
                kept[(l, side)] = x
            else:
                del x
    return kept


def decode_setup(wl: Workload, seq_cap=None, device="cuda"):
    """Decode descriptor, planned workspace and plan info for all layers of the workload."""
    H, L = wl.kv, wl.layers
    desc = cobra.decode_desc(k_head0=0, v_head0=L * H, layer_stride=H, n_layers=L, n_kv_heads=H, group=wl.group,
                             n_seqs=wl.seqs, rows_per_seq=wl.rows_per_seq, pages_per_seq=wl.pages_per_seq,
                             q_stride_layer=wl.seqs * H * wl.group * D, q_stride_seq=H * wl.group * D,
                             o_stride_layer=wl.seqs * H * wl.group * D, o_stride_seq=H * wl.group * D)
    hr, hb = wl.dev.head_rb()
    cap = np.asarray(seq_cap if seq_cap is not None else wl.tokens, np.int32)
    nbytes = cobra.cobra_decode_workspace_size(desc, hr, hb, cap)
    ws = torch.empty(nbytes, dtype=torch.uint8, device=device)
    info = cobra.cobra_decode_plan(desc, hr, hb, cap, ws, nbytes)
    return desc, ws, info


def packed_bytes_read(wl: Workload, lens=None) -> int:
    """Bytes of packed codes a decode over `lens` tokens per sequence reads: for every head of
    every sequence, ceil(T * r * b / 8 / 16) * 16."""
    lens = wl.tokens if lens is None else lens
    hr, hb = wl.dev.head_rb()
    tot = 0
    for T in np.asarray(lens, np.int64):
        bits = T * (hr.astype(np.int64) * hb.astype(np.int64))
        tot += int((((bits + 7) // 8 + 15) // 16 * 16).sum())
    return tot
