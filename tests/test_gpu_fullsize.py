"""End-to-end parity at the workloads' full sizes (Table alg:kvrobin steps 7-8).

The library compresses every layer of the synthetic cache on the GPU with the oracle's
per-head parameters and appends one new token per (layer, kv head, sequence).  For sampled
(layer, kv head, sequence) triples the oracle compresses the same input tokens itself: the
library's codes must equal the oracle's, or differ by one within 1e-4 of a cell boundary.
Those heads' rows are then overwritten with the oracle's own packed rows (so that both sides
attend over identical codes: a legitimate boundary flip on a heavily weighted token moves
the output by far more than the decode tolerance), and decode runs in the launch
configuration the benchmark times (query projection, scan, combine on one stream) over the
whole cache; sampled outputs must be within max relative error 2e-3 of the oracle's attention.
The single-call entry points (decode attention; the decode step with both appends, on device
buffers and on pinned host buffers) must reproduce the staged calls bit for bit."""
import numpy as np
import pytest
import torch

from oracle import allocator as oal
from oracle import calibrate as ocal
from oracle import compress as ocomp
from oracle import layout as olay
from paper_2609_24298_gb300 import cobra, pipeline, synth

from .gpu_util import (DEV, codes_ok, oracle_allocated_params, oracle_calibrations, oracle_decode, oracle_head_params,
                       read_head_codes, rel_err)

pytestmark = pytest.mark.gpu
TOL = 2e-3
D = 128


@pytest.fixture(scope="module", autouse=True)
def need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    cobra.lib()


def head_region(wl, idx):
    hp = wl.dev.hp
    off, rb = int(wl.dev.offsets[idx]), 16 * int(hp.r[idx]) * int(hp.b[idx])
    return off, rb, wl.dev.cache[off:off + wl.dev.n_slots * rb]


def page_table_host(wl):
    return wl.page_table.cpu().numpy().reshape(wl.seqs, -1) if wl.page_table is not None else None


def head_codes(wl, idx, side, seq, T):
    """Codes [T, r] of one (head, sequence) read back from the device cache."""
    hp = wl.dev.hp
    _, _, region = head_region(wl, idx)
    pt = page_table_host(wl)
    return read_head_codes(region.cpu().numpy(), 0, side, int(hp.r[idx]), int(hp.b[idx]), T, page_table=pt,
                           seq=seq, rows_per_seq=wl.rows_per_seq if pt is None else None)


def put_oracle_rows(wl, idx, side, seq, codes):
    """Overwrite one (head, sequence)'s rows in the device cache with the oracle's packing."""
    hp = wl.dev.hp
    r, b = int(hp.r[idx]), int(hp.b[idx])
    _, rb, region = head_region(wl, idx)
    host = region.cpu().numpy()
    pt = page_table_host(wl)
    rows = olay.pack_tokens(codes, side, b)
    for row in range(rows.shape[0]):
        a = olay.row_address(0, r, b, seq, row, wl.rows_per_seq, pt)
        host[a:a + rb] = rows[row]
    region.copy_(torch.from_numpy(host))


def run_workload(cfg, layers, params, srcs, lens, samples, paged=False, seed=5):
    spec = synth.CONFIGS[cfg]
    H = spec["kv_heads"]
    G = spec["q_heads"] // H
    L, S = layers, len(lens)
    lens = np.asarray(lens, np.int64)
    rows = int(-(-lens.max() // 128))
    hp = oracle_head_params(params)
    wl = pipeline.Workload(cfg=cfg, layers=L, kv=H, group=G, seqs=S, tokens=lens - 1, bpd=0.0, joint=False)
    if paged:
        pps = -(-rows // 2)
        pt = synth.shuffled_pages(cfg, S * pps)
        wl.pages_per_seq, wl.page_table = pps, torch.tensor(pt, dtype=torch.int32, device=DEV)
        n_slots = 2 * S * pps
    else:
        wl.rows_per_seq = rows
        n_slots = S * rows
    wl.dev = pipeline.DeviceParams(hp, n_slots, device=DEV)
    keep = sorted({l for l, _, _ in samples})
    kept = pipeline.fill_cache(wl, srcs, device=DEV, keep_layers=keep)
    wl.tokens = lens
    desc, ws, info = pipeline.decode_setup(wl, device=DEV)
    nws = ws.numel()

    gen = torch.Generator(device=DEV)
    gen.manual_seed(seed)
    xk = torch.randn((L, S, H, D), generator=gen, device=DEV).to(torch.bfloat16)
    xv = torch.randn((L, S, H, D), generator=gen, device=DEV).to(torch.bfloat16)
    qh = np.stack([np.concatenate([synth.decode_queries(cfg, l, h, S, G) for h in range(H)], axis=1)
                   for l in range(L)])  # [L, S, H * G, d]
    q = torch.tensor(qh, dtype=torch.bfloat16, device=DEV)
    pos = torch.tensor(lens - 1, dtype=torch.int32, device=DEV)
    lens_d = torch.tensor(lens, dtype=torch.int32, device=DEV)
    adesc = [cobra.compress_desc(head0=side * L * H, layer_stride=H, n_layers=L, n_kv_heads=H, side=side, n_seqs=S,
                                 rows_per_seq=wl.rows_per_seq, pages_per_seq=wl.pages_per_seq,
                                 x_stride_layer=S * H * D, x_stride_seq=H * D, x_stride_tok=0, x_stride_head=D)
             for side in (0, 1)]
    block, cache, pt = wl.dev.block, wl.dev.cache, wl.page_table
    stream = torch.cuda.current_stream()
    before = cache.clone()
    pre = cache.clone()
    cobra.cobra_append(block, adesc[0], xk, pos, cache, pt, stream)
    cobra.cobra_append(block, adesc[1], xv, pos, cache, pt, stream)
    torch.cuda.synchronize()
    assert cobra.cobra_check(stream) == cobra.COBRA_OK

    # the one-call decode step (query projection fused with the K and V appends, scan, combine)
    # writes the same cache bytes and the same outputs as the separate calls
    step_out = torch.full((L, S, H * G, D), float("nan"), dtype=torch.float32, device=DEV)
    cobra.cobra_decode_step(block, desc, info, adesc[0], adesc[1], xk, xv, pos, q, before, lens_d, pt, step_out, ws,
                            nws, stream)
    staged_out = torch.full_like(step_out, float("nan"))
    cobra.cobra_decode_attn(block, desc, info, q, cache, lens_d, pt, staged_out, ws, nws, stream)
    # and on pinned host buffers: the kernels read the tokens and queries from host memory and
    # write the output there (coherent NVLink-C2C), with the same result
    host_cache = pre.clone()
    host_out = torch.full((L, S, H * G, D), float("nan"), dtype=torch.float32).pin_memory()
    hk_, hv_, hq_ = xk.cpu().pin_memory(), xv.cpu().pin_memory(), q.cpu().pin_memory()
    cobra.cobra_decode_step(block, desc, info, adesc[0], adesc[1], hk_, hv_, pos, hq_, host_cache, lens_d, pt, host_out,
                            ws, nws, stream)
    torch.cuda.synchronize()
    assert cobra.cobra_check(stream) == cobra.COBRA_OK
    assert torch.equal(before, cache)
    assert torch.equal(host_cache, cache)
    assert torch.equal(step_out, staged_out)
    assert torch.equal(host_out, staged_out.cpu())
    # the step can be captured in a CUDA graph (a serving loop's replay): one replay writes the
    # same cache bytes and the same outputs as the eager call
    graph_cache = pre.clone()
    graph_out = torch.full_like(step_out, float("nan"))
    g = torch.cuda.CUDAGraph()
    cap = torch.cuda.Stream()
    cap.wait_stream(stream)
    with torch.cuda.graph(g, stream=cap):
        cobra.cobra_decode_step(block, desc, info, adesc[0], adesc[1], xk, xv, pos, q, graph_cache, lens_d, pt,
                                graph_out, ws, nws, torch.cuda.current_stream())
    g.replay()
    torch.cuda.synchronize()
    assert cobra.cobra_check(stream) == cobra.COBRA_OK
    assert torch.equal(graph_cache, cache)
    assert torch.equal(graph_out, staged_out)
    del before, step_out, staged_out, host_cache, pre, graph_cache, graph_out, g

    # compress + append parity on the sampled heads, then the oracle's rows in their place
    hk, hv = xk.float().cpu().numpy(), xv.float().cpu().numpy()
    oracle_codes = {}
    for l, h, s in samples:
        T = int(lens[s])
        for side, idx, new in ((0, l * H + h, hk), (1, L * H + l * H + h, hv)):
            p = params[idx]
            if p["r"] == 0:
                oracle_codes[(idx, s)] = np.zeros((T, 0), np.int64)
                continue
            x = np.concatenate([kept[(l, side)][s, :T - 1, h].float().cpu().numpy(), new[l, s, h][None]])
            u, want = ocomp.compress(x.astype(np.float64), p["W"], p["mu"], p["delta"], p["b"])
            got = head_codes(wl, idx, side, s, T)
            assert codes_ok(got, u, want), (cfg, l, h, s, side)
            oracle_codes[(idx, s)] = want
            put_oracle_rows(wl, idx, side, s, want)
    torch.cuda.synchronize()

    out = torch.full((L, S, H * G, D), float("nan"), dtype=torch.float32, device=DEV)
    cobra.cobra_decode_qproj(block, desc, info, q, ws, nws, stream)
    cobra.cobra_decode_scan(block, desc, info, cache, lens_d, pt, ws, nws, stream)
    cobra.cobra_decode_combine(block, desc, info, lens_d, out, ws, nws, stream)
    out2 = torch.full_like(out, float("nan"))
    cobra.cobra_decode_attn(block, desc, info, q, cache, lens_d, pt, out2, ws, nws, stream)
    torch.cuda.synchronize()
    assert cobra.cobra_check(stream) == cobra.COBRA_OK
    o = out.cpu().numpy()
    assert np.array_equal(o, out2.cpu().numpy())
    assert np.all(np.isfinite(o))

    worst = 0.0
    for l, h, s in samples:
        ik, iv = l * H + h, L * H + l * H + h
        ref = oracle_decode(qh[l, s, h * G:(h + 1) * G].astype(np.float64), oracle_codes[(ik, s)],
                            oracle_codes[(iv, s)], params[ik], params[iv])
        err = rel_err(o[l, s, h * G:(h + 1) * G], ref)
        worst = max(worst, err)
        assert err <= TOL, (cfg, l, h, s, err)
    return worst


def test_tiny_config_end_to_end():
    """1 layer, 8 kv heads, 32 query heads, 2048 tokens at 2 bpd: every head checked."""
    cals, srcs = oracle_calibrations(1, 1)
    params = oracle_allocated_params(cals, srcs, 2.0)
    run_workload(1, 1, params, srcs, [2048], [(0, h, 0) for h in range(8)])


def test_llama3_8b_full_size_bench_launch():
    """32 layers x 8 kv heads x batch 8 x 32768 tokens, K and V at 1 bpd: the benchmark's
    workload and launch sequence."""
    cals, srcs = oracle_calibrations(2, 32)
    params = oracle_allocated_params(cals, srcs, 1.0)
    samples = [(0, 0, 0), (0, 5, 3), (13, 2, 6), (31, 7, 7), (31, 1, 2)]
    run_workload(2, 32, params, srcs, [32768] * 8, samples)


def test_llama3_70b_joint_half_bpd_full_size():
    """80 layers x 8 kv heads, GQA 8, one 131072-token sequence, joint K+V allocation at
    0.5 bpd, plus the append-compress of the new token."""
    cals, srcs = oracle_calibrations(3, 80, joint=True)
    params = oracle_allocated_params(cals, srcs, 0.5, joint=True)
    samples = [(0, 0, 0), (0, 7, 0), (41, 3, 0), (79, 5, 0)]
    run_workload(3, 80, params, srcs, [131072], samples)


@pytest.mark.parametrize("bpd", [0.5, 1.0, 2.0, 3.0, 4.0])
def test_ragged_paged_rate_sweep(bpd):
    """Batch 32, lengths uniform in [1024, 65536], 256-token pages (shuffled physical pages),
    per-head (r, b) re-allocated at each rate; 4 of the 32 layers (every layer is independent
    and shaped alike)."""
    spec = synth.CONFIGS[5]
    layers = 4
    cals, srcs = _sweep_calibrations(layers)
    params = oracle_allocated_params(cals, srcs, bpd)
    lens = synth.ragged_lengths(5, spec["seqs"], *spec["tokens"])
    order = np.argsort(lens)
    samples = [(0, 0, int(order[0])), (1, 3, int(order[-1])), (3, 6, int(order[len(order) // 2])), (2, 1, 5)]
    run_workload(5, layers, params, srcs, lens, samples, paged=True)


_SWEEP = {}


def _sweep_calibrations(layers):
    if layers not in _SWEEP:
        _SWEEP[layers] = oracle_calibrations(5, layers)
    return _SWEEP[layers]


@pytest.mark.parametrize("k_bpd,v_bpd", [(1.5, 0.5), (0.5, 1.5)])
def test_kv_split_with_uniform_v(k_bpd, v_bpd):
    """The K+V protocol of Sec. 5 ("Joint K+V compression") and App. vside: a total of 2 bpd
    split between the sides, K allocated by the damped allocator on attention-KL weights and V
    by the uniform per-head budget (C1 only); Llama-3-8B shape (batch 8 x 32768 tokens), 4 of
    its 32 layers (the layers are independent and shaped alike)."""
    cals, srcs = oracle_calibrations(2, 4)
    n = len(cals) // 2
    w = np.stack([c["w"] for c in cals])
    k = oal.allocate(w[:n], k_bpd)
    v = oal.allocate(w[n:], v_bpd, oal.Opts(mode=oal.MODE_UNIFORM))
    r, b = np.concatenate([k["r"], v["r"]]), np.concatenate([k["b"], v["b"]])
    params = [ocal.head_params(c, int(rr), int(bb) if rr else 1, synth.hadamard_signs(*s.key))
              for c, s, rr, bb in zip(cals, srcs, r, b)]
    run_workload(2, 4, params, srcs, [32768] * 8, [(0, 0, 0), (1, 5, 3), (3, 7, 7)])


def test_prefill_compress_full_size():
    """The prefill workload compressed in the benchmark's launch geometry: 32 layers x 8 kv heads
    x batch 64 x 4096 tokens of bf16 K and V at 4 bpd (about 34 GB of input), one cobra_compress
    launch per side over all layers (the grid of (layer, head, tile chunk) CTAs the benchmark
    times).  Sampled (layer, kv head, side, sequence, token range) slices: codes equal the
    oracle's, or differ by one within 1e-4 of a cell boundary, and re-packing the kernel's codes
    with the oracle's packer reproduces the rows bit for bit (Table alg:kvrobin step 7)."""
    spec = synth.CONFIGS[4]
    L, H, S, T = spec["layers"], spec["kv_heads"], spec["seqs"], spec["tokens"]
    cals, srcs = oracle_calibrations(4, L)
    params = oracle_allocated_params(cals, srcs, spec["bpd"])
    hp = oracle_head_params(params)
    rows = T // 128
    dp = pipeline.DeviceParams(hp, S * rows, device=DEV)
    # (layer, kv head, side, seq, first token, tokens)
    samples = [(0, 0, 0, 0, 0, 384), (0, 7, 1, 63, 3712, 384), (13, 3, 0, 31, 1000, 700),
               (31, 5, 1, 17, 0, 4096), (31, 0, 0, 40, 2048, 256), (22, 6, 1, 5, 128, 130)]
    xs = {}
    for side in (0, 1):
        x = torch.empty((L, S, T, H, D), dtype=torch.bfloat16, device=DEV)
        for l in range(L):
            x[l] = pipeline.device_tokens([srcs[side * L * H + l * H + h] for h in range(H)], S, T,
                                          seed=4 * 1000003 + 2 * l + side, device=DEV)
        desc = cobra.compress_desc(head0=side * L * H, layer_stride=H, n_layers=L, n_kv_heads=H, side=side, n_seqs=S,
                                   rows_per_seq=rows, x_stride_layer=S * T * H * D, x_stride_seq=T * H * D,
                                   x_stride_tok=H * D, x_stride_head=D)
        cobra.cobra_compress(dp.block, desc, x, 0, T, dp.cache)
        for (l, h, sd, q, t0, n) in samples:
            if sd == side:
                xs[(l, h, q, t0, n)] = x[l, q, t0:t0 + n, h].float().cpu().numpy()
        del x
    torch.cuda.synchronize()
    assert cobra.cobra_check() == cobra.COBRA_OK
    for (l, h, side, q, t0, n) in samples:
        idx = side * L * H + l * H + h
        p = params[idx]
        r, b = p["r"], p["b"]
        if r == 0:
            continue
        rb = olay.row_bytes(r, b)
        base = int(dp.offsets[idx]) + q * rows * rb
        host_rows = dp.cache[base:base + rows * rb].cpu().numpy()
        got_all = read_head_codes(host_rows, 0, side, r, b, T, seq=0, rows_per_seq=rows)
        x = xs[(l, h, q, t0, n)]
        u, want = ocomp.compress(x, p["W"], p["mu"], p["delta"], b)
        got = got_all[t0:t0 + n]
        assert codes_ok(got, u, want), (l, h, side, q, np.argwhere(got != want)[:5])
        # the rows holding the slice, re-packed from the kernel's own codes, are its bytes
        rep = olay.pack_tokens(got_all, side, b)
        for row in range(t0 // 128, -(-(t0 + n) // 128)):
            assert np.array_equal(rep[row], host_rows[row * rb:(row + 1) * rb]), (l, h, side, q, row)
