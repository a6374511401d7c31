"""GPU parity of cobra_compress / cobra_append (Table alg:kvrobin step 7) against the oracle:
codes equal except +-1 where the oracle's pre-rounding value is within 1e-4 of a cell
boundary; packed bytes bit-exact given the codes (re-packing the kernel's codes with the
oracle's packer reproduces every byte, zero tails included)."""
import numpy as np
import pytest
import torch

from oracle import compress as ocomp
from oracle import layout as olay
from paper_2609_24298_gb300 import cobra, synth

from .gpu_util import DEV, codes_ok, oracle_head, read_head_codes, upload

pytestmark = pytest.mark.gpu

RB = [(r, b) for b in range(1, 9) for r in (2, 18, 64, 128)] + [(6, 3), (14, 5), (16, 7), (30, 2), (100, 1), (126, 6)]


@pytest.fixture(scope="module", autouse=True)
def need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    cobra.lib()


def run_compress(params, srcs, T, side, seqs=1, t0=0, page_table=None, rows_per_seq=None, x_override=None):
    H = len(params)
    nrows = -(-(t0 + T) // 128)
    rows_per_seq = rows_per_seq or nrows
    n_slots = seqs * rows_per_seq if page_table is None else 2 * int(page_table.max() + 1)
    block, offs, total, r, b = upload(params, n_slots)
    cache = torch.zeros(total, dtype=torch.uint8, device=DEV)
    xs = x_override if x_override is not None else np.stack(
        [np.stack([s.tokens(T, seq=q) for s in srcs], axis=1) for q in range(seqs)])  # [S, T, H, d]
    x = torch.tensor(xs, dtype=torch.bfloat16, device=DEV)
    pt = None
    pps = 0
    if page_table is not None:
        pps = page_table.shape[1]
        pt = torch.tensor(page_table.reshape(-1), dtype=torch.int32, device=DEV)
    desc = cobra.compress_desc(head0=0, layer_stride=H, n_layers=1, n_kv_heads=H, side=side, n_seqs=seqs,
                               rows_per_seq=rows_per_seq, pages_per_seq=pps, x_stride_layer=0,
                               x_stride_seq=T * H * 128, x_stride_tok=H * 128, x_stride_head=128)
    cobra.cobra_compress(block, desc, x, t0, T, cache, pt)
    assert cobra.cobra_check() == cobra.COBRA_OK
    return cache.cpu().numpy(), offs, r, b, xs


def check_head(host, off, side, p, x, T, t0=0, seq=0, page_table=None, rows_per_seq=None):
    r, b = p["r"], p["b"]
    full = read_head_codes(host, off, side, r, b, t0 + T, page_table=page_table, seq=seq,
                           rows_per_seq=rows_per_seq)
    got = full[t0:t0 + T]
    u, want = ocomp.compress(x, p["W"], p["mu"], p["delta"], b)
    assert codes_ok(got, u, want), (r, b, side, np.argwhere(got != want)[:5])
    # bit-exact packing of the kernel's own codes, zero tail included
    nrows = -(-(t0 + T) // 128)
    rbytes = olay.row_bytes(r, b)
    for row in range(t0 // 128, nrows):
        addr = olay.row_address(int(off), r, b, seq, row, rows_per_seq or nrows, page_table)
        lo, hi = row * 128, min((row + 1) * 128, t0 + T)
        codes = np.zeros((128, r), np.int64)
        codes[: hi - lo] = full[lo:hi]
        assert np.array_equal(olay.pack_row(codes, side, b), host[addr:addr + rbytes]), (r, b, row)
    return int(np.sum(got != want))


@pytest.mark.parametrize("side", [0, 1])
def test_compress_every_bit_width(side):
    srcs = [synth.HeadSource(11, 0, i, side, (0.3, 2.5)) for i in range(len(RB))]
    params = [oracle_head(s, r, b) for s, (r, b) in zip(srcs, RB)]
    T = 300
    host, offs, r, b, xs = run_compress(params, srcs, T, side)
    flips, n = 0, 0
    for h, p in enumerate(params):
        flips += check_head(host, offs[h], side, p, xs[0, :, h], T)
        n += T * p["r"]
    # every flip is already confined to a cell boundary by codes_ok; they must also be rare
    assert flips <= 1e-4 * n


@pytest.mark.parametrize("T", [1, 127, 128, 129, 255, 256, 257])
def test_compress_ragged_lengths(T):
    srcs = [synth.HeadSource(12, 0, i, 0, (0.5, 2.0)) for i in range(3)]
    params = [oracle_head(s, r, b) for s, (r, b) in zip(srcs, [(64, 2), (18, 3), (128, 1)])]
    host, offs, r, b, xs = run_compress(params, srcs, T, 0)
    for h, p in enumerate(params):
        check_head(host, offs[h], 0, p, xs[0, :, h], T)


def test_compress_seqs_offset_and_paged():
    srcs = [synth.HeadSource(13, 0, i, 1, (0.5, 2.0)) for i in range(2)]
    params = [oracle_head(s, r, b) for s, (r, b) in zip(srcs, [(32, 4), (96, 2)])]
    seqs, T, t0 = 3, 200, 256
    # rows 2..3 of each sequence written; 2 pages per sequence needed, shuffled physical ids
    pt = synth.shuffled_pages(13, seqs * 2).reshape(seqs, 2)
    host, offs, r, b, xs = run_compress(params, srcs, T, 1, seqs=seqs, t0=t0, page_table=pt)
    for q in range(seqs):
        for h, p in enumerate(params):
            check_head(host, offs[h], 1, p, xs[q, :, h], T, t0=t0, seq=q, page_table=pt)


def test_compress_clamps_at_both_ends():
    """Tokens scaled by 0, +-40 and +-400 push y / Delta far outside [-2^{b-1}, 2^{b-1}) for
    every bit width: wherever the oracle's pre-rounding value u lies outside [-0.5, 2^b + 0.5]
    the code must be exactly 0 or 2^b - 1, the zero tokens must give the code of the mean's
    projection, and the rest may differ by one near a cell boundary (the scaled inputs scale
    the rounding error of the projection with them).  The packed bytes must re-pack exactly."""
    srcs = [synth.HeadSource(17, 0, i, 0, (0.5, 2.0)) for i in range(8)]
    params = [oracle_head(s, 16 * (1 + i % 3), i + 1) for i, s in enumerate(srcs)]
    T = 260
    scale = np.array([0.0, 1.0, 40.0, -40.0, 400.0, -400.0, 0.5, -1.0])[np.arange(T) % 8]
    xs = np.stack([s.tokens(T) for s in srcs], axis=1)[None] * scale[None, :, None, None]
    xs = torch.tensor(xs).to(torch.bfloat16).double().numpy()  # the values the kernel reads
    host, offs, r, b, xs = run_compress(params, srcs, T, 0, x_override=xs)
    saturated = 0
    for h, p in enumerate(params):
        r_, b_ = p["r"], p["b"]
        got = read_head_codes(host, offs[h], 0, r_, b_, T)
        u, want = ocomp.compress(xs[0, :, h], p["W"], p["mu"], p["delta"], b_)
        outside = (u < -0.5) | (u > (1 << b_) + 0.5)
        assert np.array_equal(got[outside], want[outside]), (r_, b_)
        assert np.all(np.abs(got - want) <= 1), (r_, b_)
        zero = scale == 0.0
        assert codes_ok(got[zero], u[zero], want[zero]), (r_, b_)
        saturated += int(outside.sum())
        for row in range(-(-T // 128)):
            addr = olay.row_address(int(offs[h]), r_, b_, 0, row, -(-T // 128), None)
            codes = np.zeros((128, r_), np.int64)
            lo, hi = row * 128, min((row + 1) * 128, T)
            codes[: hi - lo] = got[lo:hi]
            assert np.array_equal(olay.pack_row(codes, 0, b_), host[addr:addr + olay.row_bytes(r_, b_)]), (r_, b_, row)
    assert saturated > 2000  # both clamps were exercised


def test_compress_zero_rank_head_writes_nothing():
    srcs = [synth.HeadSource(14, 0, i, 0, (0.5, 2.0)) for i in range(2)]
    params = [oracle_head(srcs[0], 0, 1), oracle_head(srcs[1], 16, 4)]
    host, offs, r, b, xs = run_compress(params, srcs, 130, 0)
    assert offs[0] == offs[1]
    check_head(host, offs[1], 0, params[1], xs[0, :, 1], 130)


@pytest.mark.parametrize("side", [0, 1])
def test_append_matches_compress(side):
    srcs = [synth.HeadSource(15, 0, i, side, (0.3, 2.5)) for i in range(4)]
    params = [oracle_head(s, r, b) for s, (r, b) in zip(srcs, [(128, 1), (50, 3), (24, 5), (64, 8)])]
    seqs, T, extra = 2, 260, 6
    nrows = -(-(T + extra) // 128)
    block, offs, total, r, b = upload(params, seqs * nrows)
    cache = torch.zeros(total, dtype=torch.uint8, device=DEV)
    xs = np.stack([np.stack([s.tokens(T + extra, seq=q) for s in srcs], axis=1) for q in range(seqs)])
    x = torch.tensor(xs, dtype=torch.bfloat16, device=DEV)
    H = len(srcs)
    desc = cobra.compress_desc(head0=0, layer_stride=H, n_layers=1, n_kv_heads=H, side=side, n_seqs=seqs,
                               rows_per_seq=nrows, x_stride_layer=0, x_stride_seq=(T + extra) * H * 128,
                               x_stride_tok=H * 128, x_stride_head=128)
    cobra.cobra_compress(block, desc, x, 0, T, cache)
    for k in range(extra):
        xt = x[:, T + k].contiguous()
        pos = torch.full((seqs,), T + k, dtype=torch.int32, device=DEV)
        d2 = cobra.compress_desc(head0=0, layer_stride=H, n_layers=1, n_kv_heads=H, side=side, n_seqs=seqs,
                                 rows_per_seq=nrows, x_stride_layer=0, x_stride_seq=H * 128, x_stride_tok=0,
                                 x_stride_head=128)
        cobra.cobra_append(block, d2, xt, pos, cache)
    assert cobra.cobra_check() == cobra.COBRA_OK
    host = cache.cpu().numpy()
    for q in range(seqs):
        for h, p in enumerate(params):
            check_head(host, offs[h], side, p, xs[q, :, h], T + extra, seq=q, rows_per_seq=nrows)


def test_compress_head_major_layers_padded_tokens():
    """x stored [layer][head][seq][token][136] (head-major, 8 padding elements per token):
    the tensor-map dimensions are ordered by stride, not by the descriptor's field order."""
    L, H, seqs, T, dpad = 2, 3, 2, 300, 136
    srcs = [synth.HeadSource(16, l, h, 0, (0.3, 2.5)) for l in range(L) for h in range(H)]
    rbs = [(128, 2), (40, 4), (22, 7), (64, 1), (90, 3), (128, 5)]
    params = [oracle_head(s, r, b) for s, (r, b) in zip(srcs, rbs)]
    nrows = -(-T // 128)
    block, offs, total, r, b = upload(params, seqs * nrows)
    cache = torch.zeros(total, dtype=torch.uint8, device=DEV)
    xs = np.zeros((L, H, seqs, T, dpad), np.float32)
    for l in range(L):
        for h in range(H):
            for q in range(seqs):
                xs[l, h, q, :, :128] = srcs[l * H + h].tokens(T, seq=q)
    x = torch.tensor(xs, dtype=torch.bfloat16, device=DEV)
    desc = cobra.compress_desc(head0=0, layer_stride=H, n_layers=L, n_kv_heads=H, side=0, n_seqs=seqs,
                               rows_per_seq=nrows, x_stride_layer=H * seqs * T * dpad, x_stride_seq=T * dpad,
                               x_stride_tok=dpad, x_stride_head=seqs * T * dpad)
    cobra.cobra_compress(block, desc, x, 0, T, cache)
    assert cobra.cobra_check() == cobra.COBRA_OK
    host = cache.cpu().numpy()
    for l in range(L):
        for h in range(H):
            for q in range(seqs):
                check_head(host, offs[l * H + h], 0, params[l * H + h], xs[l, h, q, :, :128], T, seq=q,
                           rows_per_seq=nrows)
