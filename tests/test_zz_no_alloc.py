"""cobra_decode_attn_static: decode attention for callers that cannot allocate device memory
(its workspace is a fixed array inside the library).  Two calls in a row, with different
queries, must match the workspace-based cobra_decode_attn within the decode tolerance.
Collected last on purpose (file name) so that a failure here does not hide other tests."""
import numpy as np
import pytest
import torch

from paper_2609_24298_gb300 import cobra, synth

from .gpu_util import DEV, oracle_head, rel_err, upload

pytestmark = pytest.mark.gpu
TOL = 2e-3


@pytest.fixture(scope="module", autouse=True)
def need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    cobra.lib()


@pytest.mark.parametrize("G", [4, 8])
def test_static_scratch_matches_workspace_path(G):
    L, H, S = 2, 2, 3
    lens = np.array([700, 129, 300], np.int32)
    cap_rows = int(-(-lens.max() // 128))
    rbs = [(64, 2), (128, 1), (30, 3), (16, 8)] * 2  # K heads (l, h) then V heads
    srcs = [synth.HeadSource(61, l, h, side, (0.3, 2.5)) for side in (0, 1) for l in range(L) for h in range(H)]
    params = [oracle_head(s, r, b) for s, (r, b) in zip(srcs, rbs)]
    block, offs, total, r, b = upload(params, S * cap_rows)
    cache = torch.zeros(total, dtype=torch.uint8, device=DEV)
    T = int(lens.max())
    for side in (0, 1):
        for l in range(L):
            x = np.stack([np.stack([srcs[side * L * H + l * H + h].tokens(T, seq=q) for h in range(H)], axis=1)
                          for q in range(S)])
            xd = torch.tensor(x, dtype=torch.bfloat16, device=DEV)
            desc = cobra.compress_desc(head0=side * L * H + l * H, layer_stride=H, n_layers=1, n_kv_heads=H, side=side,
                                       n_seqs=S, rows_per_seq=cap_rows, x_stride_layer=0, x_stride_seq=T * H * 128,
                                       x_stride_tok=H * 128, x_stride_head=128)
            cobra.cobra_compress(block, desc, xd, 0, T, cache)
    desc = cobra.decode_desc(k_head0=0, v_head0=L * H, layer_stride=H, n_layers=L, n_kv_heads=H, group=G, n_seqs=S,
                             rows_per_seq=cap_rows, q_stride_layer=S * H * G * 128, q_stride_seq=H * G * 128,
                             o_stride_layer=S * H * G * 128, o_stride_seq=H * G * 128)
    hb = np.where(r > 0, b, 0)
    wsb = cobra.cobra_decode_workspace_size(desc, r, hb, lens)
    ws = torch.empty(wsb, dtype=torch.uint8, device=DEV)
    info = cobra.cobra_decode_plan(desc, r, hb, lens, ws, wsb)
    lens_d = torch.tensor(lens, device=DEV)
    for call in range(2):
        q = torch.tensor(synth.to_bf16(np.random.default_rng(100 + call).standard_normal((L, S, H * G, 128)) * 2),
                         dtype=torch.bfloat16, device=DEV)
        ref = torch.full((L, S, H * G, 128), float("nan"), dtype=torch.float32, device=DEV)
        out = torch.full_like(ref, float("nan"))
        cobra.cobra_decode_attn(block, desc, info, q, cache, lens_d, None, ref, ws, wsb)
        cobra.cobra_decode_attn_static(block, desc, q, cache, lens_d, None, out)
        assert cobra.cobra_check() == cobra.COBRA_OK
        o, rr = out.cpu().numpy(), ref.cpu().numpy()
        assert np.all(np.isfinite(o))
        assert rel_err(o, rr) < TOL, (call, rel_err(o, rr))


def test_static_scratch_rejects_too_many_chunks():
    # 8 seqs x 32 layers x 8 kv heads = 2048 chunks need about 13 MB, more than the array holds
    desc = cobra.decode_desc(k_head0=0, v_head0=256, layer_stride=8, n_layers=32, n_kv_heads=8, group=4, n_seqs=8,
                             rows_per_seq=256)
    with pytest.raises(cobra.CobraError) as e:
        cobra.cobra_decode_attn_static(256, desc, 256, 256, 256, None, 256)
    assert e.value.status == cobra.COBRA_ESPACE


@pytest.mark.parametrize("G", [4, 8])
def test_static_scratch_paged_cache(G):
    """A paged cache (256-token pages of a shuffled pool): the fixed-scratch plan covers
    2 x pages_per_seq rows per sequence and looks rows up through the page table."""
    from oracle import compress as ocomp
    from oracle import layout as olay

    L, H = 1, 2
    lens = np.array([900, 300, 513, 1], np.int32)
    S = len(lens)
    pps = int(-(-lens.max() // 256))
    page_table = synth.shuffled_pages(31, S * pps).reshape(S, pps)
    rbs = [(64, 2), (42, 3), (128, 1), (16, 8)]
    srcs = [synth.HeadSource(62, 0, h, side, (0.3, 2.5)) for side in (0, 1) for h in range(H)]
    params = [oracle_head(s, r, b) for s, (r, b) in zip(srcs, rbs)]
    block, offs, total, r, b = upload(params, 2 * S * pps)
    host = np.zeros(total, np.uint8)
    for idx, (p, s) in enumerate(zip(params, srcs)):
        side = 0 if idx < H else 1
        for q in range(S):
            _, c = ocomp.compress(s.tokens(int(lens[q]), seq=q), p["W"], p["mu"], p["delta"], p["b"])
            rows = olay.pack_tokens(c, side, p["b"])
            for row in range(rows.shape[0]):
                addr = olay.row_address(int(offs[idx]), p["r"], p["b"], q, row, 2 * pps, page_table)
                host[addr:addr + rows.shape[1]] = rows[row]
    cache = torch.tensor(host, device=DEV)
    pt = torch.tensor(page_table.reshape(-1), dtype=torch.int32, device=DEV)
    desc = cobra.decode_desc(k_head0=0, v_head0=H, layer_stride=H, n_layers=L, n_kv_heads=H, group=G, n_seqs=S,
                             rows_per_seq=2 * pps, pages_per_seq=pps, q_stride_layer=S * H * G * 128,
                             q_stride_seq=H * G * 128, o_stride_layer=S * H * G * 128, o_stride_seq=H * G * 128)
    hb = np.where(r > 0, b, 0)
    wsb = cobra.cobra_decode_workspace_size(desc, r, hb, lens)
    ws = torch.empty(wsb, dtype=torch.uint8, device=DEV)
    info = cobra.cobra_decode_plan(desc, r, hb, lens, ws, wsb)
    lens_d = torch.tensor(lens, device=DEV)
    for call in range(2):
        q = torch.tensor(synth.to_bf16(np.random.default_rng(200 + call).standard_normal((L, S, H * G, 128)) * 2),
                         dtype=torch.bfloat16, device=DEV)
        ref = torch.full((L, S, H * G, 128), float("nan"), dtype=torch.float32, device=DEV)
        out = torch.full_like(ref, float("nan"))
        cobra.cobra_decode_attn(block, desc, info, q, cache, lens_d, pt, ref, ws, wsb)
        cobra.cobra_decode_attn_static(block, desc, q, cache, lens_d, pt, out)
        assert cobra.cobra_check() == cobra.COBRA_OK
        o, rr = out.cpu().numpy(), ref.cpu().numpy()
        assert np.all(np.isfinite(o))
        assert rel_err(o, rr) < TOL, (call, rel_err(o, rr))


def test_static_scratch_reports_heads_outside_the_block():
    """A descriptor whose V heads lie past the parameter block's head table is reported through
    cobra_check (nothing is read past the table); the context keeps working."""
    H, G, S, T = 2, 4, 1, 200
    srcs = [synth.HeadSource(63, 0, h, side, (0.3, 2.5)) for side in (0, 1) for h in range(H)]
    params = [oracle_head(s, 32, 2) for s in srcs]
    block, offs, total, r, b = upload(params, 2)
    cache = torch.zeros(total, dtype=torch.uint8, device=DEV)
    desc = cobra.decode_desc(k_head0=0, v_head0=H + 5, layer_stride=H, n_layers=1, n_kv_heads=H, group=G, n_seqs=S,
                             rows_per_seq=2, q_stride_layer=H * G * 128, q_stride_seq=H * G * 128,
                             o_stride_layer=H * G * 128, o_stride_seq=H * G * 128)
    q = torch.zeros((1, S, H * G, 128), dtype=torch.bfloat16, device=DEV)
    out = torch.full((1, S, H * G, 128), float("nan"), dtype=torch.float32, device=DEV)
    lens_d = torch.tensor([T], dtype=torch.int32, device=DEV)
    cobra.cobra_decode_attn_static(block, desc, q, cache, lens_d, None, out)
    torch.cuda.synchronize()
    assert cobra.cobra_check() == cobra.COBRA_EINVAL
    assert cobra.cobra_check() == cobra.COBRA_OK  # reported once, then cleared
    x = torch.ones(4, device=DEV) * 2
    assert float(x.sum()) == 8.0
