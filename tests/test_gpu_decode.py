"""GPU parity of cobra_decode_attn (Table alg:kvrobin step 8; App. G) against the oracle's
plain-definition attention over the same packed codes: max over query heads of
||o - o*||_inf / ||o*||_inf <= 2e-3 (bf16 queries, fp32 accumulation)."""
import numpy as np
import pytest
import torch

from oracle import compress as ocomp
from oracle import layout as olay
from oracle import rope as orope
from paper_2609_24298_gb300 import cobra, synth

from .gpu_util import DEV, oracle_decode, oracle_head, oracle_heads_allocated, rel_err, upload

pytestmark = pytest.mark.gpu
TOL = 2e-3


@pytest.fixture(scope="module", autouse=True)
def need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    cobra.lib()


def run_decode(params, srcs, layers, kv, G, lens, q_scale=1.0, paged=False, seed=21, cap=None, rope=None):
    """params/srcs in library order [K(l, h)..., V(l, h)...].  Packs the oracle's codes into the
    cache, runs the library's decode, returns (out, reference).  rope = dict(theta, q_pos
    (per sequence, or None for len - 1), max_pos) runs the RoPE decode against oracle.rope."""
    seqs = len(lens)
    cap = np.asarray(cap if cap is not None else lens, np.int32)
    rows_per_seq = max(1, int(-(-cap.max() // 128)))
    n = layers * kv
    page_table = None
    if paged:
        pps = -(-rows_per_seq // 2)
        page_table = synth.shuffled_pages(seed, seqs * pps).reshape(seqs, pps)
        n_slots = 2 * seqs * pps
    else:
        n_slots = seqs * rows_per_seq
    block, offs, total, r, b = upload(params, n_slots)
    host = np.zeros(total, np.uint8)
    codes = {}
    for idx, (p, s) in enumerate(zip(params, srcs)):
        side = 0 if idx < n else 1
        for q in range(seqs):
            T = int(lens[q])
            x = s.tokens(T, seq=q)
            if p["r"] == 0 or T == 0:
                codes[(idx, q)] = np.zeros((T, p["r"]), np.int64)
                continue
            _, c = ocomp.compress(x, p["W"], p["mu"], p["delta"], p["b"])
            codes[(idx, q)] = c
            rows = olay.pack_tokens(c, side, p["b"])
            for row in range(rows.shape[0]):
                addr = olay.row_address(int(offs[idx]), p["r"], p["b"], q, row, rows_per_seq, page_table)
                host[addr:addr + rows.shape[1]] = rows[row]
    cache = torch.tensor(host, device=DEV)
    qh = np.stack([[np.concatenate([synth.decode_queries(seed, l, h, seqs, G, scale=q_scale)[:, None]
                                    for h in range(kv)], axis=1).reshape(seqs, kv * G, 128)] for l in range(layers)])
    qh = qh.reshape(layers, seqs, kv * G, 128)
    qd = torch.tensor(qh, dtype=torch.bfloat16, device=DEV)
    desc = cobra.decode_desc(k_head0=0, v_head0=n, layer_stride=kv, n_layers=layers, n_kv_heads=kv, group=G,
                             n_seqs=seqs, rows_per_seq=rows_per_seq, pages_per_seq=page_table.shape[1] if paged else 0,
                             q_stride_layer=seqs * kv * G * 128, q_stride_seq=kv * G * 128,
                             o_stride_layer=seqs * kv * G * 128, o_stride_seq=kv * G * 128)
    hb = np.where(r > 0, b, 0)
    wsb = cobra.cobra_decode_workspace_size(desc, r, hb, cap)
    ws = torch.empty(wsb, dtype=torch.uint8, device=DEV)
    info = cobra.cobra_decode_plan(desc, r, hb, cap, ws, wsb)
    out = torch.full((layers, seqs, kv * G, 128), float("nan"), dtype=torch.float32, device=DEV)
    lens_d = torch.tensor(np.asarray(lens, np.int32), device=DEV)
    pt = torch.tensor(page_table.reshape(-1), dtype=torch.int32, device=DEV) if paged else None
    if rope is None:
        cobra.cobra_decode_attn(block, desc, info, qd, cache, lens_d, pt, out, ws, wsb)
    else:
        max_pos = rope.get("max_pos") or max(1, int(cap.max()))
        tb = cobra.cobra_rope_table_bytes(max_pos)
        table = torch.empty(tb // 4, dtype=torch.float32, device=DEV)
        cobra.cobra_rope_table(rope["theta"], max_pos, table, tb)
        qp = rope.get("q_pos")
        qpd = torch.tensor(np.asarray(qp, np.int32), device=DEV) if qp is not None else None
        cobra.cobra_decode_rope_attn(block, desc, info, qd, qpd, table, max_pos, cache, lens_d, pt, out, ws, wsb)
    assert cobra.cobra_check() == cobra.COBRA_OK
    o = out.cpu().numpy()
    ref = np.zeros_like(o, dtype=np.float64)
    for l in range(layers):
        for h in range(kv):
            ik, iv = l * kv + h, n + l * kv + h
            for q in range(seqs):
                qq = qh[l, q, h * G:(h + 1) * G].astype(np.float64)
                if rope is None:
                    ref[l, q, h * G:(h + 1) * G] = oracle_decode(qq, codes[(ik, q)], codes[(iv, q)], params[ik],
                                                                 params[iv])
                elif lens[q] > 0:
                    qp = rope.get("q_pos")
                    pos = int(qp[q]) if qp is not None else int(lens[q]) - 1
                    ref[l, q, h * G:(h + 1) * G] = orope.decode(qq, codes[(ik, q)], codes[(iv, q)], params[ik],
                                                                params[iv], pos, rope["theta"])
    return o, ref, info


def mixed_heads(kv, rbs, cfg=31, layers=1):
    srcs = [synth.HeadSource(cfg, l, h, side, (0.3, 2.5)) for side in (0, 1) for l in range(layers) for h in range(kv)]
    params = [oracle_head(s, r, b) for s, (r, b) in zip(srcs, rbs)]
    return params, srcs


def test_tiny_config_full():
    """The tiny workload: 1 layer, 8 KV heads, 32 query heads, 2048 tokens, oracle allocation at 2 bpd."""
    params, srcs = oracle_heads_allocated(1, 1, 2.0)
    o, ref, _ = run_decode(params, srcs, 1, 8, 4, [2048])
    assert rel_err(o, ref) < TOL


# every width on each side, plus the pairs whose item loops have their own code at G = 4
@pytest.mark.parametrize("bk,bv", [(1, 8), (2, 7), (3, 6), (4, 5), (5, 4), (6, 3), (7, 2), (8, 1),
                                   (3, 4), (4, 3), (4, 4), (5, 5)])
def test_every_bit_width(bk, bv):
    rbs = [(128 if bk <= 2 else 48, bk), (18, bk), (128 if bv <= 2 else 40, bv), (2, bv)]
    params, srcs = mixed_heads(2, rbs, cfg=32 + bk)
    o, ref, _ = run_decode(params, srcs, 1, 2, 4, [700])
    assert rel_err(o, ref) < TOL


def test_zero_rank_sides():
    # head 0: r_K = 0 (uniform attention); head 1: r_V = 0 (output = mu_V)
    rbs = [(0, 1), (32, 3), (64, 2), (0, 1)]
    params, srcs = mixed_heads(2, rbs, cfg=41)
    o, ref, _ = run_decode(params, srcs, 1, 2, 4, [300])
    assert rel_err(o, ref) < TOL


def test_ragged_lengths_and_empty_sequence():
    rbs = [(64, 2), (100, 1), (32, 4), (128, 2)]
    params, srcs = mixed_heads(2, rbs, cfg=42)
    lens = [1, 127, 128, 129, 255, 256, 257, 0, 1000]
    o, ref, _ = run_decode(params, srcs, 1, 2, 4, lens, cap=[1024] * len(lens))
    assert rel_err(np.delete(o, 7, axis=1), np.delete(ref, 7, axis=1)) < TOL
    assert np.all(o[:, 7] == 0)


def test_paged_layout():
    rbs = [(64, 2), (30, 3), (128, 1), (16, 8)]
    params, srcs = mixed_heads(2, rbs, cfg=43)
    o, ref, _ = run_decode(params, srcs, 1, 2, 4, [900, 300, 513], paged=True)
    assert rel_err(o, ref) < TOL


def test_group_of_eight():
    rbs = [(32, 2), (14, 4), (128, 1), (40, 3)]
    params, srcs = mixed_heads(2, rbs, cfg=44)
    o, ref, _ = run_decode(params, srcs, 1, 2, 8, [400, 130])
    assert rel_err(o, ref) < TOL


def test_peaked_queries_and_many_chunks():
    """Scaled queries make attention peaked; 20k tokens split into several chunks per head."""
    rbs = [(128, 2), (64, 3), (128, 2), (96, 2)]
    params, srcs = mixed_heads(2, rbs, cfg=45)
    o, ref, info = run_decode(params, srcs, 1, 2, 4, [20000], q_scale=4.0)
    assert info.n_items > info.n_groups
    assert rel_err(o, ref) < TOL


@pytest.mark.parametrize("G", [4, 8])
def test_many_chunks_partial_channel_quads(G):
    """The combine reads the chunk sums four channels at a time: V ranks that are not a
    multiple of 4 (42, 6) leave a partly used last quad, over groups cut into many chunks."""
    rbs = [(128, 2), (64, 3), (42, 2), (6, 3)]
    params, srcs = mixed_heads(2, rbs, cfg=47)
    o, ref, info = run_decode(params, srcs, 1, 2, G, [24000, 9000])
    assert info.n_items > info.n_groups
    assert rel_err(o, ref) < TOL


def test_multi_layer_strides():
    rbs = [(64, 2), (32, 3), (48, 2), (128, 1)] * 2
    srcs = [synth.HeadSource(46, l, h, side, (0.3, 2.5)) for side in (0, 1) for l in range(2) for h in range(2)]
    params = [oracle_head(s, r, b) for s, (r, b) in zip(srcs, rbs)]
    o, ref, _ = run_decode(params, srcs, 2, 2, 4, [333, 64])
    assert rel_err(o, ref) < TOL
