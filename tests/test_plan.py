"""CPU tests of the decode work plan (host logic, no device): the chunks of every
(seq, layer, kv-head) group tile its code rows exactly once, their partial slots are the
group's consecutive range, the head-group table points back at the right groups, chunks of
one code variant are taken together in the variants' (b_K, b_V) order, and the chunk sizes
shrink towards the end of the order without cutting a group into more than 32 chunks."""
import os

import numpy as np
import pytest

from paper_2609_24298_gb300 import cobra

ITEM_MIN, ITEM_MAX = 16 * 1024, 128 * 1024


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not os.path.exists(cobra.LIB_PATH):
        from paper_2609_24298_gb300 import build

        build.build()
    cobra.lib()


def parse(img):
    u32 = img[:128].view(np.uint32)
    i32 = img[:128].view(np.int32)
    u64 = img[:128].view(np.uint64)
    h = dict(magic=int(u32[0]), n_groups=int(i32[2]), n_items=int(i32[3]), group=int(i32[4]), n_layers=int(i32[5]),
             n_kv=int(i32[6]), n_seqs=int(i32[7]), groups_off=int(u64[4]), items_off=int(u64[5]), qt_off=int(u64[6]),
             part_off=int(u64[7]), part_stride=int(i32[16]), hg_off=int(u64[11]), done=int(u32[30]),
             next_item=int(u32[31]))
    g = img[h["groups_off"]:h["groups_off"] + 32 * h["n_groups"]].view(np.int32).reshape(-1, 8)
    it = img[h["items_off"]:h["items_off"] + 16 * h["n_items"]].view(np.int32).reshape(-1, 4)
    hg = img[h["hg_off"]:h["hg_off"] + 4 * h["n_groups"]].view(np.int32)
    return h, g, it, hg


def row_bytes(r, b):
    return 16 * r * b if r > 0 else 0


def make(L, H, S, caps, r, b, G=4):
    d = cobra.decode_desc(k_head0=0, v_head0=L * H, layer_stride=H, n_layers=L, n_kv_heads=H, group=G, n_seqs=S,
                          rows_per_seq=max(1, (max(caps) + 127) // 128), pages_per_seq=0)
    img, info = cobra.cobra_decode_plan_host(d, r, b, caps)
    return d, img, info


def check_plan(L, H, S, caps, r, b):
    d, img, info = make(L, H, S, caps, r, b)
    h, g, it, hg = parse(img)
    assert h["n_groups"] == L * H * S == info.n_groups and h["n_items"] == info.n_items == len(it)
    assert h["done"] == 0 and h["next_item"] == 0
    ws = cobra.cobra_decode_workspace_size(d, r, b, caps)
    assert h["part_off"] + 4 * h["part_stride"] * h["n_items"] <= ws
    # groups: one per (seq, layer, kv), heads as the descriptor places them, hg points back
    seen = set()
    for gi, (s, l, kv, first, n, hk, hv, _) in enumerate(g):
        assert (s, l, kv) not in seen
        seen.add((s, l, kv))
        assert hk == l * H + kv and hv == L * H + l * H + kv
        assert hg[(l * H + kv) * S + s] == gi
    # chunks tile each group's rows once; slots are the group's consecutive range
    slots = np.sort(it[:, 3])
    assert np.array_equal(slots, np.arange(len(it)))
    for gi, (s, l, kv, first, n, hk, hv, _) in enumerate(g):
        mine = it[it[:, 0] == gi]
        assert len(mine) == n >= 1
        assert np.array_equal(np.sort(mine[:, 3]), np.arange(first, first + n))
        rows = (caps[s] + 127) // 128
        rb = row_bytes(r[hk], b[hk]) + row_bytes(r[hv], b[hv])
        spans = mine[np.argsort(mine[:, 1]), 1:3]
        if rows == 0 or rb == 0:
            assert n == 1 and spans[0].tolist() == [0, rows]
            continue
        assert spans[0, 0] == 0 and spans[-1, 1] == rows
        assert np.all(spans[1:, 0] == spans[:-1, 1]) and np.all(spans[:, 1] > spans[:, 0])
        assert np.all((spans[:, 1] - spans[:, 0]) * rb <= 1.5 * ITEM_MAX + 2 * rb)
    # variants: each (b_K, b_V) is one run of the order, runs in ascending (b_K, b_V)
    def variant(gi):
        hk, hv = g[gi, 5], g[gi, 6]
        return (b[hk] if r[hk] else 0, b[hv] if r[hv] else 0)

    order = [variant(x) for x in it[:, 0]]
    runs = [order[0]] + [v for p, v in zip(order, order[1:]) if v != p]
    assert runs == sorted(set(runs))
    assert g[:, 4].max() <= 33
    # the RoPE decode's staging bound: K row in whole 16-channel tiles + V row (128-aligned)
    tiles = [256 * (b[hk] if r[hk] else 0) * ((r[hk] + 15) // 16) + (row_bytes(r[hv], b[hv]) + 127) // 128 * 128
             for (_, _, _, _, _, hk, hv, _) in g]
    assert info.max_stage_bytes == max(tiles)
    assert info.max_row_bytes == max(max(row_bytes(r[hk], b[hk]), row_bytes(r[hv], b[hv])) for (*_, hk, hv, _) in g)
    return h, g, it


def test_plan_tiles_rows_and_slots_uniform_lengths():
    rng = np.random.default_rng(7)
    L, H, S = 4, 8, 8
    r = 2 * rng.integers(0, 65, 2 * L * H)
    b = rng.integers(1, 9, 2 * L * H)
    r[:3] = 0  # heads without codes
    check_plan(L, H, S, [32768] * S, r.astype(np.int32), b.astype(np.int32))


def test_plan_ragged_and_empty_sequences():
    rng = np.random.default_rng(11)
    L, H = 2, 8
    caps = [0, 1, 127, 128, 129, 5000, 65536, 300]
    r = 2 * rng.integers(1, 65, 2 * L * H)
    b = rng.integers(1, 4, 2 * L * H)
    check_plan(L, H, len(caps), caps, r.astype(np.int32), b.astype(np.int32))


def test_plan_chunks_shrink_towards_the_end():
    # the Llama-3-8B decode shape at 1 bit per dimension: every head r * b = 128
    L, H, S = 32, 8, 8
    r = np.full(2 * L * H, 64, np.int32)
    b = np.full(2 * L * H, 2, np.int32)
    r[::3], b[::3] = 128, 1
    h, g, it = check_plan(L, H, S, [32768] * S, r, b)
    rb = np.array([row_bytes(r[g[x, 5]], b[g[x, 5]]) + row_bytes(r[g[x, 6]], b[g[x, 6]]) for x in it[:, 0]])
    nbytes = (it[:, 2] - it[:, 1]) * rb
    assert nbytes.sum() == S * 256 * 4096 * L * H
    # large chunks first, short ones last: the final round of one chunk per resident warp is
    # made of short chunks (a group's 1 MB in at most 32 chunks: 32 KB)
    assert nbytes[:2432].min() >= ITEM_MAX - 4096
    assert nbytes[-2432:].max() <= 2 * 32 * 1024
    assert np.median(nbytes[-2432:]) <= 32 * 1024
    # fewer partials than fixed 64 KB chunks
    assert len(it) < nbytes.sum() // (64 * 1024)


def test_plan_host_reports_size_without_buffer():
    L, H, S = 1, 8, 1
    r = np.full(2 * L * H, 16, np.int32)
    b = np.full(2 * L * H, 2, np.int32)
    d = cobra.decode_desc(k_head0=0, v_head0=L * H, layer_stride=H, n_layers=L, n_kv_heads=H, group=4, n_seqs=S,
                          rows_per_seq=16, pages_per_seq=0)
    img, info = cobra.cobra_decode_plan_host(d, r, b, [2048])
    assert info.n_groups == 8 and img.size > 128
    with pytest.raises(RuntimeError):
        cobra.cobra_decode_plan_host(d, r, b, [4096])  # beyond rows_per_seq
