"""Guard bytes around every buffer the device entry points read or write (the stand-in for a
device memory checker, which is closed on this machine): each buffer sits between two 4 KB
guards filled with a pattern, and after every call the guards must be unchanged.  Covers
compress, the decode step (both appends, query projection, scan, combine), the RoPE table
and the RoPE decode on a small model with ragged lengths, a head without K codes and every
group's work split into several chunks."""
import numpy as np
import pytest
import torch

from paper_2609_24298_gb300 import cobra

from .gpu_util import DEV, upload
from .test_gpu_decode import mixed_heads

pytestmark = pytest.mark.gpu
GUARD = 4096
PATTERN = 0xA5


@pytest.fixture(scope="module", autouse=True)
def need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    cobra.lib()


class Guarded:
    """A device buffer of `shape` x `dtype` between two guard regions."""

    def __init__(self, shape, dtype):
        self.nbytes = int(np.prod(shape)) * torch.empty((), dtype=dtype).element_size()
        self.raw = torch.full((GUARD + self.nbytes + GUARD,), PATTERN, dtype=torch.uint8, device=DEV)
        self.t = self.raw[GUARD:GUARD + self.nbytes].view(dtype).view(shape)

    def intact(self) -> bool:
        return bool((self.raw[:GUARD] == PATTERN).all()) and bool((self.raw[GUARD + self.nbytes:] == PATTERN).all())


def check(bufs, what):
    torch.cuda.synchronize()
    assert cobra.cobra_check() == cobra.COBRA_OK, what
    bad = [name for name, g in bufs.items() if not g.intact()]
    assert not bad, f"{what}: guard bytes overwritten around {bad}"


def test_guards_around_compress_step_and_rope_decode():
    L, H, G, S = 2, 2, 4, 3
    rows, n_tok = 3, 256
    rbs = [(0, 1), (64, 2), (128, 1), (40, 3), (96, 2), (30, 5), (128, 1), (16, 8)]  # K(l, h)..., V(l, h)...
    params, srcs = mixed_heads(H, rbs, cfg=47, layers=L)
    block, offs, total, r, b = upload(params, S * rows)
    gen = torch.Generator(device=DEV)
    gen.manual_seed(47)
    bufs = {"cache": Guarded((int(total),), torch.uint8)}
    bufs["cache"].t.zero_()

    # compress the first two rows of every sequence, layer by layer and side by side
    for l in range(L):
        for side in (0, 1):
            x = Guarded((S, n_tok, H, 128), torch.bfloat16)
            x.t.copy_(torch.randn((S, n_tok, H, 128), generator=gen, device=DEV))
            desc = cobra.compress_desc(head0=side * L * H + l * H, layer_stride=H, n_layers=1, n_kv_heads=H,
                                       side=side, n_seqs=S, rows_per_seq=rows, pages_per_seq=0, x_stride_layer=0,
                                       x_stride_seq=n_tok * H * 128, x_stride_tok=H * 128, x_stride_head=128)
            cobra.cobra_compress(block, desc, x.t, 0, n_tok, bufs["cache"].t)
            check(bufs | {"x": x}, f"compress layer {l} side {side}")

    # one decode step: append a token at position 256, then attend over ragged lengths
    Hq = H * G
    cap = np.full(S, rows * 128, np.int32)
    hb = np.where(r > 0, b, 0)
    desc = cobra.decode_desc(k_head0=0, v_head0=L * H, layer_stride=H, n_layers=L, n_kv_heads=H, group=G, n_seqs=S,
                             rows_per_seq=rows, pages_per_seq=0, q_stride_layer=S * Hq * 128, q_stride_seq=Hq * 128,
                             o_stride_layer=S * Hq * 128, o_stride_seq=Hq * 128)
    wsb = cobra.cobra_decode_workspace_size(desc, r, hb, cap)
    bufs["ws"] = Guarded((wsb,), torch.uint8)
    info = cobra.cobra_decode_plan(desc, r, hb, cap, bufs["ws"].t, wsb)
    check(bufs, "plan")
    for name, shape, dt in (("k_new", (L, S, H, 128), torch.bfloat16), ("v_new", (L, S, H, 128), torch.bfloat16),
                            ("q", (L, S, Hq, 128), torch.bfloat16), ("out", (L, S, Hq, 128), torch.float32),
                            ("pos", (S,), torch.int32), ("lens", (S,), torch.int32), ("q_pos", (S,), torch.int32)):
        bufs[name] = Guarded(shape, dt)
    for name in ("k_new", "v_new", "q"):
        bufs[name].t.copy_(torch.randn(bufs[name].t.shape, generator=gen, device=DEV))
    bufs["pos"].t.copy_(torch.tensor([256, 256, 256], dtype=torch.int32))
    bufs["lens"].t.copy_(torch.tensor([257, 129, 1], dtype=torch.int32))
    bufs["q_pos"].t.copy_(torch.tensor([256, 3, 0], dtype=torch.int32))
    adesc = [cobra.compress_desc(head0=side * L * H, layer_stride=H, n_layers=L, n_kv_heads=H, side=side, n_seqs=S,
                                 rows_per_seq=rows, x_stride_layer=S * H * 128, x_stride_seq=H * 128, x_stride_tok=0,
                                 x_stride_head=128) for side in (0, 1)]
    cobra.cobra_decode_step(block, desc, info, adesc[0], adesc[1], bufs["k_new"].t, bufs["v_new"].t, bufs["pos"].t,
                            bufs["q"].t, bufs["cache"].t, bufs["lens"].t, None, bufs["out"].t, bufs["ws"].t, wsb)
    check(bufs, "decode step")
    assert torch.isfinite(bufs["out"].t).all()

    # the RoPE table and decode over the same cache and plan
    max_pos = rows * 128
    tb = cobra.cobra_rope_table_bytes(max_pos)
    bufs["table"] = Guarded((tb // 4,), torch.float32)
    cobra.cobra_rope_table(500000.0, max_pos, bufs["table"].t, tb)
    check(bufs, "rope table")
    for qpos in (None, bufs["q_pos"].t):
        bufs["out"].t.fill_(float("nan"))
        cobra.cobra_decode_rope_attn(block, desc, info, bufs["q"].t, qpos, bufs["table"].t, max_pos, bufs["cache"].t,
                                     bufs["lens"].t, None, bufs["out"].t, bufs["ws"].t, wsb)
        check(bufs, "rope decode")
        assert torch.isfinite(bufs["out"].t).all()
