"""Device status reporting without any GPU fault: an expired bounded wait (the library's
self-test waits on a barrier that nothing completes) and skipped work (an append position past
the cache's capacity) are reported by cobra_check, which clears the status; the context stays
usable afterwards."""
import numpy as np
import pytest
import torch

from paper_2609_24298_gb300 import cobra, synth

from .gpu_util import DEV, oracle_head, upload

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    cobra.lib()


def _small_cache():
    srcs = [synth.HeadSource(17, 0, i, 0, (0.5, 2.0)) for i in range(2)]
    params = [oracle_head(s, r, b) for s, (r, b) in zip(srcs, [(32, 2), (16, 3)])]
    block, offs, total, r, b = upload(params, 2)
    cache = torch.zeros(total, dtype=torch.uint8, device=DEV)
    x = torch.tensor(np.stack([np.stack([s.tokens(200, seq=0) for s in srcs], axis=1)]), dtype=torch.bfloat16,
                     device=DEV)
    desc = cobra.compress_desc(head0=0, layer_stride=2, n_layers=1, n_kv_heads=2, side=0, n_seqs=1, rows_per_seq=2,
                               x_stride_layer=0, x_stride_seq=200 * 2 * 128, x_stride_tok=2 * 128, x_stride_head=128)
    return block, cache, x, desc


def test_expired_wait_is_reported_and_cleared():
    assert cobra.cobra_check() == cobra.COBRA_OK
    cobra.cobra_selftest_wait_timeout(1_000_000)  # 1 ms
    assert cobra.cobra_check() == cobra.COBRA_ETIMEOUT
    assert cobra.cobra_check() == cobra.COBRA_OK  # the check cleared it
    # the context still runs work: compress a few tokens
    block, cache, x, desc = _small_cache()
    cobra.cobra_compress(block, desc, x, 0, 200, cache)
    assert cobra.cobra_check() == cobra.COBRA_OK
    assert int(cache.count_nonzero()) > 0


def test_append_past_capacity_is_skipped_and_flagged():
    block, cache, x, desc = _small_cache()
    cobra.cobra_compress(block, desc, x, 0, 200, cache)
    assert cobra.cobra_check() == cobra.COBRA_OK
    before = cache.clone()
    d2 = cobra.compress_desc(head0=0, layer_stride=2, n_layers=1, n_kv_heads=2, side=0, n_seqs=1, rows_per_seq=2,
                             x_stride_layer=0, x_stride_seq=2 * 128, x_stride_tok=0, x_stride_head=128)
    xt = x[:, 0].contiguous()
    pos = torch.tensor([256], dtype=torch.int32, device=DEV)  # capacity is 2 rows = 256 tokens
    cobra.cobra_append(block, d2, xt, pos, cache)
    assert cobra.cobra_check() == cobra.COBRA_EINVAL
    assert torch.equal(cache, before)
    assert cobra.cobra_check() == cobra.COBRA_OK
