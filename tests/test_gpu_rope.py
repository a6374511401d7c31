"""GPU parity of cobra_decode_rope_attn (decode with the rotary embedding applied to the
rebuilt keys and the query; the paper compresses K before it, Sec. 5 "Scope") against
oracle.rope over the same packed codes: max over query heads of ||o - o*||_inf / ||o*||_inf
<= 2e-3, as for the plain decode.  The keys are rebuilt from fp16 hi + lo parts of W_K and
scored with hi + lo parts of both operands (about 22 bits each), the angles composed from
fp32 tables of fp64 values (relative error ~1e-7), so the measured error sits far below the
bound; the cases span every bit width, r = 0 on either side, ragged and empty sequences, the
paged layout, groups of 4 and 8, explicit query positions and a position near 32k."""
import numpy as np
import pytest
import torch

from paper_2609_24298_gb300 import cobra

from .gpu_util import DEV, rel_err
from .test_gpu_decode import mixed_heads, run_decode

pytestmark = pytest.mark.gpu
TOL = 2e-3
LLAMA3_THETA = 500000.0


@pytest.fixture(scope="module", autouse=True)
def need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    cobra.lib()


@pytest.mark.parametrize("bk,bv", [(1, 8), (2, 7), (3, 6), (4, 5), (5, 4), (6, 3), (7, 2), (8, 1)])
def test_every_bit_width(bk, bv):
    rbs = [(128 if bk <= 2 else 48, bk), (18, bk), (128 if bv <= 2 else 40, bv), (2, bv)]
    params, srcs = mixed_heads(2, rbs, cfg=32 + bk)
    o, ref, _ = run_decode(params, srcs, 1, 2, 4, [700], rope=dict(theta=LLAMA3_THETA))
    assert rel_err(o, ref) < TOL


def test_zero_rank_sides():
    rbs = [(0, 1), (32, 3), (64, 2), (0, 1)]
    params, srcs = mixed_heads(2, rbs, cfg=41)
    o, ref, _ = run_decode(params, srcs, 1, 2, 4, [300], rope=dict(theta=10000.0))
    assert rel_err(o, ref) < TOL


def test_ragged_lengths_empty_sequence_and_positions():
    rbs = [(64, 2), (100, 1), (32, 4), (128, 2)]
    params, srcs = mixed_heads(2, rbs, cfg=42)
    lens = [1, 127, 128, 129, 255, 256, 257, 0, 1000]
    qpos = [0, 126, 500, 129, 3, 1023, 256, 0, 999]
    o, ref, _ = run_decode(params, srcs, 1, 2, 4, lens, cap=[1024] * len(lens),
                           rope=dict(theta=LLAMA3_THETA, q_pos=qpos, max_pos=1024))
    assert rel_err(np.delete(o, 7, axis=1), np.delete(ref, 7, axis=1)) < TOL
    assert np.all(o[:, 7] == 0)


def test_paged_layout_two_layers():
    rbs = [(64, 2), (30, 3), (128, 1), (16, 8), (48, 2), (96, 1), (20, 5), (64, 3)]
    params, srcs = mixed_heads(2, rbs, cfg=43, layers=2)
    o, ref, _ = run_decode(params, srcs, 2, 2, 4, [900, 300, 513], paged=True, rope=dict(theta=LLAMA3_THETA))
    assert rel_err(o, ref) < TOL


def test_group_of_eight():
    rbs = [(32, 2), (14, 4), (128, 1), (40, 3)]
    params, srcs = mixed_heads(2, rbs, cfg=44)
    o, ref, _ = run_decode(params, srcs, 1, 2, 8, [400, 130], rope=dict(theta=1000000.0))
    assert rel_err(o, ref) < TOL


def test_long_sequence_and_peaked_queries():
    """32k positions (the largest angles), queries scaled so that attention is peaked, several
    chunks per head."""
    rbs = [(128, 2), (64, 3), (128, 2), (96, 2)]
    params, srcs = mixed_heads(2, rbs, cfg=45)
    o, ref, _ = run_decode(params, srcs, 1, 2, 4, [32768, 20000], q_scale=3.0, rope=dict(theta=LLAMA3_THETA))
    assert rel_err(o, ref) < TOL


def test_positions_outside_the_table_are_reported():
    rbs = [(32, 2), (32, 2), (32, 2), (32, 2)]
    params, srcs = mixed_heads(2, rbs, cfg=46)
    with pytest.raises(AssertionError):
        run_decode(params, srcs, 1, 2, 4, [200], rope=dict(theta=LLAMA3_THETA, q_pos=[5000], max_pos=256))
    assert cobra.cobra_check() == cobra.COBRA_OK  # the status word was read and cleared
