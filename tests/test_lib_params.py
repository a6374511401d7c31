"""CPU tests of the parameter block as a host image (the calibration checkpoint; Table
alg:kvrobin step 6 stores the calibration once per model): its layout holds the inputs where
the header and head table say, the header's checksum is the FNV-1a 64 of the block (restated
here from the published algorithm), a file round trip verifies, and any corruption, a wrong
version or a truncated image is rejected before a device is touched."""
import os
import struct

import numpy as np
import pytest

from paper_2609_24298_gb300 import cobra

from .gpu_util import oracle_head


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not os.path.exists(cobra.LIB_PATH):
        from paper_2609_24298_gb300 import build

        build.build()
    cobra.lib()


def fnv1a64(data: bytes) -> int:
    h = 0xCBF29CE484222325
    for c in data:
        h = ((h ^ c) * 0x100000001B3) & 0xFFFFFFFFFFFFFFFF
    return h


def image():
    from paper_2609_24298_gb300 import synth

    rb = [(64, 2), (0, 1), (18, 3), (128, 1)]
    srcs = [synth.HeadSource(51, 0, h, 0, (0.3, 2.5)) for h in range(len(rb))]
    params = [oracle_head(s, r, b) for s, (r, b) in zip(srcs, rb)]
    r = np.array([p["r"] for p in params], np.int32)
    b = np.array([p["b"] if p["r"] else 1 for p in params], np.int32)
    delta = np.array([p["delta"] if p["r"] else 0.0 for p in params], np.float32)
    offs, _ = cobra.cobra_plan_layout(r, b, 6)
    mu = np.stack([p["mu"] for p in params]).astype(np.float32)
    img = cobra.cobra_params_image(r, b, delta, offs, [p["W"] for p in params], mu.reshape(-1))
    return img, params, r, b, delta, offs, mu


def test_image_layout_and_checksum():
    img, params, r, b, delta, offs, mu = image()
    raw = img.tobytes()
    magic, version, n_heads, d, heads_off, pool_off, pool_floats, checksum = struct.unpack_from("<IIiiQQQQ", raw, 0)
    assert (magic, n_heads, d, heads_off) == (0x52424F43, 4, 128, 64)
    assert pool_off % 256 == 0 and pool_off + 4 * pool_floats == len(raw)
    zeroed = raw[:40] + bytes(8) + raw[48:]
    assert checksum == fnv1a64(zeroed)
    pool = np.frombuffer(raw, np.float32, count=pool_floats, offset=pool_off)
    for h, p in enumerate(params):
        er, eb, edelta, einv, coff, w_off, mu_off, wmu_off = struct.unpack_from("<iiffQQQQ", raw, heads_off + 64 * h)
        assert er == r[h] and coff == offs[h]
        if er:
            assert eb == b[h] and edelta == delta[h]
        W = np.asarray(p["W"], np.float32)
        assert np.array_equal(pool[w_off:w_off + 128 * er].reshape(er, 128).T, W)
        assert np.array_equal(pool[mu_off:mu_off + 128], mu[h])
        wmu = W.astype(np.float64).T @ mu[h].astype(np.float64)
        assert np.allclose(pool[wmu_off:wmu_off + er], wmu, rtol=1e-6, atol=1e-7)
    assert cobra.cobra_params_verify(img) == cobra.COBRA_OK


def test_file_round_trip(tmp_path):
    img = image()[0]
    path = tmp_path / "calibration.bin"
    img.tofile(path)
    back = np.fromfile(path, np.uint8)
    assert np.array_equal(back, img)
    assert cobra.cobra_params_verify(back) == cobra.COBRA_OK


def test_corrupt_images_are_rejected():
    img = image()[0]
    n = img.nbytes
    for pos in (8, 70, 200, n // 2, n - 1):  # header, head table, padding / pool
        bad = img.copy()
        bad[pos] ^= 0x10
        assert cobra.cobra_params_verify(bad) == cobra.COBRA_EINVAL, pos
    assert cobra.cobra_params_verify(img[:-4]) == cobra.COBRA_EINVAL
    assert cobra.cobra_params_verify(np.concatenate([img, np.zeros(256, np.uint8)])) == cobra.COBRA_EINVAL
    bad = img.copy()
    bad[4] = 99  # version
    assert cobra.cobra_params_verify(bad) == cobra.COBRA_EINVAL
    # the upload checks the image before any device work
    with pytest.raises(cobra.CobraError) as e:
        cobra.cobra_params_upload(256, n, img[:-4])
    assert e.value.status == cobra.COBRA_EINVAL


def resign(raw: bytearray) -> np.ndarray:
    """The image with its header checksum recomputed (so that only the field checks can reject it)."""
    raw[40:48] = bytes(8)
    raw[40:48] = struct.pack("<Q", fnv1a64(bytes(raw)))
    return np.frombuffer(bytes(raw), np.uint8)


@pytest.mark.parametrize("field", ["delta_inf", "delta_nan", "inv_delta", "r0_b", "r0_delta", "r0_inv"])
def test_inconsistent_head_fields_are_rejected_with_a_valid_checksum(field):
    """A checkpoint written by another tool with a correct checksum is still checked field by
    field, as strictly as the build path: a finite step, its reciprocal as the build rounds it,
    and zeros in the quantiser fields of a head without codes (Sec. 3, static scalar quantizer)."""
    img = image()[0]
    raw = bytearray(img.tobytes())
    heads_off = 64
    h_codes, h_empty = 0, 1  # rb = [(64, 2), (0, 1), ...]
    base = heads_off + 64 * h_codes
    if field == "delta_inf":
        struct.pack_into("<f", raw, base + 8, float("inf"))
        struct.pack_into("<f", raw, base + 12, 0.0)
    elif field == "delta_nan":
        struct.pack_into("<f", raw, base + 8, float("nan"))
    elif field == "inv_delta":
        inv = struct.unpack_from("<I", raw, base + 12)[0]
        struct.pack_into("<I", raw, base + 12, inv + 1)  # one ulp off
    else:
        e = heads_off + 64 * h_empty
        off = {"r0_b": 4, "r0_delta": 8, "r0_inv": 12}[field]
        if field == "r0_b":
            struct.pack_into("<i", raw, e + off, 3)
        else:
            struct.pack_into("<f", raw, e + off, 0.5)
    good = resign(bytearray(img.tobytes()))
    assert cobra.cobra_params_verify(good) == cobra.COBRA_OK  # re-signing alone keeps it valid
    assert cobra.cobra_params_verify(resign(raw)) == cobra.COBRA_EINVAL
