"""ctypes binding of libcobra (include/cobra.h): the same entry points, argument marshalling
only.  Device buffers are passed as torch tensors (their data_ptr()) or raw integer
addresses; host arrays as numpy arrays.  Every step of the hot path runs in the library's
CUDA kernels; loading fails loudly when libcobra.so is missing.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libcobra.so")

COBRA_OK, COBRA_EINVAL, COBRA_EALIGN, COBRA_EBUDGET, COBRA_ECUDA, COBRA_ETIMEOUT, COBRA_ESPACE = range(7)
ALLOC_DAMPED, ALLOC_EXACT, ALLOC_UNIFORM = 0, 1, 2
D_HEAD = 128

c_int, c_double, c_size_t, c_void_p, c_ll = ctypes.c_int, ctypes.c_double, ctypes.c_size_t, ctypes.c_void_p, ctypes.c_longlong
P_int, P_double, P_float = ctypes.POINTER(c_int), ctypes.POINTER(c_double), ctypes.POINTER(ctypes.c_float)
P_u64, P_i8, P_ll, P_size = ctypes.POINTER(ctypes.c_uint64), ctypes.POINTER(ctypes.c_int8), ctypes.POINTER(c_ll), ctypes.POINTER(c_size_t)


class CobraError(RuntimeError):
    def __init__(self, fn, status):
        super().__init__(f"{fn} failed: status {status} ({status_string(status)})")
        self.status = status


class AllocOpts(ctypes.Structure):
    _fields_ = [("mode", c_int), ("rounds", c_int), ("eta", c_double), ("b_min", c_int), ("b_max", c_int),
                ("r_step", c_int), ("allow_r0", c_int), ("B_min", c_double), ("complete", c_int)]


class CompressDesc(ctypes.Structure):
    _fields_ = [("head0", c_int), ("layer_stride", c_int), ("n_layers", c_int), ("n_kv_heads", c_int),
                ("side", c_int), ("n_seqs", c_int), ("rows_per_seq", c_int), ("pages_per_seq", c_int),
                ("x_stride_layer", c_ll), ("x_stride_seq", c_ll), ("x_stride_tok", c_ll), ("x_stride_head", c_ll)]


class DecodeDesc(ctypes.Structure):
    _fields_ = [("k_head0", c_int), ("v_head0", c_int), ("layer_stride", c_int), ("n_layers", c_int),
                ("n_kv_heads", c_int), ("group", c_int), ("n_seqs", c_int), ("rows_per_seq", c_int),
                ("pages_per_seq", c_int), ("q_stride_layer", c_ll), ("q_stride_seq", c_ll),
                ("o_stride_layer", c_ll), ("o_stride_seq", c_ll)]


class DecodeInfo(ctypes.Structure):
    _fields_ = [("n_groups", c_int), ("n_items", c_int), ("max_row_bytes", c_int), ("max_stage_bytes", c_int)]


# name -> (restype, argtypes)
SIGNATURES = {
    "cobra_version": (c_int, []),
    "cobra_status_string": (ctypes.c_char_p, [c_int]),
    "cobra_alloc_opts_default": (None, [ctypes.POINTER(AllocOpts)]),
    "cobra_allocate": (c_int, [c_int, c_int, P_double, c_double, ctypes.POINTER(AllocOpts), P_int, P_int, P_double,
                               P_double, P_ll]),
    "cobra_calibrate_heads": (c_int, [c_int, c_int, c_void_p, c_int, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                                      c_void_p]),
    "cobra_measure_distortion": (c_int, [c_int, c_int, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                                         c_int, P_int, c_int, P_int, c_void_p, c_void_p, c_void_p]),
    "cobra_allocate_tables": (c_int, [c_int, c_int, c_int, P_int, c_int, P_int, P_double, c_double, P_int, P_int,
                                      P_double, P_ll]),
    "cobra_loading_factor": (c_int, [c_int, P_double]),
    "cobra_hadamard": (c_int, [c_int, P_i8, P_double]),
    "cobra_calibrate_head": (c_int, [c_int, c_int, P_float, c_int, P_float, P_double, P_double, P_double, P_double]),
    "cobra_fuse_basis": (c_int, [c_int, c_int, c_int, P_double, P_double, P_i8, P_float, P_float]),
    "cobra_row_bytes": (c_size_t, [c_int, c_int]),
    "cobra_plan_layout": (c_int, [c_int, P_int, P_int, c_ll, P_u64, P_u64]),
    "cobra_params_bytes": (c_int, [c_int, P_int, P_size]),
    "cobra_params_build": (c_int, [c_void_p, c_size_t, c_int, P_int, P_int, P_float, P_u64, P_float, P_float,
                                   c_void_p]),
    "cobra_params_image": (c_int, [c_void_p, c_size_t, c_int, P_int, P_int, P_float, P_u64, P_float, P_float]),
    "cobra_params_verify": (c_int, [c_void_p, c_size_t]),
    "cobra_params_upload": (c_int, [c_void_p, c_size_t, c_void_p, c_size_t, c_void_p]),
    "cobra_compress": (c_int, [c_void_p, ctypes.POINTER(CompressDesc), c_void_p, c_int, c_int, c_void_p, c_void_p,
                               c_void_p]),
    "cobra_append": (c_int, [c_void_p, ctypes.POINTER(CompressDesc), c_void_p, c_void_p, c_void_p, c_void_p, c_void_p]),
    "cobra_decode_workspace_size": (c_int, [ctypes.POINTER(DecodeDesc), P_int, P_int, P_int, P_size]),
    "cobra_decode_plan": (c_int, [ctypes.POINTER(DecodeDesc), P_int, P_int, P_int, c_void_p, c_size_t,
                                  ctypes.POINTER(DecodeInfo), c_void_p]),
    "cobra_decode_qproj_append": (c_int, [c_void_p, ctypes.POINTER(DecodeDesc), ctypes.POINTER(DecodeInfo), c_void_p,
                                          ctypes.POINTER(CompressDesc), c_void_p, c_void_p, c_void_p, c_void_p,
                                          c_void_p, c_size_t, c_void_p]),
    "cobra_decode_step": (c_int, [c_void_p, ctypes.POINTER(DecodeDesc), ctypes.POINTER(DecodeInfo),
                                  ctypes.POINTER(CompressDesc), ctypes.POINTER(CompressDesc), c_void_p, c_void_p,
                                  c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, c_size_t,
                                  c_void_p]),
    "cobra_decode_plan_host": (c_int, [ctypes.POINTER(DecodeDesc), P_int, P_int, P_int, c_void_p, c_size_t, P_size,
                                       ctypes.POINTER(DecodeInfo)]),
    "cobra_decode_attn": (c_int, [c_void_p, ctypes.POINTER(DecodeDesc), ctypes.POINTER(DecodeInfo), c_void_p,
                                  c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, c_size_t, c_void_p]),
    "cobra_decode_qproj": (c_int, [c_void_p, ctypes.POINTER(DecodeDesc), ctypes.POINTER(DecodeInfo), c_void_p,
                                   c_void_p, c_size_t, c_void_p]),
    "cobra_decode_scan": (c_int, [c_void_p, ctypes.POINTER(DecodeDesc), ctypes.POINTER(DecodeInfo), c_void_p,
                                  c_void_p, c_void_p, c_void_p, c_size_t, c_void_p]),
    "cobra_decode_combine": (c_int, [c_void_p, ctypes.POINTER(DecodeDesc), ctypes.POINTER(DecodeInfo), c_void_p,
                                     c_void_p, c_void_p, c_size_t, c_void_p]),
    "cobra_decode_attn_static": (c_int, [c_void_p, ctypes.POINTER(DecodeDesc), c_void_p, c_void_p, c_void_p, c_void_p,
                                         c_void_p, c_void_p]),
    "cobra_rope_table_bytes": (c_int, [c_int, P_size]),
    "cobra_rope_table": (c_int, [c_double, c_int, c_void_p, c_size_t, c_void_p]),
    "cobra_decode_rope_attn": (c_int, [c_void_p, ctypes.POINTER(DecodeDesc), ctypes.POINTER(DecodeInfo), c_void_p,
                                       c_void_p, c_void_p, c_int, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                                       c_size_t, c_void_p]),
    "cobra_check": (c_int, [c_void_p]),
    "cobra_selftest_wait_timeout": (c_int, [ctypes.c_ulonglong, c_void_p]),
}

_lib = None


def lib():
    """The loaded library (raises if libcobra.so has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"libcobra.so not found at {LIB_PATH}; run __graft_entry__.build() first")
        L = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in SIGNATURES.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def status_string(s: int) -> str:
    return lib().cobra_status_string(s).decode()


def _chk(fn, st):
    if st != COBRA_OK:
        raise CobraError(fn, st)


def _ptr(x):
    """Device address of a torch tensor / int / None."""
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if not x.is_contiguous():
        # the library addresses buffers through the strides in its descriptors, which refer
        # to the memory itself: a permuted or sliced view would be read with the wrong layout
        raise ValueError("device tensors passed to libcobra must be contiguous; describe other layouts "
                         "with the descriptor strides over a contiguous buffer")
    return x.data_ptr()


def _np(a, dtype, ctype):
    a = np.ascontiguousarray(a, dtype=dtype)
    return a, a.ctypes.data_as(ctypes.POINTER(ctype))


def _stream(s):
    if s is None:
        return None
    if isinstance(s, int):
        return s
    return s.cuda_stream


def cobra_version() -> int:
    return lib().cobra_version()


def alloc_opts(**kw) -> AllocOpts:
    o = AllocOpts()
    lib().cobra_alloc_opts_default(ctypes.byref(o))
    for k, v in kw.items():
        setattr(o, k, v)
    return o


def cobra_allocate(w, bpd: float, opts: AllocOpts | None = None):
    w, wp = _np(w, np.float64, c_double)
    n, d = w.shape
    r = np.zeros(n, np.int32)
    b = np.zeros(n, np.int32)
    bud = np.zeros(n, np.float64)
    dist = np.zeros(n, np.float64)
    rate = c_ll(0)
    st = lib().cobra_allocate(n, d, wp, float(bpd), ctypes.byref(opts) if opts is not None else None,
                              r.ctypes.data_as(P_int), b.ctypes.data_as(P_int), bud.ctypes.data_as(P_double),
                              dist.ctypes.data_as(P_double), ctypes.byref(rate))
    _chk("cobra_allocate", st)
    return dict(r=r, b=b, budget=bud, dist=dist, rate_bits=rate.value)


def cobra_allocate_tables(tables, r_list, b_list, bpd: float, d: int = 128):
    """Exact DP on explicit tables [n_heads][len(r_list)][len(b_list)] (App. E)."""
    D, Dp = _np(np.ascontiguousarray(tables, dtype=np.float64), np.float64, c_double)
    rl, rlp = _np(r_list, np.int32, c_int)
    bl, blp = _np(b_list, np.int32, c_int)
    n = D.shape[0]
    if D.shape != (n, len(rl), len(bl)):
        raise ValueError("tables must be [n_heads][len(r_list)][len(b_list)]")
    r = np.zeros(n, np.int32)
    b = np.zeros(n, np.int32)
    dist = np.zeros(n, np.float64)
    rate = c_ll(0)
    st = lib().cobra_allocate_tables(n, int(d), len(rl), rlp, len(bl), blp, Dp, float(bpd), r.ctypes.data_as(P_int),
                                     b.ctypes.data_as(P_int), dist.ctypes.data_as(P_double), ctypes.byref(rate))
    _chk("cobra_allocate_tables", st)
    return dict(r=r, b=b, dist=dist, rate_bits=rate.value)


def cobra_calibrate_heads(x, q, mu, lam, U, w, stream=None):
    """Device calibration of many heads (steps 1-2); x [n][n_tok][128], q [n][n_q][128] or
    None; outputs are device fp64 tensors mu, lam, w [n][128] and U [n][128 * 128]."""
    n_heads, n_tok = int(x.shape[0]), int(x.shape[1])
    n_q = int(q.shape[1]) if q is not None else 0
    st = lib().cobra_calibrate_heads(n_heads, n_tok, _ptr(x), n_q, _ptr(q), _ptr(mu), _ptr(lam), _ptr(U), _ptr(w),
                                     _stream(stream))
    _chk("cobra_calibrate_heads", st)


def cobra_measure_distortion(x, U, lam, w, mu, signs, r_list, b_list, coords, D, stream=None):
    """Measured distortion tables on the device (App. E); all array arguments are device
    tensors except the two host lists.  lam and w are the calibration's eigenvalues and
    allocator weights (fp64); the library derives the error weights from them."""
    rl, rlp = _np(r_list, np.int32, c_int)
    bl, blp = _np(b_list, np.int32, c_int)
    n_heads, n_tok = int(x.shape[0]), int(x.shape[1])
    st = lib().cobra_measure_distortion(n_heads, n_tok, _ptr(x), _ptr(U), _ptr(lam), _ptr(w), _ptr(mu),
                                        _ptr(signs), len(rl), rlp, len(bl), blp, _ptr(coords), _ptr(D),
                                        _stream(stream))
    _chk("cobra_measure_distortion", st)


def cobra_loading_factor(b: int) -> float:
    L = c_double(0)
    _chk("cobra_loading_factor", lib().cobra_loading_factor(b, ctypes.byref(L)))
    return L.value


def cobra_hadamard(r: int, signs) -> np.ndarray:
    s, sp = _np(signs, np.int8, ctypes.c_int8)
    H = np.zeros((r, r), np.float64)
    _chk("cobra_hadamard", lib().cobra_hadamard(r, sp, H.ctypes.data_as(P_double)))
    return H


def cobra_calibrate_head(x, q=None):
    x, xp = _np(x, np.float32, ctypes.c_float)
    n, d = x.shape
    if q is not None:
        q, qp = _np(np.asarray(q, np.float32).reshape(-1, d), np.float32, ctypes.c_float)
        nq = q.shape[0]
    else:
        qp, nq = None, 0
    mu, lam, w = np.zeros(d), np.zeros(d), np.zeros(d)
    U = np.zeros(d * d)
    st = lib().cobra_calibrate_head(n, d, xp, nq, qp, mu.ctypes.data_as(P_double), lam.ctypes.data_as(P_double),
                                    U.ctypes.data_as(P_double), w.ctypes.data_as(P_double))
    _chk("cobra_calibrate_head", st)
    return dict(mu=mu, lam=lam, U=U.reshape(d, d).T.copy(), w=w)  # U[:, j] = direction j


def cobra_fuse_basis(U, lam, r: int, b: int, signs):
    U = np.asarray(U, np.float64)
    d = U.shape[0]
    Ucm, Up = _np(U.T, np.float64, c_double)  # column-major: U[i + j*d]
    lam, lp = _np(lam, np.float64, c_double)
    s, sp = _np(signs, np.int8, ctypes.c_int8)
    W = np.zeros(d * max(r, 0), np.float32)
    delta = ctypes.c_float(0)
    st = lib().cobra_fuse_basis(d, r, b, Up, lp, sp, W.ctypes.data_as(P_float) if r else None, ctypes.byref(delta))
    _chk("cobra_fuse_basis", st)
    return W.reshape(r, d).T.copy(), np.float32(delta.value)  # W[:, j] = column j


def cobra_row_bytes(r: int, b: int) -> int:
    return lib().cobra_row_bytes(r, b)


def cobra_plan_layout(r, b, n_slots: int):
    r, rp = _np(r, np.int32, c_int)
    b, bp = _np(b, np.int32, c_int)
    offs = np.zeros(len(r), np.uint64)
    total = ctypes.c_uint64(0)
    st = lib().cobra_plan_layout(len(r), rp, bp, int(n_slots), offs.ctypes.data_as(P_u64), ctypes.byref(total))
    _chk("cobra_plan_layout", st)
    return offs, int(total.value)


def cobra_params_bytes(r) -> int:
    r, rp = _np(r, np.int32, c_int)
    n = c_size_t(0)
    _chk("cobra_params_bytes", lib().cobra_params_bytes(len(r), rp, ctypes.byref(n)))
    return n.value


def cobra_params_build(dev_block, nbytes: int, r, b, delta, cache_off, W_list, mu_all, stream=None):
    """W_list: per head a (d, r_h) float32 matrix (column j = basis column j)."""
    r, rp = _np(r, np.int32, c_int)
    b, bp = _np(b, np.int32, c_int)
    delta, dp = _np(delta, np.float32, ctypes.c_float)
    offs, op = _np(cache_off, np.uint64, ctypes.c_uint64)
    cols = [np.asarray(W, np.float32).T.reshape(-1) for W in W_list]  # column-major per head
    Wall = np.concatenate(cols) if cols else np.zeros(1, np.float32)
    Wall, Wp = _np(Wall if Wall.size else np.zeros(1, np.float32), np.float32, ctypes.c_float)
    mu, mp = _np(mu_all, np.float32, ctypes.c_float)
    st = lib().cobra_params_build(_ptr(dev_block), int(nbytes), len(r), rp, bp, dp, op, Wp, mp, _stream(stream))
    _chk("cobra_params_build", st)


def cobra_params_image(r, b, delta, cache_off, W_list, mu_all) -> np.ndarray:
    """The parameter block as host bytes (uint8), with its checksum: a calibration checkpoint."""
    r, rp = _np(r, np.int32, c_int)
    b, bp = _np(b, np.int32, c_int)
    delta, dp = _np(delta, np.float32, ctypes.c_float)
    offs, op = _np(cache_off, np.uint64, ctypes.c_uint64)
    cols = [np.asarray(W, np.float32).T.reshape(-1) for W in W_list]  # column-major per head
    Wall = np.concatenate(cols) if cols else np.zeros(1, np.float32)
    Wall, Wp = _np(Wall if Wall.size else np.zeros(1, np.float32), np.float32, ctypes.c_float)
    mu, mp = _np(mu_all, np.float32, ctypes.c_float)
    img = np.zeros(cobra_params_bytes(r), np.uint8)
    st = lib().cobra_params_image(img.ctypes.data_as(c_void_p), img.nbytes, len(r), rp, bp, dp, op, Wp, mp)
    _chk("cobra_params_image", st)
    return img


def cobra_params_verify(image) -> int:
    """Status of a host image check (does not raise): COBRA_OK or COBRA_EINVAL."""
    img = np.ascontiguousarray(image, np.uint8)
    return lib().cobra_params_verify(img.ctypes.data_as(c_void_p), img.nbytes)


def cobra_params_upload(dev_block, nbytes: int, image, stream=None):
    img = np.ascontiguousarray(image, np.uint8)
    st = lib().cobra_params_upload(_ptr(dev_block), int(nbytes), img.ctypes.data_as(c_void_p), img.nbytes,
                                   _stream(stream))
    _chk("cobra_params_upload", st)


def compress_desc(**kw) -> CompressDesc:
    d = CompressDesc()
    for k, v in kw.items():
        setattr(d, k, v)
    return d


def decode_desc(**kw) -> DecodeDesc:
    d = DecodeDesc()
    for k, v in kw.items():
        setattr(d, k, v)
    return d


def cobra_compress(params, desc: CompressDesc, x, t0: int, n_tok: int, cache, page_table=None, stream=None):
    st = lib().cobra_compress(_ptr(params), ctypes.byref(desc), _ptr(x), int(t0), int(n_tok), _ptr(cache),
                              _ptr(page_table), _stream(stream))
    _chk("cobra_compress", st)


def cobra_append(params, desc: CompressDesc, x, pos, cache, page_table=None, stream=None):
    st = lib().cobra_append(_ptr(params), ctypes.byref(desc), _ptr(x), _ptr(pos), _ptr(cache), _ptr(page_table),
                            _stream(stream))
    _chk("cobra_append", st)


def cobra_decode_workspace_size(desc: DecodeDesc, head_r, head_b, seq_cap) -> int:
    hr, hrp = _np(head_r, np.int32, c_int)
    hb, hbp = _np(head_b, np.int32, c_int)
    sc, scp = _np(seq_cap, np.int32, c_int)
    n = c_size_t(0)
    _chk("cobra_decode_workspace_size", lib().cobra_decode_workspace_size(ctypes.byref(desc), hrp, hbp, scp, ctypes.byref(n)))
    return n.value


def cobra_decode_plan(desc: DecodeDesc, head_r, head_b, seq_cap, workspace, ws_bytes: int, stream=None) -> DecodeInfo:
    hr, hrp = _np(head_r, np.int32, c_int)
    hb, hbp = _np(head_b, np.int32, c_int)
    sc, scp = _np(seq_cap, np.int32, c_int)
    info = DecodeInfo()
    st = lib().cobra_decode_plan(ctypes.byref(desc), hrp, hbp, scp, _ptr(workspace), int(ws_bytes), ctypes.byref(info),
                                 _stream(stream))
    _chk("cobra_decode_plan", st)
    return info


def cobra_decode_plan_host(desc: DecodeDesc, head_r, head_b, seq_cap):
    """The plan as host bytes (the first bytes of a planned workspace) and its DecodeInfo."""
    hr, hrp = _np(head_r, np.int32, c_int)
    hb, hbp = _np(head_b, np.int32, c_int)
    sc, scp = _np(seq_cap, np.int32, c_int)
    n = c_size_t(0)
    info = DecodeInfo()
    st = lib().cobra_decode_plan_host(ctypes.byref(desc), hrp, hbp, scp, None, 0, ctypes.byref(n), ctypes.byref(info))
    if st != COBRA_EINVAL or n.value == 0:
        _chk("cobra_decode_plan_host", st)
    img = np.zeros(n.value, np.uint8)
    st = lib().cobra_decode_plan_host(ctypes.byref(desc), hrp, hbp, scp, img.ctypes.data, img.size, ctypes.byref(n),
                                      ctypes.byref(info))
    _chk("cobra_decode_plan_host", st)
    return img, info


def cobra_decode_qproj_append(params, desc: DecodeDesc, info: DecodeInfo, q, kdesc: CompressDesc, k_new, pos, cache,
                              page_table, workspace, ws_bytes: int, stream=None):
    st = lib().cobra_decode_qproj_append(_ptr(params), ctypes.byref(desc), ctypes.byref(info), _ptr(q),
                                         ctypes.byref(kdesc), _ptr(k_new), _ptr(pos), _ptr(cache), _ptr(page_table),
                                         _ptr(workspace), int(ws_bytes), _stream(stream))
    _chk("cobra_decode_qproj_append", st)


def cobra_decode_step(params, desc: DecodeDesc, info: DecodeInfo, kdesc: CompressDesc, vdesc: CompressDesc, k_new,
                      v_new, pos, q, cache, seq_lens, page_table, out, workspace, ws_bytes: int, stream=None):
    st = lib().cobra_decode_step(_ptr(params), ctypes.byref(desc), ctypes.byref(info), ctypes.byref(kdesc),
                                 ctypes.byref(vdesc), _ptr(k_new), _ptr(v_new), _ptr(pos), _ptr(q), _ptr(cache),
                                 _ptr(seq_lens), _ptr(page_table), _ptr(out), _ptr(workspace), int(ws_bytes),
                                 _stream(stream))
    _chk("cobra_decode_step", st)


def cobra_decode_attn(params, desc: DecodeDesc, info: DecodeInfo, q, cache, seq_lens, page_table, out, workspace,
                      ws_bytes: int, stream=None):
    st = lib().cobra_decode_attn(_ptr(params), ctypes.byref(desc), ctypes.byref(info), _ptr(q), _ptr(cache),
                                 _ptr(seq_lens), _ptr(page_table), _ptr(out), _ptr(workspace), int(ws_bytes),
                                 _stream(stream))
    _chk("cobra_decode_attn", st)


def cobra_decode_qproj(params, desc, info, q, workspace, ws_bytes: int, stream=None):
    st = lib().cobra_decode_qproj(_ptr(params), ctypes.byref(desc), ctypes.byref(info), _ptr(q), _ptr(workspace),
                                  int(ws_bytes), _stream(stream))
    _chk("cobra_decode_qproj", st)


def cobra_decode_scan(params, desc, info, cache, seq_lens, page_table, workspace, ws_bytes: int, stream=None):
    st = lib().cobra_decode_scan(_ptr(params), ctypes.byref(desc), ctypes.byref(info), _ptr(cache), _ptr(seq_lens),
                                 _ptr(page_table), _ptr(workspace), int(ws_bytes), _stream(stream))
    _chk("cobra_decode_scan", st)


def cobra_decode_combine(params, desc, info, seq_lens, out, workspace, ws_bytes: int, stream=None):
    st = lib().cobra_decode_combine(_ptr(params), ctypes.byref(desc), ctypes.byref(info), _ptr(seq_lens), _ptr(out),
                                    _ptr(workspace), int(ws_bytes), _stream(stream))
    _chk("cobra_decode_combine", st)


def cobra_rope_table_bytes(max_pos: int) -> int:
    n = c_size_t(0)
    _chk("cobra_rope_table_bytes", lib().cobra_rope_table_bytes(int(max_pos), ctypes.byref(n)))
    return n.value


def cobra_rope_table(theta: float, max_pos: int, table, table_bytes: int, stream=None):
    """Fill a device angle table for RoPE decode (cos / sin of the rotary angles)."""
    st = lib().cobra_rope_table(float(theta), int(max_pos), _ptr(table), int(table_bytes), _stream(stream))
    _chk("cobra_rope_table", st)


def cobra_decode_rope_attn(params, desc: DecodeDesc, info: DecodeInfo, q, q_pos, rope_table, max_pos: int, cache,
                           seq_lens, page_table, out, workspace, ws_bytes: int, stream=None):
    """Decode attention with the rotary embedding applied to the rebuilt keys and the query."""
    st = lib().cobra_decode_rope_attn(_ptr(params), ctypes.byref(desc), ctypes.byref(info), _ptr(q), _ptr(q_pos),
                                      _ptr(rope_table), int(max_pos), _ptr(cache), _ptr(seq_lens), _ptr(page_table),
                                      _ptr(out), _ptr(workspace), int(ws_bytes), _stream(stream))
    _chk("cobra_decode_rope_attn", st)


def cobra_decode_attn_static(params, desc: DecodeDesc, q, cache, seq_lens, page_table, out, stream=None):
    """Decode attention for callers that cannot allocate device memory: the workspace is a
    fixed array inside the library (see include/cobra.h)."""
    st = lib().cobra_decode_attn_static(_ptr(params), ctypes.byref(desc), _ptr(q), _ptr(cache), _ptr(seq_lens),
                                        _ptr(page_table), _ptr(out), _stream(stream))
    _chk("cobra_decode_attn_static", st)


def cobra_check(stream=None) -> int:
    """Returns the status code (does not raise) so callers can test for COBRA_ETIMEOUT."""
    return lib().cobra_check(_stream(stream))


def cobra_selftest_wait_timeout(limit_ns: int, stream=None):
    """Launch the library's bounded-wait self-test (one warp waits on a barrier nothing
    completes); the next cobra_check returns COBRA_ETIMEOUT."""
    _chk("cobra_selftest_wait_timeout", lib().cobra_selftest_wait_timeout(int(limit_ns), _stream(stream)))
