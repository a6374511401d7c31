"""Packed code-row layout of the compressed cache (Table alg:kvrobin step 8 "Cache z_t";
App. G "packed b-bit codes").

The paper fixes only that the cache holds b-bit codes of the r retained channels, with no
per-token metadata (App. "effective bpd": the per-(channel, token) cost is exactly r*b/d).
The bit order inside a row is this implementation's choice (format v1); this module is its
plain definition.  Sizes:

  code row   128 consecutive tokens of one head: 128*r*b bits = 16*r*b bytes (a multiple of
             16, so rows are 16-byte aligned when the head region is).
  strip s    channels (2s, 2s+1) of all 128 tokens: bytes [32*b*s, 32*b*(s+1)) of the row;
             a row has r/2 strips (r is even).
  piece p    32 codes of a strip: bytes [4*b*p, 4*b*(p+1)) of the strip, read as b
             little-endian 32-bit words.
  sub-stream h in {0, 1} of a piece: 16*b bits; its bit x is bit 16*h + (x mod 16) of word
             floor(x / 16).  Code (rho, h), rho in 0..15, occupies bits [rho*b, rho*b + b)
             of sub-stream h, least significant bit first.
  K rows     token t, channel i:  tau = t // 16, tt = t % 16,
             piece = tt % 8, rho = 2*tau + tt // 8, h = i % 2.
  V rows     token t, channel i:  tau = t // 16, tt = t % 16,
             piece = 4*(i % 2) + (tt // 2) % 4, rho = 2*tau + tt // 8, h = tt % 2.
  tail       tokens past the end of a sequence are zero bits.
  regions    every head's region starts at a 256-byte aligned offset, heads in index order;
             a region holds n_slots rows; row slot k is at region + k*16*r*b.  Contiguous
             caches use slot = seq*rows_per_seq + row; paged caches (256-token pages) use
             slot = 2*page + (row % 2) with page = page_table[seq][row // 2].
"""
from __future__ import annotations

import numpy as np

TOKENS_PER_ROW = 128
SIDE_K, SIDE_V = 0, 1


def row_bytes(r: int, b: int) -> int:
    return 16 * r * b


def piece_and_slot(side: int, t, i):
    """(piece, rho, h) of code (t, i) inside its strip, for K (side 0) or V (side 1) rows."""
    t = np.asarray(t)
    i = np.asarray(i)
    tau = t // 16
    tt = t % 16
    rho = 2 * tau + tt // 8
    if side == SIDE_K:
        piece = tt % 8
        h = i % 2
    else:
        piece = 4 * (i % 2) + (tt // 2) % 4
        h = tt % 2
    return piece, rho, h


def bit_positions(side: int, r: int, b: int) -> np.ndarray:
    """Row bit index of code bit k of (token t, channel i): array [128, r, b]."""
    t = np.arange(TOKENS_PER_ROW)[:, None, None]
    i = np.arange(r)[None, :, None]
    k = np.arange(b)[None, None, :]
    piece, rho, h = piece_and_slot(side, t, i)
    s = i // 2
    x = rho * b + k
    return 8 * (32 * b * s + 4 * b * piece) + 32 * (x // 16) + 16 * h + (x % 16)


def pack_row(codes, side: int, b: int) -> np.ndarray:
    """codes [128, r] (ints in [0, 2^b)) -> one row of 16*r*b bytes."""
    codes = np.asarray(codes, dtype=np.int64)
    r = codes.shape[1]
    out_bits = np.zeros(TOKENS_PER_ROW * r * b, dtype=np.uint8)
    pos = bit_positions(side, r, b)
    bits = (codes[:, :, None] >> np.arange(b)[None, None, :]) & 1
    out_bits[pos.ravel()] = bits.ravel()
    return np.packbits(out_bits, bitorder="little")


def unpack_row(row, side: int, r: int, b: int) -> np.ndarray:
    """One row of 16*r*b bytes -> codes [128, r]."""
    bits = np.unpackbits(np.asarray(row, dtype=np.uint8), bitorder="little")
    pos = bit_positions(side, r, b)
    vals = bits[pos].astype(np.int64)
    return (vals << np.arange(b)[None, None, :]).sum(axis=2)


def pack_tokens(codes, side: int, b: int) -> np.ndarray:
    """codes [T, r] -> rows [ceil(T/128), 16*r*b] with zero codes after token T."""
    codes = np.asarray(codes, dtype=np.int64)
    T, r = codes.shape
    n_rows = -(-T // TOKENS_PER_ROW)
    padded = np.zeros((n_rows * TOKENS_PER_ROW, r), dtype=np.int64)
    padded[:T] = codes
    return np.stack([pack_row(padded[k * 128:(k + 1) * 128], side, b) for k in range(n_rows)]) \
        if n_rows else np.zeros((0, row_bytes(r, b)), dtype=np.uint8)


def unpack_tokens(rows, side: int, r: int, b: int, T: int) -> np.ndarray:
    rows = np.asarray(rows, dtype=np.uint8)
    if T == 0:
        return np.zeros((0, r), dtype=np.int64)
    codes = np.concatenate([unpack_row(rows[k], side, r, b) for k in range(rows.shape[0])])
    return codes[:T]


def plan_regions(r, b, n_slots) -> tuple[np.ndarray, int]:
    """Byte offset of each head's region (256-aligned, heads in index order) and the total
    cache size.  n_slots is the number of code rows each region holds."""
    offs = np.zeros(len(r), dtype=np.int64)
    pos = 0
    for h in range(len(r)):
        offs[h] = pos
        pos += int(n_slots) * row_bytes(int(r[h]), int(b[h]))
        pos = (pos + 255) // 256 * 256
    return offs, pos


def row_address(off: int, r: int, b: int, seq: int, row: int, rows_per_seq: int, page_table=None) -> int:
    """Byte address of (seq, row) inside a head region (contiguous or paged)."""
    if page_table is None:
        slot = seq * rows_per_seq + row
    else:
        slot = 2 * int(page_table[seq][row // 2]) + row % 2
    return off + slot * row_bytes(r, b)
