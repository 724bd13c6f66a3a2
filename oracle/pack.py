"""Oracle, part 3: the packed 2-bit code format (plain CPU).

TEST INFRASTRUCTURE. Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline leg may
import this package; the product library never does, and shares no code with it.

The paper stores the quantized frame coefficients at 2 bits each with a per-row scale and bias
(Appendix K) and fixes no bit layout.  The layout below is the one the library header declares
for fq_pack, written out here from that definition:
  * rows are grouped in tiles of 128, columns in blocks of 64; n_out and n_in are padded up to
    those multiples with code 0;
  * the 64 codes of one (row, column block) are 4 consecutive uint32 words, and the words of a
    (row tile, column block) pair are contiguous: word index
        ((row // 128) * KB + col // 64) * 512 + (row % 128) * 4 + (col % 64) // 16,
    with KB = ceil(n_in / 64);
  * inside a word, column c = col % 16 occupies bits [2 (c // 2) + 16 (c % 2), +2).
"""
from __future__ import annotations

import numpy as np

ROW_TILE = 128
COL_BLOCK = 64


def padded(n_out: int, n_in: int) -> tuple:
    return (-(-n_out // ROW_TILE) * ROW_TILE, -(-n_in // COL_BLOCK) * COL_BLOCK)


def packed_words(n_out: int, n_in: int) -> int:
    po, pi = padded(n_out, n_in)
    return po * pi // 16


def word_index(row: int, col: int, n_in: int) -> int:
    KB = -(-n_in // COL_BLOCK)
    return (((row // ROW_TILE) * KB + col // COL_BLOCK) * (ROW_TILE * 4)
            + (row % ROW_TILE) * 4 + (col % COL_BLOCK) // 16)


def bit_offset(col: int) -> int:
    c = col % 16
    return 2 * (c // 2) + 16 * (c % 2)


def pack(codes: np.ndarray) -> np.ndarray:
    """uint8 codes (n_out x n_in, values 0..3) -> uint32 words in the layout above."""
    n_out, n_in = codes.shape
    if codes.size and int(codes.max()) > 3:
        raise ValueError("codes must be in [0, 3]")
    po, pi = padded(n_out, n_in)
    full = np.zeros((po, pi), dtype=np.uint32)
    full[:n_out, :n_in] = codes
    # (tile, r, kb, w, c) -> (tile, kb, r, w) words
    t = full.reshape(po // ROW_TILE, ROW_TILE, pi // COL_BLOCK, 4, 16)
    shifts = np.array([bit_offset(c) for c in range(16)], dtype=np.uint32)
    words = np.bitwise_or.reduce(t << shifts, axis=-1)           # (tile, r, kb, w)
    return np.ascontiguousarray(words.transpose(0, 2, 1, 3)).reshape(-1)


def unpack(words: np.ndarray, n_out: int, n_in: int) -> np.ndarray:
    """Inverse of pack (padding dropped)."""
    po, pi = padded(n_out, n_in)
    w = words.reshape(po // ROW_TILE, pi // COL_BLOCK, ROW_TILE, 4).transpose(0, 2, 1, 3)
    shifts = np.array([bit_offset(c) for c in range(16)], dtype=np.uint32)
    codes = (w[..., None] >> shifts) & 3                           # (tile, r, kb, w, c)
    return codes.reshape(po, pi)[:n_out, :n_in].astype(np.uint8)
