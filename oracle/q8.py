"""Oracle of the 8-bit block weight format (test infrastructure only).

The format (a GGUF-style block format, as the paper's models are GGUF files):
row r of a [rows, cols] matrix is split into blocks of 32 consecutive input
columns; block b holds int8 codes q[r, 32b .. 32b+31] in [-127, 127] and one fp16
scale d[r, b].  The matrix it stands for is W[r, c] = d[r, c // 32] * q[r, c],
and a matrix-vector product is, by that definition,

    y[r] = sum_b d[r, b] * sum_{c in block b} q[r, c] * x[c].

Both are written out here in fp64.  A code times an fp16 scale is exact in
fp64, so the dequantised matrix carries no rounding of its own.
"""
from __future__ import annotations

import numpy as np

Q8_BLOCK = 32


def fp16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    return np.asarray(bits, np.uint16).view(np.float16).astype(np.float64)


def q8_dequantize(codes: np.ndarray, scales: np.ndarray) -> np.ndarray:
    """W[r, c] = d[r, c // 32] * q[r, c] in fp64 (exact)."""
    codes = np.asarray(codes, np.int8)
    rows, cols = codes.shape
    d = fp16_bits_to_f64(scales).reshape(rows, cols // Q8_BLOCK)
    return codes.astype(np.float64) * np.repeat(d, Q8_BLOCK, axis=1)


def q8_matvec(codes: np.ndarray, scales: np.ndarray, x: np.ndarray) -> np.ndarray:
    """y = W x block by block: the per-block code dot products, then the scales."""
    codes = np.asarray(codes, np.int8)
    rows, cols = codes.shape
    nb = cols // Q8_BLOCK
    q = codes.astype(np.float64).reshape(rows, nb, Q8_BLOCK)
    xb = np.asarray(x, np.float64).reshape(nb, Q8_BLOCK)
    block_dots = np.einsum("rbk,bk->rb", q, xb)
    return (block_dots * fp16_bits_to_f64(scales).reshape(rows, nb)).sum(axis=1)
