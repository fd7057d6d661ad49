"""Seeded synthetic weights in an 8-bit block format (codes + per-block scales).

Format: every row of a matrix [rows, cols] is cut into blocks of Q8_BLOCK = 32
consecutive input columns; block b of row r holds 32 int8 codes in
[-127, 127] and one fp16 scale d[r, b].  The weight the format stands for is
d[r, b] * code[r, c] for c in block b (a GGUF-style 8-bit block format; the
paper's models are GGUF files).

This module only synthesises codes and scales from the same counter-based
generator as the bf16 weights (with tags of their own); it contains none of
the arithmetic that consumes them.  Codes are a normal draw scaled to the
code range, scales vary per block by up to +-50% around 0.02 * 4 / 127, so the
dequantised weights have about the bf16 models' ~N(0, 0.02) statistics.
"""
from __future__ import annotations

import numpy as np

from . import normal_f64
from .configs import ModelConfig, tensor_specs

Q8_BLOCK = 32
Q8_CODE_TAG = 0x100000    # + the tensor's canonical tag: the codes' stream
Q8_SCALE_TAG = 0x200000   # + the tensor's canonical tag: the scales' stream
Q8_MATRICES = ("wq", "wk", "wv", "wo", "wg", "wu", "wd", "w_up", "w_down")   # per-layer matrices in the format


def q8_names(cfg: ModelConfig) -> list:
    """Names of the tensors stored in the 8-bit format: every layer's matrices
    whose input width is a whole number of blocks (the others stay bf16)."""
    return [nm for nm, (_, cols), _ in tensor_specs(cfg)
            if nm.split(".")[-1] in Q8_MATRICES and cols % Q8_BLOCK == 0]


def make_q8_tensor(cfg: ModelConfig, name: str):
    """(codes int8 [rows, cols], scales as fp16 bits uint16 [rows, cols / 32])."""
    specs = tensor_specs(cfg)
    for tag, (nm, (rows, cols), _) in enumerate(specs):
        if nm == name:
            break
    else:
        raise KeyError(name)
    if name not in q8_names(cfg):
        raise ValueError(f"{name} is not stored in the 8-bit format")
    if cols % Q8_BLOCK:
        raise ValueError(f"{name}: {cols} columns are not a multiple of {Q8_BLOCK}")
    s = normal_f64(cfg.weight_seed, Q8_CODE_TAG + tag, rows * cols)
    codes = np.clip(np.rint(s * (127.0 / 4.0)), -127, 127).astype(np.int8).reshape(rows, cols)
    t = normal_f64(cfg.weight_seed, Q8_SCALE_TAG + tag, rows * (cols // Q8_BLOCK))
    scale = cfg.weight_std * (4.0 / 127.0) * (1.0 + 0.25 * np.clip(t, -2.0, 2.0))
    scales = scale.astype(np.float16).view(np.uint16).reshape(rows, cols // Q8_BLOCK)
    return codes, scales


def make_q8_weights(cfg: ModelConfig) -> dict:
    """{name: (codes, scales)} for every tensor stored in the 8-bit format."""
    return {nm: make_q8_tensor(cfg, nm) for nm in q8_names(cfg)}
