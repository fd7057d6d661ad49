"""Seeded synthetic inputs (weights and prompts) shared by the oracle and the
CUDA path.  The generator is defined in `wicigen.c`; this module only builds and
calls it.  It holds none of the forward pass's arithmetic."""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

from .configs import (CONFIGS, FALCON_40B, FALCON_TINY, LLAMA_1B, LLAMA_8B, LLAMA_8B_AGENTIC, QWEN3_8B, QWEN_14B, TINY,
                      ModelConfig, decode_bytes_per_token, prefill_flops, tensor_specs)

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "wicigen.c")
_LIB = os.path.join(_HERE, "libwicigen.so")
_lock = threading.Lock()
_lib = None

PROMPT_TAG = 0x7FFFFFFF
GAIN_STD = 0.25   # per-head q/k norm gains: 1 + 0.25 N(0, 1), rounded to bf16


def build(force: bool = False) -> str:
    """Compile wicigen.c with the host gcc (OpenMP, no fused multiply-add)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".{os.getpid()}.tmp"
        subprocess.check_call(["gcc", "-O2", "-fopenmp", "-ffp-contract=off", "-fPIC", "-shared",
                               _SRC, "-o", tmp])
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            u64, dbl, p = ctypes.c_uint64, ctypes.c_double, ctypes.c_void_p
            lib.wicigen_draw.argtypes = [u64, u64]
            lib.wicigen_draw.restype = u64
            lib.wicigen_stream.argtypes = [u64, u64]
            lib.wicigen_stream.restype = u64
            lib.wicigen_normal_bf16.argtypes = [u64, u64, dbl, u64, u64, p]
            lib.wicigen_normal_f64.argtypes = [u64, u64, u64, u64, p]
            lib.wicigen_tokens.argtypes = [u64, u64, u64, u64, p]
            lib.wicigen_fill_bf16.argtypes = [ctypes.c_float, u64, p]
            lib.wicigen_gain_bf16.argtypes = [u64, u64, dbl, u64, u64, p]
            _lib = lib
    return _lib


def draw(key: int, i: int) -> int:
    return int(_load().wicigen_draw(key, i))


def stream(seed: int, tag: int) -> int:
    return int(_load().wicigen_stream(seed, tag))


def normal_f64(seed: int, tag: int, n: int, e0: int = 0) -> np.ndarray:
    out = np.empty(n, np.float64)
    _load().wicigen_normal_f64(seed, tag, e0, n, out.ctypes.data)
    return out


def make_tensor(cfg: ModelConfig, name: str, out: np.ndarray | None = None) -> np.ndarray:
    """bf16 bits (np.uint16, shape (rows, cols)) of one named weight tensor."""
    specs = tensor_specs(cfg)
    for tag, (nm, shape, kind) in enumerate(specs):
        if nm == name:
            break
    else:
        raise KeyError(name)
    if out is None:
        out = np.empty(shape, np.uint16)
    assert out.shape == shape and out.dtype == np.uint16 and out.flags.c_contiguous
    lib = _load()
    if kind == "ones":
        lib.wicigen_fill_bf16(1.0, out.size, out.ctypes.data)
    elif kind == "gain":
        lib.wicigen_gain_bf16(cfg.weight_seed, tag, GAIN_STD, 0, out.size, out.ctypes.data)
    else:
        lib.wicigen_normal_bf16(cfg.weight_seed, tag, cfg.weight_std, 0, out.size, out.ctypes.data)
    return out


def make_weights(cfg: ModelConfig, names=None) -> dict:
    """All (or the listed) weight tensors of `cfg` as {name: uint16 array}."""
    want = None if names is None else set(names)
    return {nm: make_tensor(cfg, nm) for nm, _, _ in tensor_specs(cfg)
            if want is None or nm in want}


def make_prompt(cfg: ModelConfig, n: int, seed: int = 1) -> np.ndarray:
    """n uniform-random token ids in [0, vocab) (int32)."""
    out = np.empty(n, np.int32)
    _load().wicigen_tokens(seed, PROMPT_TAG, cfg.vocab, n, out.ctypes.data)
    return out


__all__ = ["CONFIGS", "TINY", "LLAMA_1B", "LLAMA_8B", "LLAMA_8B_AGENTIC", "QWEN_14B", "QWEN3_8B", "FALCON_TINY", "FALCON_40B",
           "ModelConfig", "tensor_specs", "decode_bytes_per_token", "prefill_flops",
           "make_tensor", "make_weights", "make_prompt", "normal_f64", "draw", "stream", "build"]
