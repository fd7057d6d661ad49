"""ctypes binding of include/wici.h (argument marshalling only).

Every entry point of the C ABI is exposed under the same name.  `WiciModel` is
a small convenience wrapper: it allocates the three device buffers with torch
(plumbing: device memory and the stream), creates a context and forwards calls.
There is no fallback: when libwici.so or a GPU is missing these calls raise.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libwici.so")

WICI_OK, WICI_E_ARG, WICI_E_STATE, WICI_E_CAPACITY, WICI_E_CUDA, WICI_E_TIMEOUT = 0, -1, -2, -3, -4, -5
STATUS_NAMES = {0: "WICI_OK", -1: "WICI_E_ARG", -2: "WICI_E_STATE", -3: "WICI_E_CAPACITY",
                -4: "WICI_E_CUDA", -5: "WICI_E_TIMEOUT"}

# the entry points declared in include/wici.h
EXPORTS = ("wici_get_sizes", "wici_create", "wici_load_weights", "wici_load_weights_q8", "wici_prefill",
           "wici_decode_step",
           "wici_decode", "wici_reset", "wici_set_page_table", "wici_kv_len", "wici_last_error",
           "wici_profile_decode", "wici_check_bounded_wait", "wici_destroy", "wici_lm_head_argmax_noalloc",
           "wici_conv_workspace_bytes", "wici_conv_forward", "wici_conv_backward_data", "wici_conv_backward_filter",
           "wici_conv_status", "wici_profile_prefill")


class wici_config(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int32), ("hidden", ctypes.c_int32), ("n_q_heads", ctypes.c_int32),
                ("n_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32), ("ffn_dim", ctypes.c_int32),
                ("vocab", ctypes.c_int32), ("max_tokens", ctypes.c_int32), ("max_chunk", ctypes.c_int32),
                ("page_tokens", ctypes.c_int32), ("rms_eps", ctypes.c_float), ("rope_theta", ctypes.c_double),
                ("tied_embeddings", ctypes.c_int32), ("qkv_bias", ctypes.c_int32),
                ("weight_format", ctypes.c_int32), ("qk_norm", ctypes.c_int32), ("max_sms", ctypes.c_int32)]

WICI_WEIGHTS_BF16, WICI_WEIGHTS_Q8 = 0, 1


class wici_sizes(ctypes.Structure):
    _fields_ = [("weight_bytes", ctypes.c_size_t), ("kv_bytes", ctypes.c_size_t),
                ("workspace_bytes", ctypes.c_size_t)]


class wici_tensor(ctypes.Structure):
    _fields_ = [("name", ctypes.c_char_p), ("data", ctypes.c_void_p), ("rows", ctypes.c_int64),
                ("cols", ctypes.c_int64), ("on_device", ctypes.c_int32)]


class wici_q8_tensor(ctypes.Structure):
    _fields_ = [("name", ctypes.c_char_p), ("codes", ctypes.c_void_p), ("scales", ctypes.c_void_p),
                ("rows", ctypes.c_int64), ("cols", ctypes.c_int64), ("on_device", ctypes.c_int32)]


_lib = None


def lib():
    """Load libwici.so (built by __graft_entry__.build()); raises if it is missing."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError(f"{LIB_PATH} is missing: build it first (python -c 'import __graft_entry__ as g; "
                              "g.build()')")
        L = ctypes.CDLL(LIB_PATH)
        P, i32, i64, vp = ctypes.POINTER, ctypes.c_int32, ctypes.c_int64, ctypes.c_void_p
        L.wici_get_sizes.argtypes = [P(wici_config), P(wici_sizes)]
        L.wici_create.argtypes = [P(wici_config), vp, vp, vp, vp, P(vp)]
        L.wici_load_weights.argtypes = [vp, P(wici_tensor), i32]
        L.wici_load_weights_q8.argtypes = [vp, P(wici_q8_tensor), i32]
        L.wici_prefill.argtypes = [vp, P(i32), i32, P(ctypes.c_float), P(i32)]
        L.wici_decode_step.argtypes = [vp, i32, P(ctypes.c_float), P(i32)]
        L.wici_decode.argtypes = [vp, i32, i32, P(i32)]
        L.wici_reset.argtypes = [vp]
        L.wici_set_page_table.argtypes = [vp, P(i32), i32]
        L.wici_kv_len.argtypes = [vp]
        L.wici_kv_len.restype = i32
        L.wici_last_error.argtypes = [vp]
        L.wici_last_error.restype = ctypes.c_char_p
        L.wici_profile_decode.argtypes = [vp, i32, P(ctypes.c_char_p), P(i32), P(ctypes.c_double), i32, P(i32)]
        L.wici_check_bounded_wait.argtypes = [vp, i64]
        L.wici_profile_prefill.argtypes = [vp, P(i32), i32, P(ctypes.c_char_p), P(i32), P(ctypes.c_double), i32,
                                           P(i32)]
        L.wici_destroy.argtypes = [vp]
        L.wici_destroy.restype = None
        L.wici_lm_head_argmax_noalloc.argtypes = [vp, vp, vp, vp, i32, i32, ctypes.c_float, vp, vp]
        cs = P(wici_conv_shape)
        L.wici_conv_workspace_bytes.argtypes = [cs, P(ctypes.c_size_t)]
        L.wici_conv_forward.argtypes = [vp, cs, vp, vp, vp, vp]
        L.wici_conv_backward_data.argtypes = [vp, cs, vp, vp, vp, vp]
        L.wici_conv_backward_filter.argtypes = [vp, cs, vp, vp, vp, vp]
        L.wici_conv_status.argtypes = [vp, vp]
        for name in ("wici_get_sizes", "wici_create", "wici_load_weights", "wici_load_weights_q8", "wici_prefill",
                     "wici_decode_step",
                     "wici_decode", "wici_reset", "wici_set_page_table", "wici_profile_decode",
                     "wici_check_bounded_wait", "wici_lm_head_argmax_noalloc", "wici_conv_workspace_bytes",
                     "wici_conv_forward", "wici_conv_backward_data", "wici_conv_backward_filter",
                     "wici_conv_status", "wici_profile_prefill"):
            getattr(L, name).restype = ctypes.c_int
        _lib = L
    return _lib


class WiciError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {msg}")
        self.status = status


def _check(rc, ctx=None):
    if rc != WICI_OK:
        raise WiciError(rc, (lib().wici_last_error(ctx) or b"").decode())
    return rc


def make_config(cfg, max_tokens: int, max_chunk: int | None = None, q8: bool = False,
                max_sms: int = 0) -> wici_config:
    """wici_config from a gen.ModelConfig-like object (Llama / Qwen blocks; the
    library has no kernels for another block, such as Falcon's)."""
    if getattr(cfg, "block", "llama") != "llama":
        raise ValueError(f"{cfg.name}: the {cfg.block} block has no CUDA path in this library")
    return wici_config(cfg.n_layers, cfg.hidden, cfg.n_q_heads, cfg.n_kv_heads, cfg.head_dim, cfg.ffn_dim,
                       cfg.vocab, max_tokens, min(max_chunk or cfg.max_chunk, max_tokens), 16, cfg.rms_eps,
                       cfg.rope_theta, int(cfg.tied_embeddings), int(cfg.qkv_bias),
                       WICI_WEIGHTS_Q8 if q8 else WICI_WEIGHTS_BF16, int(getattr(cfg, "qk_norm", False)),
                       max_sms)


# ---------------------------------------------------------------- thin wrappers
def wici_get_sizes(cfg: wici_config) -> wici_sizes:
    out = wici_sizes()
    _check(lib().wici_get_sizes(ctypes.byref(cfg), ctypes.byref(out)))
    return out


def wici_create(cfg: wici_config, stream: int, weight_dev: int, kv_dev: int, ws_dev: int):
    ctx = ctypes.c_void_p()
    _check(lib().wici_create(ctypes.byref(cfg), stream, weight_dev, kv_dev, ws_dev, ctypes.byref(ctx)))
    return ctx


def wici_load_weights(ctx, tensors) -> None:
    """tensors: iterable of (name, array-or-(ptr, on_device), rows, cols)."""
    keep, arr = [], []
    for name, data, rows, cols in tensors:
        if isinstance(data, np.ndarray):
            assert data.dtype == np.uint16 and data.flags.c_contiguous
            keep.append(data)
            ptr, dev = data.ctypes.data, 0
        else:
            ptr, dev = data
        arr.append(wici_tensor(name.encode(), ptr, rows, cols, dev))
    tarr = (wici_tensor * len(arr))(*arr)
    _check(lib().wici_load_weights(ctx, tarr, len(arr)), ctx)


def wici_load_weights_q8(ctx, tensors) -> None:
    """tensors: iterable of (name, codes int8 [rows, cols], scales fp16 bits uint16 [rows, cols/32]) host arrays."""
    keep, arr = [], []
    for name, codes, scales in tensors:
        codes = np.ascontiguousarray(codes, np.int8)
        scales = np.ascontiguousarray(scales, np.uint16)
        keep += [codes, scales]
        arr.append(wici_q8_tensor(name.encode(), codes.ctypes.data, scales.ctypes.data, codes.shape[0],
                                  codes.shape[1], 0))
    tarr = (wici_q8_tensor * len(arr))(*arr)
    _check(lib().wici_load_weights_q8(ctx, tarr, len(arr)), ctx)


def _i32p(a):
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_int32))


def wici_prefill(ctx, tokens: np.ndarray, logits_out: np.ndarray | None = None) -> int:
    tok = np.ascontiguousarray(tokens, np.int32)
    out = np.zeros(1, np.int32)
    lp = None if logits_out is None else logits_out.ctypes.data_as(ctypes.POINTER(ctypes.c_float))
    _check(lib().wici_prefill(ctx, _i32p(tok), len(tok), lp, _i32p(out)), ctx)
    return int(out[0])


def wici_decode_step(ctx, token_in: int = -1, logits_out: np.ndarray | None = None) -> int:
    out = np.zeros(1, np.int32)
    lp = None if logits_out is None else logits_out.ctypes.data_as(ctypes.POINTER(ctypes.c_float))
    _check(lib().wici_decode_step(ctx, token_in, lp, _i32p(out)), ctx)
    return int(out[0])


def wici_decode(ctx, n_steps: int, token_in: int = -1, tokens_out: np.ndarray | None = None) -> None:
    tp = None if tokens_out is None else _i32p(tokens_out)
    _check(lib().wici_decode(ctx, n_steps, token_in, tp), ctx)


def wici_reset(ctx) -> None:
    _check(lib().wici_reset(ctx), ctx)


def wici_set_page_table(ctx, pages: np.ndarray) -> None:
    p = np.ascontiguousarray(pages, np.int32)
    _check(lib().wici_set_page_table(ctx, _i32p(p), len(p)), ctx)


def wici_kv_len(ctx) -> int:
    return int(lib().wici_kv_len(ctx))


def wici_last_error(ctx=None) -> str:
    return (lib().wici_last_error(ctx) or b"").decode()


def wici_profile_decode(ctx, n_steps: int, cap: int = 16) -> dict:
    names = (ctypes.c_char_p * cap)()
    launches = (ctypes.c_int32 * cap)()
    ms = (ctypes.c_double * cap)()
    n = ctypes.c_int32()
    _check(lib().wici_profile_decode(ctx, n_steps, names, launches, ms, cap, ctypes.byref(n)), ctx)
    return {names[i].decode(): (int(launches[i]), float(ms[i])) for i in range(n.value)}


def wici_profile_prefill(ctx, tokens: np.ndarray, cap: int = 16) -> dict:
    tok = np.ascontiguousarray(tokens, np.int32)
    names = (ctypes.c_char_p * cap)()
    launches = (ctypes.c_int32 * cap)()
    ms = (ctypes.c_double * cap)()
    n = ctypes.c_int32()
    _check(lib().wici_profile_prefill(ctx, _i32p(tok), len(tok), names, launches, ms, cap, ctypes.byref(n)), ctx)
    return {names[i].decode(): (int(launches[i]), float(ms[i])) for i in range(n.value)}


def wici_check_bounded_wait(stream: int, limit_ns: int) -> int:
    return int(lib().wici_check_bounded_wait(stream, limit_ns))


def wici_destroy(ctx) -> None:
    lib().wici_destroy(ctx)


def wici_lm_head_argmax_noalloc(stream: int, lm_head_dev: int, norm_gain_dev: int, x_dev: int, hidden: int,
                                vocab: int, rms_eps: float, logits_dev: int, token_dev: int) -> None:
    """Final RMSNorm + LM head + argmax on device pointers, without any device
    allocation (for callers whose device memory is owned elsewhere); the
    scratch is a fixed array inside the library.  Enqueued on `stream`."""
    _check(lib().wici_lm_head_argmax_noalloc(stream, lm_head_dev, norm_gain_dev, x_dev, hidden, vocab, rms_eps,
                                              logits_dev, token_dev))


# ------------------------------------------------------- CNN-training sample
class wici_conv_shape(ctypes.Structure):
    _fields_ = [("n", ctypes.c_int32), ("c", ctypes.c_int32), ("h", ctypes.c_int32), ("w", ctypes.c_int32),
                ("k", ctypes.c_int32)]


def wici_conv_workspace_bytes(shape: wici_conv_shape) -> int:
    out = ctypes.c_size_t()
    _check(lib().wici_conv_workspace_bytes(ctypes.byref(shape), ctypes.byref(out)))
    return int(out.value)


def wici_conv_forward(stream: int, shape: wici_conv_shape, x: int, w: int, y: int, ws: int) -> None:
    _check(lib().wici_conv_forward(stream, ctypes.byref(shape), x, w, y, ws))


def wici_conv_backward_data(stream: int, shape: wici_conv_shape, dy: int, w: int, dx: int, ws: int) -> None:
    _check(lib().wici_conv_backward_data(stream, ctypes.byref(shape), dy, w, dx, ws))


def wici_conv_backward_filter(stream: int, shape: wici_conv_shape, x: int, dy: int, dw: int, ws: int) -> None:
    _check(lib().wici_conv_backward_filter(stream, ctypes.byref(shape), x, dy, dw, ws))


def wici_conv_status(stream: int, ws: int) -> None:
    _check(lib().wici_conv_status(stream, ws))


# ------------------------------------------------------------- convenience
class WiciModel:
    """Owns torch-allocated device buffers and one context on the current device."""

    def __init__(self, cfg, max_tokens: int | None = None, max_chunk: int | None = None, stream=None,
                 q8: bool = False, max_sms: int = 0):
        import torch
        if not torch.cuda.is_available():
            raise RuntimeError("WiciModel needs a CUDA device")
        self.cfg = cfg
        self.max_tokens = max_tokens or cfg.total_tokens
        self.ccfg = make_config(cfg, self.max_tokens, max_chunk, q8, max_sms)
        sizes = wici_get_sizes(self.ccfg)
        self.sizes = sizes

        def alloc(n):
            return torch.empty(max(n, 256) + 256, dtype=torch.uint8, device="cuda")

        self._w, self._kv, self._ws = alloc(sizes.weight_bytes), alloc(sizes.kv_bytes), \
            alloc(sizes.workspace_bytes)
        self.stream = stream or torch.cuda.current_stream()

        def aligned(t):
            return (t.data_ptr() + 255) // 256 * 256

        self.ctx = wici_create(self.ccfg, self.stream.cuda_stream, aligned(self._w), aligned(self._kv),
                               aligned(self._ws))

    def load(self, weights: dict, q8_weights: dict | None = None) -> "WiciModel":
        """bf16 tensors {name: uint16 [rows, cols]}; with the 8-bit format, the
        per-layer matrices come as q8_weights {name: (codes, scales)} and the
        bf16 dict's entries of the same names are skipped."""
        q8_weights = q8_weights or {}
        items = []
        for name, arr in weights.items():
            if name in q8_weights:
                continue
            r, c = arr.shape
            items.append((name, arr, r, c))
        wici_load_weights(self.ctx, items)
        if q8_weights:
            wici_load_weights_q8(self.ctx, [(n, c, s) for n, (c, s) in q8_weights.items()])
        return self

    def prefill(self, tokens, logits: bool = False):
        out = np.empty(self.cfg.vocab, np.float32) if logits else None
        tok = wici_prefill(self.ctx, tokens, out)
        return (out, tok) if logits else tok

    def decode_step(self, token_in: int = -1, logits: bool = False):
        out = np.empty(self.cfg.vocab, np.float32) if logits else None
        tok = wici_decode_step(self.ctx, token_in, out)
        return (out, tok) if logits else tok

    def decode(self, n_steps: int, token_in: int = -1) -> np.ndarray:
        out = np.empty(n_steps, np.int32)
        wici_decode(self.ctx, n_steps, token_in, out)
        return out

    def reset(self):
        wici_reset(self.ctx)

    @property
    def kv_len(self) -> int:
        return wici_kv_len(self.ctx)

    def close(self):
        if getattr(self, "ctx", None) is not None:
            wici_destroy(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
