"""Seeded synthetic tensors of the CNN-training sample (one 3x3, stride-2
convolution layer): input x [N, H, W, C], filter w [K, 3, 3, C] and upstream
gradient dy [N, H/2, W/2, K], channels-last bf16 bits.  Data synthesis only:
the counter-based generator of the decoder weights with tags of their own;
none of the convolution's arithmetic lives here."""
from __future__ import annotations

import math
from dataclasses import dataclass

import numpy as np

from . import _load

CONV_X_TAG, CONV_W_TAG, CONV_DY_TAG = 0x300001, 0x300002, 0x300003


@dataclass(frozen=True)
class ConvShape:
    n: int
    c: int
    h: int
    w: int
    k: int
    seed: int = 0

    @property
    def p(self) -> int:
        return self.h // 2

    @property
    def q(self) -> int:
        return self.w // 2

    def flops(self) -> float:
        """Algorithmic FLOPs of one of the three products (forward, data or filter
        gradient): 2 N P Q K C 9."""
        return 2.0 * self.n * self.p * self.q * self.k * self.c * 9


# the paper's sample: 4 x 1024 x 224 x 224 input, 3x3 filter, stride 2 (Sec. 5.4)
CNN_SAMPLE = ConvShape(n=4, c=1024, h=224, w=224, k=1024)


def _normal_bf16(seed: int, tag: int, std: float, shape) -> np.ndarray:
    out = np.empty(int(np.prod(shape)), np.uint16)
    _load().wicigen_normal_bf16(seed, tag, std, 0, out.size, out.ctypes.data)
    return out.reshape(shape)


def make_conv_inputs(s: ConvShape):
    """(x, w, dy) as bf16 bits: x and dy ~ N(0, 1); w ~ N(0, 1 / (9 C)) so that y ~ N(0, 1)."""
    x = _normal_bf16(s.seed, CONV_X_TAG, 1.0, (s.n, s.h, s.w, s.c))
    w = _normal_bf16(s.seed, CONV_W_TAG, 1.0 / math.sqrt(9.0 * s.c), (s.k, 3, 3, s.c))
    dy = _normal_bf16(s.seed, CONV_DY_TAG, 1.0, (s.n, s.p, s.q, s.k))
    return x, w, dy
