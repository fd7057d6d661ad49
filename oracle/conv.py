"""Oracle of the CNN-training sample: one 3x3, stride-2 convolution layer,
forward and backward (test infrastructure only; never imported by the product
path).

The paper's second evaluated application (Sec. 5.4, "Multiple applications")
is NVIDIA's CNN-training sample with an input of 4 x 1024 x 224 x 224, a 3x3
filter and a stride of 2.  It gives nothing else, so these are readings: zero
padding of 1 on each side (a 224 x 224 input gives a 112 x 112 output), as many
output channels as input channels, no bias, and a training step of the layer
is its forward pass plus the two gradients of backpropagation for an upstream
gradient dy.  Layout is channels-last: x [N, H, W, C], w [K, 3, 3, C],
y and dy [N, P, Q, K] with P = H/2, Q = W/2 (H and W even).

Each function is the plain definition, written per filter tap with array
slices, in fp64:
    y[n,p,q,k]  = sum_{r,s,c} x[n, 2p+r-1, 2q+s-1, c] w[k,r,s,c]
    dx[n,h,v,c] = sum_{p,q,r,s,k : 2p+r-1 = h, 2q+s-1 = v} dy[n,p,q,k] w[k,r,s,c]
    dw[k,r,s,c] = sum_{n,p,q} dy[n,p,q,k] x[n, 2p+r-1, 2q+s-1, c]
with x taken as zero outside [0, H) x [0, W).
"""
from __future__ import annotations

import numpy as np

STRIDE = 2
TAPS = 3


def out_hw(h: int, w: int):
    return h // 2, w // 2


def _padded(x):
    return np.pad(np.asarray(x, np.float64), ((0, 0), (1, 1), (1, 1), (0, 0)))


def conv_forward(x: np.ndarray, w: np.ndarray) -> np.ndarray:
    """y [N, P, Q, K] from x [N, H, W, C] and w [K, 3, 3, C]."""
    N, H, W, C = x.shape
    P, Q = out_hw(H, W)
    xp = _padded(x)
    w = np.asarray(w, np.float64)
    y = np.zeros((N, P, Q, w.shape[0]), np.float64)
    for r in range(TAPS):
        for s in range(TAPS):
            patch = xp[:, r:r + STRIDE * P:STRIDE, s:s + STRIDE * Q:STRIDE, :]      # x[n, 2p+r-1, 2q+s-1, :]
            y += patch @ w[:, r, s, :].T
    return y


def conv_backward_data(dy: np.ndarray, w: np.ndarray, H: int, W: int) -> np.ndarray:
    """dx [N, H, W, C]: every tap scatters dy[n,p,q,:] w[:,r,s,:] back to x[n, 2p+r-1, 2q+s-1]."""
    N, P, Q, K = dy.shape
    w = np.asarray(w, np.float64)
    dy = np.asarray(dy, np.float64)
    dxp = np.zeros((N, H + 2, W + 2, w.shape[3]), np.float64)
    for r in range(TAPS):
        for s in range(TAPS):
            dxp[:, r:r + STRIDE * P:STRIDE, s:s + STRIDE * Q:STRIDE, :] += dy @ w[:, r, s, :]
    return dxp[:, 1:H + 1, 1:W + 1, :]


def conv_backward_filter(x: np.ndarray, dy: np.ndarray) -> np.ndarray:
    """dw [K, 3, 3, C] = sum over n, p, q of dy[n,p,q,k] x[n, 2p+r-1, 2q+s-1, c]."""
    N, H, W, C = x.shape
    _, P, Q, K = dy.shape
    xp = _padded(x)
    dy = np.asarray(dy, np.float64).reshape(-1, K)
    dw = np.zeros((K, TAPS, TAPS, C), np.float64)
    for r in range(TAPS):
        for s in range(TAPS):
            patch = xp[:, r:r + STRIDE * P:STRIDE, s:s + STRIDE * Q:STRIDE, :].reshape(-1, C)
            dw[:, r, s, :] = dy.T @ patch
    return dw


def abs_sum_bound(fn, *args) -> np.ndarray:
    """The same map applied to |operands|: the sum of |products| behind every
    output, which bounds its accumulated rounding error."""
    return fn(*[np.abs(np.asarray(a, np.float64)) if isinstance(a, np.ndarray) else a for a in args])


# ---- single outputs, for sampled comparisons at sizes the whole arrays would
# take too long for; each is the same definition restricted to one output

def conv_forward_at(x: np.ndarray, w: np.ndarray, n: int, p: int, q: int) -> np.ndarray:
    """y[n, p, q, :]."""
    _, H, W, _ = x.shape
    w = np.asarray(w, np.float64)
    out = np.zeros(w.shape[0], np.float64)
    for r in range(TAPS):
        for s in range(TAPS):
            h, v = STRIDE * p + r - 1, STRIDE * q + s - 1
            if 0 <= h < H and 0 <= v < W:
                out += w[:, r, s, :] @ np.asarray(x[n, h, v, :], np.float64)
    return out


def conv_backward_data_at(dy: np.ndarray, w: np.ndarray, n: int, h: int, v: int) -> np.ndarray:
    """dx[n, h, v, :]."""
    _, P, Q, _ = dy.shape
    w = np.asarray(w, np.float64)
    out = np.zeros(w.shape[3], np.float64)
    for r in range(TAPS):
        for s in range(TAPS):
            if (h + 1 - r) % STRIDE or (v + 1 - s) % STRIDE:
                continue
            p, q = (h + 1 - r) // STRIDE, (v + 1 - s) // STRIDE
            if 0 <= p < P and 0 <= q < Q:
                out += np.asarray(dy[n, p, q, :], np.float64) @ w[:, r, s, :]
    return out


def conv_backward_filter_at(x: np.ndarray, dy: np.ndarray, k: int) -> np.ndarray:
    """dw[k, :, :, :]."""
    N, H, W, C = x.shape
    _, P, Q, _ = dy.shape
    xp = _padded(x)
    g = np.asarray(dy[..., k], np.float64).reshape(-1)
    out = np.zeros((TAPS, TAPS, C), np.float64)
    for r in range(TAPS):
        for s in range(TAPS):
            out[r, s] = g @ xp[:, r:r + STRIDE * P:STRIDE, s:s + STRIDE * Q:STRIDE, :].reshape(-1, C)
    return out
