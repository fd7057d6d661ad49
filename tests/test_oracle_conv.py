"""Pins of the convolution oracle (oracle/conv.py), none of which re-types its
formulas: scalar brute force straight from the index definitions, PyTorch's
conv2d and autograd (fp64), the adjoint identities that tie the three maps
together, and single-tap closed forms."""
import numpy as np
import pytest
import torch
import torch.nn.functional as F

from gen import conv as gc
from oracle import conv as C

rng = np.random.default_rng(5)


def _rand(*shape):
    return rng.standard_normal(shape)


def test_forward_matches_scalar_brute_force():
    x, w = _rand(1, 6, 8, 3), _rand(2, 3, 3, 3)
    y = C.conv_forward(x, w)
    assert y.shape == (1, 3, 4, 2)
    for p in range(3):
        for q in range(4):
            for k in range(2):
                acc = 0.0
                for r in range(3):
                    for s in range(3):
                        h, v = 2 * p + r - 1, 2 * q + s - 1
                        if 0 <= h < 6 and 0 <= v < 8:
                            acc += float(np.dot(x[0, h, v], w[k, r, s]))
                assert abs(y[0, p, q, k] - acc) < 1e-12


def test_backward_data_matches_scalar_brute_force():
    dy, w = _rand(1, 3, 2, 2), _rand(2, 3, 3, 3)
    dx = C.conv_backward_data(dy, w, 6, 4)
    want = np.zeros((1, 6, 4, 3))
    for p in range(3):
        for q in range(2):
            for r in range(3):
                for s in range(3):
                    h, v = 2 * p + r - 1, 2 * q + s - 1
                    if 0 <= h < 6 and 0 <= v < 4:
                        want[0, h, v] += dy[0, p, q] @ w[:, r, s, :]
    np.testing.assert_allclose(dx, want, rtol=0, atol=1e-12)


def test_backward_filter_matches_scalar_brute_force():
    x, dy = _rand(2, 4, 6, 3), _rand(2, 2, 3, 2)
    dw = C.conv_backward_filter(x, dy)
    for k in range(2):
        for r in range(3):
            for s in range(3):
                for c in range(3):
                    acc = 0.0
                    for n in range(2):
                        for p in range(2):
                            for q in range(3):
                                h, v = 2 * p + r - 1, 2 * q + s - 1
                                if 0 <= h < 4 and 0 <= v < 6:
                                    acc += dy[n, p, q, k] * x[n, h, v, c]
                    assert abs(dw[k, r, s, c] - acc) < 1e-12


def test_all_three_match_torch_conv2d_and_autograd():
    x = torch.from_numpy(_rand(2, 10, 12, 5)).requires_grad_(True)
    w = torch.from_numpy(_rand(4, 3, 3, 5)).requires_grad_(True)
    dy = torch.from_numpy(_rand(2, 5, 6, 4))
    y = F.conv2d(x.permute(0, 3, 1, 2), w.permute(0, 3, 1, 2), stride=2, padding=1).permute(0, 2, 3, 1)
    y.backward(dy)
    np.testing.assert_allclose(C.conv_forward(x.detach().numpy(), w.detach().numpy()), y.detach().numpy(),
                               rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(C.conv_backward_data(dy.numpy(), w.detach().numpy(), 10, 12), x.grad.numpy(),
                               rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(C.conv_backward_filter(x.detach().numpy(), dy.numpy()), w.grad.numpy(),
                               rtol=1e-12, atol=1e-12)


def test_adjoint_identities():
    # <conv(x, w), dy> = <x, dgrad(dy, w)> = <w, wgrad(x, dy)>
    x, w, dy = _rand(2, 8, 6, 4), _rand(3, 3, 3, 4), _rand(2, 4, 3, 3)
    a = np.sum(C.conv_forward(x, w) * dy)
    b = np.sum(x * C.conv_backward_data(dy, w, 8, 6))
    c = np.sum(w * C.conv_backward_filter(x, dy))
    assert abs(a - b) < 1e-10 * abs(a) and abs(a - c) < 1e-10 * abs(a)


def test_centre_tap_alone_is_a_strided_matrix_product():
    x, w = _rand(1, 8, 8, 3), np.zeros((2, 3, 3, 3))
    w[:, 1, 1, :] = _rand(2, 3)
    np.testing.assert_allclose(C.conv_forward(x, w), x[:, ::2, ::2, :] @ w[:, 1, 1, :].T, rtol=0, atol=1e-12)


def test_generator_shapes_and_scale():
    s = gc.ConvShape(n=1, c=64, h=8, w=8, k=32)
    x, w, dy = gc.make_conv_inputs(s)
    assert x.shape == (1, 8, 8, 64) and w.shape == (32, 3, 3, 64) and dy.shape == (1, 4, 4, 32)
    wf = (w.astype(np.uint32) << 16).view(np.float32)
    assert abs(wf.std() * np.sqrt(9 * 64) - 1.0) < 0.1
    assert gc.CNN_SAMPLE.flops() == pytest.approx(2 * 4 * 112 * 112 * 1024 * 1024 * 9)


def test_single_output_forms_agree_with_the_whole_arrays():
    x, w, dy = _rand(2, 10, 8, 4), _rand(3, 3, 3, 4), _rand(2, 5, 4, 3)
    y, dx, dw = C.conv_forward(x, w), C.conv_backward_data(dy, w, 10, 8), C.conv_backward_filter(x, dy)
    for n, p, q in ((0, 0, 0), (1, 4, 3), (1, 2, 1)):
        np.testing.assert_allclose(C.conv_forward_at(x, w, n, p, q), y[n, p, q], rtol=1e-12, atol=1e-12)
    for n, h, v in ((0, 0, 0), (1, 9, 7), (0, 4, 5), (1, 3, 2)):
        np.testing.assert_allclose(C.conv_backward_data_at(dy, w, n, h, v), dx[n, h, v], rtol=1e-12, atol=1e-12)
    for k in range(3):
        np.testing.assert_allclose(C.conv_backward_filter_at(x, dy, k), dw[k], rtol=1e-12, atol=1e-12)
