"""GPU parity of the CNN-training sample's convolution layer (3x3, stride 2,
padding 1; forward, data gradient, filter gradient) through the C ABI against
the fp64 oracle (oracle/conv.py) on the same seeded bf16 tensors.

Tolerance, from the arithmetic: bf16 operands and their products are exact in
fp32, so the only error is the fp32 accumulation of each output's n products;
it stays below n * 2^-24 times the sum of |products| (the map applied to
|operands|).  The tests allow 2^-12 of that sum per element (n <= 4096 products
per output at these sizes) and a relative L2 error of 1e-5; an indexing mistake
(wrong tap, offset or parity class) moves whole outputs by O(1)."""
import numpy as np
import pytest

from gen import conv as gc
from oracle import conv as C

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2608_24204_gb300 import wici  # noqa: E402


def _f32(bits):
    return (np.asarray(bits, np.uint16).astype(np.uint32) << 16).view(np.float32)


def _dev(bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).cuda()


def _run(s: gc.ConvShape, x, w, dy):
    shape = wici.wici_conv_shape(s.n, s.c, s.h, s.w, s.k)
    ws = torch.zeros(wici.wici_conv_workspace_bytes(shape), dtype=torch.uint8, device="cuda")
    xd, wd, dyd = _dev(x), _dev(w), _dev(dy)
    y = torch.full((s.n, s.p, s.q, s.k), float("nan"), device="cuda")
    dx = torch.full((s.n, s.h, s.w, s.c), float("nan"), device="cuda")
    dw = torch.full((s.k, 3, 3, s.c), float("nan"), device="cuda")
    st = torch.cuda.current_stream().cuda_stream
    wici.wici_conv_forward(st, shape, xd.data_ptr(), wd.data_ptr(), y.data_ptr(), ws.data_ptr())
    wici.wici_conv_backward_data(st, shape, dyd.data_ptr(), wd.data_ptr(), dx.data_ptr(), ws.data_ptr())
    wici.wici_conv_backward_filter(st, shape, xd.data_ptr(), dyd.data_ptr(), dw.data_ptr(), ws.data_ptr())
    wici.wici_conv_status(st, ws.data_ptr())
    return y.cpu().numpy(), dx.cpu().numpy(), dw.cpu().numpy()


def _close(got, want, bound, what):
    got = np.asarray(got, np.float64)
    assert np.all(np.isfinite(got)), f"{what}: non-finite output"
    err = np.abs(got - want)
    worst = float(np.max(err / (bound * 2.0 ** -12 + 1e-30)))
    assert worst <= 1.0, f"{what}: error {worst:.2f} x the accumulation allowance (max abs {err.max():.3e})"
    rel = float(np.linalg.norm(got - want) / np.linalg.norm(want))
    assert rel <= 1e-5, f"{what}: rel-L2 {rel:.3e}"
    return rel


@pytest.mark.parametrize("shape", [
    gc.ConvShape(n=1, c=256, h=32, w=32, k=256),          # one tile of every kind
    gc.ConvShape(n=2, c=256, h=20, w=40, k=512),          # ragged: P = 10 rows, Q = 20 columns
    gc.ConvShape(n=1, c=512, h=16, w=48, k=256, seed=3),  # two channel tiles, three column tiles
])
def test_conv_layer_matches_oracle(shape):
    x, w, dy = gc.make_conv_inputs(shape)
    y, dx, dw = _run(shape, x, w, dy)
    xf, wf, dyf = _f32(x), _f32(w), _f32(dy)
    _close(y, C.conv_forward(xf, wf), C.abs_sum_bound(C.conv_forward, xf, wf), "forward")
    _close(dx, C.conv_backward_data(dyf, wf, shape.h, shape.w),
           C.abs_sum_bound(C.conv_backward_data, dyf, wf, shape.h, shape.w), "data gradient")
    _close(dw, C.conv_backward_filter(xf, dyf), C.abs_sum_bound(C.conv_backward_filter, xf, dyf), "filter gradient")


@pytest.mark.slow
def test_conv_layer_at_the_paper_sample_size_sampled():
    # 4 x 1024 x 224 x 224 input, 1024 output channels: sampled outputs against the
    # oracle's single-output forms, and the adjoint identity over the whole arrays
    s = gc.CNN_SAMPLE
    x, w, dy = gc.make_conv_inputs(s)
    y, dx, dw = _run(s, x, w, dy)
    xf, wf, dyf = _f32(x), _f32(w), _f32(dy)
    rng = np.random.default_rng(2026)
    for _ in range(24):
        n, p, q = int(rng.integers(s.n)), int(rng.integers(s.p)), int(rng.integers(s.q))
        want = C.conv_forward_at(xf, wf, n, p, q)
        bound = C.conv_forward_at(np.abs(xf), np.abs(wf), n, p, q)
        assert np.all(np.abs(y[n, p, q] - want) <= bound * 2.0 ** -12), ("forward", n, p, q)
    for h, v in ((0, 0), (223, 223), (1, 0), (0, 1), (117, 58), (64, 3)):   # every parity class and the borders
        n = int(rng.integers(s.n))
        want = C.conv_backward_data_at(dyf, wf, n, h, v)
        bound = C.conv_backward_data_at(np.abs(dyf), np.abs(wf), n, h, v)
        assert np.all(np.abs(dx[n, h, v] - want) <= bound * 2.0 ** -12), ("data gradient", n, h, v)
    for k in (0, 777):
        want = C.conv_backward_filter_at(xf, dyf, k)
        bound = C.conv_backward_filter_at(np.abs(xf), np.abs(dyf), k)
        # 50176 products per output: allow n * 2^-24 of the |products| sum
        assert np.all(np.abs(dw[k] - want) <= bound * (50176 * 2.0 ** -24)), ("filter gradient", k)
    a = float(np.dot(y.ravel().astype(np.float64), dyf.ravel().astype(np.float64)))
    b = float(np.dot(xf.ravel().astype(np.float64), dx.ravel().astype(np.float64)))
    c = float(np.dot(wf.ravel().astype(np.float64), dw.ravel().astype(np.float64)))
    assert abs(a - b) <= 1e-4 * abs(a) and abs(a - c) <= 1e-4 * abs(a)
