"""Pins for the oracle of the 8-bit block weight format (oracle/q8.py) and for
its seeded generator (gen/q8.py): the format's definition checked through an
independent fp16 decoding, brute force on small blocks, exact scale linearity,
a single-block closed form, and the whole tiny model against the independent
PyTorch restatement with the dequantised matrices."""
import struct

import numpy as np
import torch

import gen
import oracle
from gen import q8 as gq
from oracle import q8 as Q
from tests.test_oracle_pins import _torch_restatement

rng = np.random.default_rng(77)


def _random_block_matrix(rows, cols):
    codes = rng.integers(-127, 128, size=(rows, cols)).astype(np.int8)
    scales = (rng.uniform(0.5, 1.5, size=(rows, cols // 32)) * 1e-3).astype(np.float16).view(np.uint16)
    return codes, scales


def test_dequantize_is_code_times_the_fp16_scale_of_its_block():
    codes, scales = _random_block_matrix(5, 96)
    W = Q.q8_dequantize(codes, scales)
    for r in range(5):
        for c in range(96):
            d = struct.unpack("<e", struct.pack("<H", int(scales[r, c // 32])))[0]   # IEEE half, decoded by struct
            assert W[r, c] == d * int(codes[r, c])


def test_block_matvec_equals_brute_force_and_the_dense_product():
    codes, scales = _random_block_matrix(7, 128)
    x = rng.standard_normal(128)
    got = Q.q8_matvec(codes, scales, x)
    for r in range(7):
        acc = 0.0
        for b in range(4):
            d = struct.unpack("<e", struct.pack("<H", int(scales[r, b])))[0]
            acc += d * sum(int(codes[r, 32 * b + i]) * float(x[32 * b + i]) for i in range(32))
        assert abs(got[r] - acc) <= 1e-13 * (1 + abs(acc))
    np.testing.assert_allclose(Q.q8_dequantize(codes, scales) @ x, got, rtol=1e-13, atol=1e-16)


def test_doubling_every_scale_doubles_the_product_exactly():
    codes, scales = _random_block_matrix(4, 64)
    x = rng.standard_normal(64)
    doubled = (scales.view(np.float16) * np.float16(2)).view(np.uint16)
    assert np.array_equal(Q.q8_matvec(codes, doubled, x), 2 * Q.q8_matvec(codes, scales, x))


def test_one_nonzero_block_gives_scale_times_code_dot():
    codes = np.zeros((1, 96), np.int8)
    codes[0, 32:64] = np.arange(-16, 16)
    scales = np.array([[0x3C00, 0x3800, 0x4000]], np.uint16)   # 1.0, 0.5, 2.0 as fp16
    x = np.linspace(-1, 1, 96)
    want = 0.5 * float(np.dot(np.arange(-16, 16), x[32:64]))
    assert Q.q8_matvec(codes, scales, x)[0] == want


def test_generator_codes_scales_and_statistics():
    cfg = gen.TINY
    names = gq.q8_names(cfg)
    # ffn 688 is not a whole number of 32-column blocks: the down matrices stay bf16
    assert len(names) == 6 * cfg.n_layers and all(n.split(".")[-1] in gq.Q8_MATRICES for n in names)
    assert "layers.0.wd" not in names
    assert len(gq.q8_names(gen.LLAMA_8B)) == 7 * gen.LLAMA_8B.n_layers
    codes, scales = gq.make_q8_tensor(cfg, "layers.1.wg")
    assert codes.dtype == np.int8 and codes.min() >= -127 and codes.max() <= 127
    assert codes.shape == (cfg.ffn_dim, cfg.hidden) and scales.shape == (cfg.ffn_dim, cfg.hidden // 32)
    d = scales.view(np.float16).astype(np.float64)
    assert np.all(np.isfinite(d)) and d.min() > 0
    assert abs(Q.q8_dequantize(codes, scales).std() - cfg.weight_std) < 0.1 * cfg.weight_std
    c2, s2 = gq.make_q8_tensor(cfg, "layers.1.wg")
    assert np.array_equal(codes, c2) and np.array_equal(scales, s2)
    c3, _ = gq.make_q8_tensor(cfg, "layers.1.wu")
    assert not np.array_equal(codes, c3)


def test_tiny_model_in_the_8bit_format_matches_the_torch_restatement():
    cfg = gen.TINY
    w = gen.make_weights(cfg)
    q8 = gq.make_q8_weights(cfg)
    prompt = gen.make_prompt(cfg, cfg.prompt_len, seed=1)
    m = oracle.OracleModel(cfg, w, max_tokens=64, q8_weights=q8)
    got, tok = m.prefill(prompt)

    def dequant_torch(codes, scales):   # the format, decoded with torch ops
        d = torch.from_numpy(scales.view(np.float16).copy()).double().repeat_interleave(32, dim=1)
        return torch.from_numpy(codes.astype(np.int64)).double() * d

    want = _torch_restatement(cfg, w, prompt, mats={n: dequant_torch(*v) for n, v in q8.items()})
    np.testing.assert_allclose(got, want, rtol=0, atol=1e-6)
    assert tok == int(np.argmax(want))
    plain, _ = oracle.OracleModel(cfg, w, max_tokens=64).prefill(prompt)
    assert not np.allclose(got, plain)   # the 8-bit matrices are really used


def test_block_matvec_at_the_8b_layer_widths():
    # K = 4096 (Wo) and K = 14336 (Wd), the widths the decode GEMV phases stream:
    # the block-wise product against the dense product of the dequantised rows
    cfg = gen.LLAMA_8B
    xr = np.random.default_rng(5)
    for name in ("layers.0.wo", "layers.0.wd"):
        codes, scales = gq.make_q8_tensor(cfg, name)
        codes, scales = codes[:384], scales[:384]
        x = xr.standard_normal(codes.shape[1])
        got = Q.q8_matvec(codes, scales, x)
        want = Q.q8_dequantize(codes, scales) @ x
        np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-14 * float(np.abs(want).max()))
        # one row by the scalar definition, block by block
        d = Q.fp16_bits_to_f64(scales[7])
        acc = sum(d[b] * float(np.dot(codes[7, 32 * b:32 * b + 32].astype(np.float64), x[32 * b:32 * b + 32]))
                  for b in range(codes.shape[1] // 32))
        assert abs(got[7] - acc) <= 1e-12 * (1 + abs(acc))
