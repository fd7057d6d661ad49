"""Pins for the seeded input generator (gen/): it is a published counter-based
generator, so its bytes are checked against the published definition and
against an independent pure-Python restatement."""
import struct

import numpy as np

import gen

M64 = (1 << 64) - 1
GAMMA = 0x9E3779B97F4A7C15


def _mix(z):
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & M64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & M64
    return z ^ (z >> 31)


def test_splitmix64_published_vector():
    # splitmix64 seeded with 1234567: the first five outputs of the reference
    # generator (Vigna's public-domain splitmix64.c), as printed by its test programs.
    expect = [6457827717110365317, 3203168211198807973, 9817491932198370423,
              4593380528125082431, 16408922859458223821]
    assert [gen.draw(1234567, i) for i in range(5)] == expect


def _py_normal_bf16(seed, tag, std, e):
    key = _mix(((seed << 32) ^ tag) & M64)
    acc = 0
    for j in range(3):
        r = _mix((key + (3 * e + j + 1) * GAMMA) & M64)
        acc += sum((r >> (16 * k)) & 0xFFFF for k in range(4))
    s = (acc + 6 - 393216) / 65536.0 * std
    f = struct.unpack("<I", struct.pack("<f", s))[0]          # round double -> float (RNE)
    f += 0x7FFF + ((f >> 16) & 1)                            # float -> bf16 (RNE)
    return (f >> 16) & 0xFFFF


def test_weight_bytes_match_pure_python_restatement():
    cfg = gen.TINY
    for name in ("embed", "layers.1.wd", "lm_head"):
        t = gen.make_tensor(cfg, name).reshape(-1)
        tag = [n for n, _, _ in gen.tensor_specs(cfg)].index(name)
        for e in (0, 1, 2, 777, t.size - 1):
            assert int(t[e]) == _py_normal_bf16(cfg.weight_seed, tag, cfg.weight_std, e)


def test_norm_gains_are_one_and_prompt_in_range():
    cfg = gen.TINY
    assert np.all(gen.make_tensor(cfg, "layers.0.attn_norm") == 0x3F80)
    p = gen.make_prompt(cfg, 4096, seed=1)
    assert p.dtype == np.int32 and p.min() >= 0 and p.max() < cfg.vocab
    key = _mix(((1 << 32) ^ gen.PROMPT_TAG) & M64)
    assert [int(v) for v in p[:4]] == [_mix((key + (i + 1) * GAMMA) & M64) % cfg.vocab
                                       for i in range(4)]
    assert not np.array_equal(p, gen.make_prompt(cfg, 4096, seed=2))


def test_sum_of_twelve_uniforms_moments():
    # Irwin-Hall(12) - 6: mean 0, variance 1, excess kurtosis -1/10, support [-6, 6]
    x = gen.normal_f64(0, 3, 2_000_000)
    assert abs(x.mean()) < 3e-3
    assert abs(x.var() - 1.0) < 5e-3
    assert abs((x ** 4).mean() / x.var() ** 2 - 2.9) < 2e-2
    assert np.abs(x).max() < 6.0


def test_distinct_tensors_and_determinism():
    cfg = gen.TINY
    a = gen.make_tensor(cfg, "layers.0.wq")
    b = gen.make_tensor(cfg, "layers.0.wk")
    assert not np.array_equal(a[: b.shape[0]], b)
    assert np.array_equal(a, gen.make_tensor(cfg, "layers.0.wq"))
    f = (a.astype(np.uint32) << 16).view(np.float32)
    assert abs(f.std() - 0.02) < 1e-3


def test_byte_accounting_matches_hand_count():
    cfg = gen.LLAMA_8B
    H, F, V, L = 4096, 14336, 128256, 32
    per_layer = H * (4096 + 2 * 1024) + 4096 * H + 3 * H * F + 2 * H
    weights = 2 * (L * per_layer + V * H + H + H)           # + embed row + final norm
    assert gen.decode_bytes_per_token(cfg, 0) == weights
    assert gen.decode_bytes_per_token(cfg, 10) - weights == 10 * L * 2 * 1024 * 2
