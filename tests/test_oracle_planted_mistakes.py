"""The oracle's pins must catch a plausible mistake anywhere in it.  Each case
plants one into a patched copy of the oracle on the CPU and checks that the
pins (the independent torch restatements, the brute-force and library
comparisons) then disagree with it, while the unpatched oracle agrees with
them.  The mistakes: a flipped RoPE sign, the wrong RoPE frequency ladder, a
dropped norm gain, norm gains swapped between the two branches, a wrong
KV-head mapping, an off-by-one causal mask, a wrong softmax scale, a missing
bf16 rounding of the cache, silu as the identity, a missing Qwen3 q/k norm, a
LayerNorm without its mean, a tanh GELU, a sequential Falcon block; a shifted
padding, stride 1 or flipped taps in the convolution; unsigned codes or
per-row scales in the 8-bit format.  The synthetic hidden-vector norm gains
are all one, so the Llama cases run with non-unit gains.  Nothing here touches
the CUDA path."""
import numpy as np
import pytest

import gen
import oracle
from oracle import llama as L
from tests.test_oracle_falcon import _torch_falcon
from tests.test_oracle_pins import _torch_restatement

ATOL = 1e-6   # the tolerance of the restatement pins


def _attention_with(mapping=None, scale=None, causal_off=0):
    """causal GQA attention with one planted change (same structure as the oracle's)."""
    def attn(q, K, V, q_pos):
        T, n_q, d = q.shape
        n_kv, S, _ = K.shape
        group = n_q // n_kv
        mask = np.arange(S)[None, :] > (np.asarray(q_pos)[:, None] + causal_off)
        out = np.empty((T, n_q, d), np.float64)
        sc = (1.0 / np.sqrt(d)) if scale is None else scale(d)
        for j in range(n_q):
            g = (j // group) if mapping is None else mapping(j, n_kv, group)
            s = (q[:, j, :] @ K[g].T) * sc
            s[mask] = -np.inf
            out[:, j, :] = L.softmax(s, axis=-1) @ V[g]
        return out
    return attn


def _rope_flipped(x, cos, sin):
    half = x.shape[-1] // 2
    a, b = x[..., :half], x[..., half:]
    c, s = cos[:, None, :], sin[:, None, :]
    return np.concatenate([a * c + b * s, b * c - a * s], axis=-1)


def _rope_ladder(positions, head_dim, theta):
    i = np.arange(head_dim // 2, dtype=np.float64)
    ang = np.asarray(positions, np.float64)[:, None] * (theta ** (-i / head_dim))[None, :]
    return np.cos(ang), np.sin(ang)


LLAMA_MUTATIONS = {
    "rope sign": ("apply_rope", _rope_flipped),
    "rope frequency ladder": ("rope_cos_sin", _rope_ladder),
    "rmsnorm gain dropped": ("rmsnorm", lambda x, g, eps: x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps)),
    "kv head = j mod n_kv": ("causal_gqa_attention", _attention_with(mapping=lambda j, n_kv, group: j % n_kv)),
    "causal mask off by one": ("causal_gqa_attention", _attention_with(causal_off=1)),
    "softmax scale 1/d": ("causal_gqa_attention", _attention_with(scale=lambda d: 1.0 / d)),
    "no bf16 rounding of the cache": ("round_bf16", lambda x: np.asarray(x, np.float64)),
    "silu as identity": ("silu", lambda z: z),
}


def test_norm_gains_wired_to_the_wrong_norm_are_caught(tiny, monkeypatch):
    # the attention branch normalised with the MLP branch's gains and vice versa
    cfg, w, prompt, want = tiny
    swapped = dict(w)
    for l in range(cfg.n_layers):
        p = f"layers.{l}."
        swapped[p + "attn_norm"], swapped[p + "ffn_norm"] = w[p + "ffn_norm"], w[p + "attn_norm"]
    assert np.abs(_oracle_logits(cfg, swapped, prompt) - want).max() > 100 * ATOL


def _oracle_logits(cfg, w, prompt):
    m = oracle.OracleModel(cfg, w, max_tokens=64)
    return m.prefill(prompt)[0]


def _nonunit_norm_gains(cfg, w):
    """the synthetic models' hidden-vector norm gains are all one; here they are
    1 + 0.25 N(0, 1) (bf16), so that a gain dropped or taken from the wrong
    norm changes the logits"""
    r = np.random.default_rng(9)
    w = dict(w)
    for name in w:
        if name.endswith(("attn_norm", "ffn_norm", "final_norm")):
            g = (1.0 + 0.25 * r.standard_normal(w[name].shape)).astype(np.float32)
            w[name] = (g.view(np.uint32) >> 16).astype(np.uint16)   # truncated to bf16 bits
    return w


@pytest.fixture(scope="module")
def tiny():
    cfg = gen.TINY
    w = _nonunit_norm_gains(cfg, gen.make_weights(cfg))
    prompt = gen.make_prompt(cfg, cfg.prompt_len, seed=1)
    return cfg, w, prompt, _torch_restatement(cfg, w, prompt)


def test_unpatched_oracle_agrees_with_the_restatement(tiny):
    cfg, w, prompt, want = tiny
    assert np.abs(_oracle_logits(cfg, w, prompt) - want).max() <= ATOL


@pytest.mark.parametrize("name", sorted(LLAMA_MUTATIONS))
def test_planted_mistake_is_caught(tiny, monkeypatch, name):
    cfg, w, prompt, want = tiny
    attr, fn = LLAMA_MUTATIONS[name]
    monkeypatch.setattr(L, attr, fn)
    err = np.abs(_oracle_logits(cfg, w, prompt) - want).max()
    assert err > 100 * ATOL, f"{name}: the restatement pin would not notice ({err:.2e})"


def test_missing_qk_norm_is_caught(monkeypatch):
    cfg = gen.TINY.with_(name="tiny-qk", qk_norm=True)
    w = gen.make_weights(cfg)
    prompt = gen.make_prompt(cfg, 24, seed=2)
    want = _torch_restatement(cfg, w, prompt)
    assert np.abs(_oracle_logits(cfg, w, prompt) - want).max() <= ATOL
    real = L.rmsnorm
    # the per-head norm is the rmsnorm over head_dim: skip it there only
    monkeypatch.setattr(L, "rmsnorm", lambda x, g, eps: x if x.shape[-1] == cfg.head_dim else real(x, g, eps))
    assert np.abs(_oracle_logits(cfg, w, prompt) - want).max() > 100 * ATOL


def test_falcon_mistakes_are_caught(monkeypatch):
    cfg = gen.FALCON_TINY
    w = gen.make_weights(cfg)
    prompt = gen.make_prompt(cfg, 24, seed=2)
    want = _torch_falcon(cfg, w, prompt)
    assert np.abs(_oracle_logits(cfg, w, prompt) - want).max() <= ATOL
    # LayerNorm without the mean removed
    with monkeypatch.context() as mp:
        mp.setattr(L, "layernorm", lambda x, g, b, eps: x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps) * g + b)
        assert np.abs(_oracle_logits(cfg, w, prompt) - want).max() > 100 * ATOL
    # tanh-approximated GELU
    with monkeypatch.context() as mp:
        mp.setattr(L, "gelu", lambda z: 0.5 * z * (1 + np.tanh(np.sqrt(2 / np.pi) * (z + 0.044715 * z ** 3))))
        assert np.abs(_oracle_logits(cfg, w, prompt) - want).max() > ATOL
    # sequential instead of parallel: the MLP reads the stream after attention
    real = L.OracleModel._falcon_layer

    def sequential(self, l, x, T, P, pos, cos, sin, rnd):
        p = f"layers.{l}."
        zero_mlp = dict(self.w)
        saved = self.w
        self.w = zero_mlp
        zero_mlp[p + "w_down"] = np.zeros_like(saved[p + "w_down"])
        self._cache = None
        x1 = real(self, l, x, T, P, pos, cos, sin, rnd)          # x + attention only
        self.w = saved
        hm = L.layernorm(x1, self._vec(p + "ln_mlp"), self._vec(p + "ln_mlp_b"), self.cfg.rms_eps)
        return x1 + L.gelu(hm @ self.W(p + "w_up").T) @ self.W(p + "w_down").T
    with monkeypatch.context() as mp:
        mp.setattr(L.OracleModel, "_falcon_layer", sequential)
        assert np.abs(_oracle_logits(cfg, w, prompt) - want).max() > 100 * ATOL


# ------------------------------------------------- convolution and 8-bit format
def _conv_pin_error():
    """max deviation of the conv oracle from F.conv2d and autograd (the pin)"""
    import torch
    import torch.nn.functional as F
    from oracle import conv as C
    r = np.random.default_rng(4)
    x = torch.from_numpy(r.standard_normal((2, 10, 12, 5))).requires_grad_(True)
    w = torch.from_numpy(r.standard_normal((4, 3, 3, 5))).requires_grad_(True)
    dy = torch.from_numpy(r.standard_normal((2, 5, 6, 4)))
    y = F.conv2d(x.permute(0, 3, 1, 2), w.permute(0, 3, 1, 2), stride=2, padding=1).permute(0, 2, 3, 1)
    y.backward(dy)
    xn, wn = x.detach().numpy(), w.detach().numpy()
    return max(np.abs(C.conv_forward(xn, wn) - y.detach().numpy()).max(),
               np.abs(C.conv_backward_data(dy.numpy(), wn, 10, 12) - x.grad.numpy()).max(),
               np.abs(C.conv_backward_filter(xn, dy.numpy()) - w.grad.numpy()).max())


def test_conv_mistakes_are_caught(monkeypatch):
    from oracle import conv as C
    assert _conv_pin_error() < 1e-10
    with monkeypatch.context() as mp:     # padding on the far side only: every tap one pixel off
        mp.setattr(C, "_padded", lambda x: np.pad(np.asarray(x, np.float64), ((0, 0), (0, 2), (0, 2), (0, 0))))
        assert _conv_pin_error() > 1e-3
    with monkeypatch.context() as mp:     # stride 1 sampling
        mp.setattr(C, "STRIDE", 1)
        assert _conv_pin_error() > 1e-3
    real_fwd = C.conv_forward
    with monkeypatch.context() as mp:     # taps flipped (a true convolution, not the correlation)
        mp.setattr(C, "conv_forward", lambda x, w: real_fwd(x, np.asarray(w)[:, ::-1, ::-1, :]))
        assert _conv_pin_error() > 1e-3


def test_q8_mistakes_are_caught(monkeypatch):
    import struct
    from oracle import q8 as Q
    r = np.random.default_rng(6)
    codes = r.integers(-127, 128, size=(3, 96)).astype(np.int8)
    scales = (r.uniform(0.5, 1.5, size=(3, 3)) * 1e-3).astype(np.float16).view(np.uint16)
    x = r.standard_normal(96)

    def pin_error():
        # the brute-force pin: the block definition with an independent fp16 decoding
        got = Q.q8_matvec(codes, scales, x)
        want = [sum(struct.unpack("<e", struct.pack("<H", int(scales[i, b])))[0]
                    * sum(int(codes[i, 32 * b + k]) * float(x[32 * b + k]) for k in range(32)) for b in range(3))
                for i in range(3)]
        return float(np.abs(got - np.array(want)).max())
    assert pin_error() < 1e-12
    with monkeypatch.context() as mp:     # codes read as unsigned bytes
        mp.setattr(Q, "q8_matvec", _unsigned_matvec)
        assert pin_error() > 1e-6
    with monkeypatch.context() as mp:     # one scale per row instead of per block
        mp.setattr(Q, "fp16_bits_to_f64", lambda b: np.repeat(np.asarray(b, np.uint16).view(np.float16)
                                                              .astype(np.float64)[..., :1], np.asarray(b).shape[-1], -1))
        assert pin_error() > 1e-6


def _unsigned_matvec(codes, scales, x):
    """the block product with the codes read as unsigned bytes (the planted mistake)"""
    rows, cols = codes.shape
    nb = cols // 32
    q = np.asarray(codes).view(np.uint8).astype(np.float64).reshape(rows, nb, 32)
    d = np.asarray(scales, np.uint16).view(np.float16).astype(np.float64).reshape(rows, nb)
    return (np.einsum("rbk,bk->rb", q, np.asarray(x).reshape(nb, 32)) * d).sum(axis=1)
