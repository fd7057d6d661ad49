"""Pins for the Falcon block of the oracle (oracle/llama.py, `block == "falcon"`):
LayerNorm against torch's layer_norm and its shift invariance, GELU against
torch's exact gelu and the identity gelu(z) - gelu(-z) = z, the residual
structure (with every branch matrix zeroed the model is the final LayerNorm of
the embedding row through the head), the parallel structure (zeroing one
branch leaves exactly the other's contribution), incremental decode against
full recompute, and the whole tiny model against an independent PyTorch
restatement (F.layer_norm, F.gelu, complex-number RoPE, scaled dot-product
attention on repeated KV heads)."""
import numpy as np
import torch
import torch.nn.functional as F

import gen
import oracle
from oracle import llama as L

rng = np.random.default_rng(31)
CFG = gen.FALCON_TINY


def test_layernorm_matches_torch_and_is_shift_invariant():
    x = rng.standard_normal((5, 96)) * 3 + 1.5
    g = rng.standard_normal(96)
    b = rng.standard_normal(96)
    got = L.layernorm(x, g, b, 1e-5)
    want = F.layer_norm(torch.from_numpy(x), (96,), torch.from_numpy(g), torch.from_numpy(b), eps=1e-5).numpy()
    np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-12)
    # a constant added to every element changes nothing (the mean is removed) ...
    np.testing.assert_allclose(L.layernorm(x + 7.25, g, b, 1e-5), got, rtol=1e-9, atol=1e-9)
    # ... while RMSNorm, which keeps the mean, does change
    assert np.abs(L.rmsnorm(x + 7.25, g, 1e-5) - L.rmsnorm(x, g, 1e-5)).max() > 1e-2
    # unit weight, zero bias: zero mean and unit (biased) variance up to eps
    y = L.layernorm(x, np.ones(96), np.zeros(96), 0.0)
    np.testing.assert_allclose(y.mean(axis=-1), 0.0, atol=1e-12)
    np.testing.assert_allclose((y * y).mean(axis=-1), 1.0, rtol=1e-12)


def test_gelu_matches_torch_exact_gelu_and_its_odd_part():
    z = np.linspace(-6, 6, 241)
    np.testing.assert_allclose(L.gelu(z), F.gelu(torch.from_numpy(z), approximate="none").numpy(),
                               rtol=1e-12, atol=1e-15)
    # gelu(z) = z Phi(z) and Phi(z) + Phi(-z) = 1, so gelu(z) - gelu(-z) = z
    np.testing.assert_allclose(L.gelu(z) - L.gelu(-z), z, rtol=1e-13, atol=1e-15)
    assert L.gelu(np.array([0.0]))[0] == 0.0


def _weights():
    return gen.make_weights(CFG)


def _bf16(a):
    return L.bf16_bits_to_f64(a)


def test_generator_gives_falcon_tensors_with_nontrivial_norms():
    w = _weights()
    names = {n for n, _, _ in gen.tensor_specs(CFG)}
    assert {"layers.0.ln_attn", "layers.0.ln_attn_b", "layers.1.ln_mlp_b", "layers.1.w_up", "final_norm_b"} <= names
    assert not any(n.endswith(("wg", "wu", "wd", "attn_norm", "ffn_norm")) for n in names)
    assert "lm_head" not in names                       # tied embeddings
    g = _bf16(w["layers.0.ln_attn"])
    assert abs(g.mean() - 1.0) < 0.1 and 0.15 < g.std() < 0.35
    b = _bf16(w["layers.0.ln_mlp_b"])
    assert abs(b.mean()) < 0.01 and 0.01 < b.std() < 0.03


def test_zero_branches_reduce_to_final_layernorm_of_the_embedding():
    w = _weights()
    for name in list(w):
        if name.startswith("layers.") and name.split(".")[-1] in ("wq", "wk", "wv", "wo", "w_up", "w_down"):
            w[name] = np.zeros_like(w[name])
    tok = 333
    m = oracle.OracleModel(CFG, w, max_tokens=4)
    logits, _ = m.prefill([tok])
    e = _bf16(w["embed"][tok])
    c = e - e.mean()
    h = c / np.sqrt(float(np.mean(c * c)) + CFG.rms_eps) * _bf16(w["final_norm"])[0] + _bf16(w["final_norm_b"])[0]
    np.testing.assert_allclose(logits, _bf16(w["embed"]) @ h, rtol=1e-12, atol=1e-13)


def test_parallel_branches_add_independently():
    # one layer: logits(both branches) relate to the final LayerNorm of
    # x + A + M; zeroing Wo removes A only, zeroing W_down removes M only, so the
    # pre-norm hidden states satisfy h(both) - h(no attn) - h(no mlp) + h(none) = 0
    w = _weights()
    tokens = gen.make_prompt(CFG, 12, seed=3)
    cfg1 = CFG.with_(n_layers=1)

    def hidden(wd):
        m = oracle.OracleModel(cfg1, wd, max_tokens=64)
        captured = {}
        orig = m._falcon_layer

        def spy(*a, **k):
            captured["x"] = orig(*a, **k)
            return captured["x"]
        m._falcon_layer = spy
        m.forward(tokens)
        return captured["x"]

    def zeroed(*names):
        wd = dict(w)
        for n in names:
            wd["layers.0." + n] = np.zeros_like(w["layers.0." + n])
        return wd
    both, no_a, no_m, none = hidden(w), hidden(zeroed("wo")), hidden(zeroed("w_down")), hidden(zeroed("wo", "w_down"))
    x0 = _bf16(w["embed"][tokens])
    np.testing.assert_allclose(none, x0, rtol=0, atol=0)
    np.testing.assert_allclose(both - no_a - no_m + none, 0.0, atol=1e-12)
    assert np.abs(both - no_a).max() > 1e-3 and np.abs(both - no_m).max() > 1e-3


def test_incremental_decode_equals_full_recompute():
    w = _weights()
    prompt = gen.make_prompt(CFG, 18, seed=1)
    extra = [7, 1000, 64, 2]
    inc = oracle.OracleModel(CFG, w, max_tokens=32)
    inc.prefill(prompt)
    for t in extra:
        last, _ = inc.decode(t)
    full = oracle.OracleModel(CFG, w, max_tokens=32)
    want, _ = full.prefill(np.concatenate([prompt, extra]))
    np.testing.assert_allclose(last, want, rtol=1e-9, atol=1e-11)


def _torch_falcon(cfg, w, tokens):
    def W(n):
        return torch.from_numpy((w[n].astype(np.uint32) << 16).view(np.float32)).double()

    T = len(tokens)
    d, nq, nkv, H = cfg.head_dim, cfg.n_q_heads, cfg.n_kv_heads, cfg.hidden
    x = W("embed")[torch.from_numpy(np.asarray(tokens, np.int64))]
    pos = torch.arange(T, dtype=torch.float64)
    freq = cfg.rope_theta ** (-torch.arange(0, d, 2, dtype=torch.float64) / d)
    rot = torch.polar(torch.ones(T, d // 2, dtype=torch.float64), pos[:, None] * freq[None, :])

    def rope(t):
        z = torch.complex(t[..., : d // 2], t[..., d // 2:]) * rot[:, None, :]
        return torch.cat([z.real, z.imag], dim=-1)

    def bf16(t):
        return t.float().bfloat16().double()

    for l in range(cfg.n_layers):
        p = f"layers.{l}."
        ha = F.layer_norm(x, (H,), W(p + "ln_attn")[0], W(p + "ln_attn_b")[0], eps=cfg.rms_eps)
        hm = F.layer_norm(x, (H,), W(p + "ln_mlp")[0], W(p + "ln_mlp_b")[0], eps=cfg.rms_eps)
        q = rope(F.linear(ha, W(p + "wq")).view(T, nq, d))
        k = bf16(rope(F.linear(ha, W(p + "wk")).view(T, nkv, d))).repeat_interleave(nq // nkv, dim=1)
        v = bf16(F.linear(ha, W(p + "wv")).view(T, nkv, d)).repeat_interleave(nq // nkv, dim=1)
        o = F.scaled_dot_product_attention(q.transpose(0, 1), k.transpose(0, 1), v.transpose(0, 1),
                                           is_causal=True).transpose(0, 1).reshape(T, nq * d)
        x = x + F.linear(o, W(p + "wo")) + F.linear(F.gelu(F.linear(hm, W(p + "w_up"))), W(p + "w_down"))
    hf = F.layer_norm(x[-1], (H,), W("final_norm")[0], W("final_norm_b")[0], eps=cfg.rms_eps)
    return (W("embed") @ hf).numpy()


def test_tiny_falcon_matches_independent_torch_restatement():
    w = _weights()
    prompt = gen.make_prompt(CFG, CFG.prompt_len, seed=1)
    m = oracle.OracleModel(CFG, w, max_tokens=64)
    got, tok = m.prefill(prompt)
    want = _torch_falcon(CFG, w, prompt)
    np.testing.assert_allclose(got, want, rtol=0, atol=1e-6)
    assert tok == int(np.argmax(want))


def test_binding_refuses_a_block_it_has_no_kernels_for():
    import pytest
    from paper_2608_24204_gb300 import wici
    with pytest.raises(ValueError):
        wici.make_config(CFG, max_tokens=64)
