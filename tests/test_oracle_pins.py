"""Pins for the CPU oracle: closed forms, invariants, special cases that reduce
to library routines, brute force on tiny inputs and an independent PyTorch
restatement of the whole model.  Each pin is chosen so that a plausible slip
(dropped term, wrong sign, wrong head index, transposed operand, off-by-one
position) fails at least one test."""
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import gen
import oracle
from oracle import llama as L

rng = np.random.default_rng(1234)


# ------------------------------------------------------------------ bf16 ----

def test_bf16_bits_known_patterns():
    bits = np.array([0x3F80, 0xC000, 0x3C00, 0x0000, 0x8000, 0x4049], np.uint16)
    assert list(L.bf16_bits_to_f64(bits)) == [1.0, -2.0, 2.0 ** -7, 0.0, -0.0, 3.140625]


def test_round_bf16_matches_torch_on_float32_values():
    x = (rng.standard_normal(200_000) * np.exp(rng.uniform(-20, 20, 200_000))).astype(np.float32)
    want = torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()
    assert np.array_equal(L.round_bf16(x.astype(np.float64)), want)


def test_round_bf16_ties_to_even_and_single_rounding():
    one = 1.0
    assert L.round_bf16(np.array([one + 2 ** -8]))[0] == 1.0                 # tie -> even
    assert L.round_bf16(np.array([one + 3 * 2 ** -8]))[0] == one + 2 ** -6    # tie -> even (up)
    assert L.round_bf16(np.array([-(one + 2 ** -8)]))[0] == -1.0
    # just above the tie by 2^-40: a detour through float32 would first drop the 2^-40
    # and then round the exact tie down to 1.0; one direct rounding goes up
    assert L.round_bf16(np.array([one + 2 ** -8 + 2 ** -40]))[0] == one + 2 ** -7


# --------------------------------------------------------------- RMSNorm ----

def test_rmsnorm_closed_form_constant_vector():
    for c in (3.0, -0.25, 1e-3):
        x = np.full(64, c)
        g = np.linspace(0.5, 2.0, 64)
        eps = 1e-5
        want = g * c / math.sqrt(c * c + eps)
        np.testing.assert_allclose(L.rmsnorm(x, g, eps), want, rtol=1e-14)


def test_rmsnorm_matches_torch_rms_norm():
    x = rng.standard_normal((5, 96)) * 3
    g = rng.standard_normal(96)
    want = F.rms_norm(torch.from_numpy(x), (96,), torch.from_numpy(g), eps=1e-6).numpy()
    np.testing.assert_allclose(L.rmsnorm(x, g, 1e-6), want, rtol=1e-12, atol=1e-14)


# ------------------------------------------------------------------ RoPE ----

def test_rope_d2_is_plane_rotation_by_position():
    x = np.array([[[0.6, -1.3]]])                   # [T=1, heads=1, d=2]: one pair, frequency 1
    for p in (0, 1, 7, 1000):
        c, s = L.rope_cos_sin(np.array([p]), 2, 10000.0)
        got = L.apply_rope(x, c, s)[0, 0]
        R = np.array([[math.cos(p), -math.sin(p)], [math.sin(p), math.cos(p)]])
        np.testing.assert_allclose(got, R @ x[0, 0], rtol=1e-13, atol=1e-14)


def test_rope_pairs_i_with_i_plus_half_and_frequency_ladder():
    theta, p = 500000.0, 37
    x = rng.standard_normal((1, 1, 4))
    c, s = L.rope_cos_sin(np.array([p]), 4, theta)
    got = L.apply_rope(x, c, s)[0, 0]
    a0, a1 = p * 1.0, p * theta ** -0.5            # pair 0 = (0, 2), pair 1 = (1, 3)
    want = [x[0, 0, 0] * math.cos(a0) - x[0, 0, 2] * math.sin(a0),
            x[0, 0, 1] * math.cos(a1) - x[0, 0, 3] * math.sin(a1),
            x[0, 0, 2] * math.cos(a0) + x[0, 0, 0] * math.sin(a0),
            x[0, 0, 3] * math.cos(a1) + x[0, 0, 1] * math.sin(a1)]
    np.testing.assert_allclose(got, want, rtol=1e-13, atol=1e-14)


def test_rope_norm_identity_and_relative_position():
    d = 128
    q = rng.standard_normal((1, 1, d))
    k = rng.standard_normal((1, 1, d))
    c0, s0 = L.rope_cos_sin(np.array([0]), d, 10000.0)
    np.testing.assert_array_equal(L.apply_rope(q, c0, s0), q)
    for p in (1, 15, 16, 8447):
        c, s = L.rope_cos_sin(np.array([p]), d, 10000.0)
        r = L.apply_rope(q, c, s)[0, 0]
        pair_in = q[0, 0, : d // 2] ** 2 + q[0, 0, d // 2:] ** 2
        pair_out = r[: d // 2] ** 2 + r[d // 2:] ** 2
        np.testing.assert_allclose(pair_out, pair_in, rtol=1e-12)

    def dot(pq, pk):
        cq, sq = L.rope_cos_sin(np.array([pq]), d, 10000.0)
        ck, sk = L.rope_cos_sin(np.array([pk]), d, 10000.0)
        return float(L.apply_rope(q, cq, sq).ravel() @ L.apply_rope(k, ck, sk).ravel())

    assert dot(40, 13) == pytest.approx(dot(40 + 501, 13 + 501), rel=1e-9)
    assert dot(40, 13) != pytest.approx(dot(41, 13), rel=1e-6)


def test_rope_matches_complex_multiplication():
    T, heads, d, theta = 6, 3, 64, 500000.0
    x = rng.standard_normal((T, heads, d))
    pos = np.array([0, 1, 2, 100, 2047, 8447])
    c, s = L.rope_cos_sin(pos, d, theta)
    z = torch.complex(torch.from_numpy(x[..., : d // 2]), torch.from_numpy(x[..., d // 2:]))
    freq = theta ** (-torch.arange(0, d, 2, dtype=torch.float64) / d)
    rot = torch.polar(torch.ones(T, d // 2, dtype=torch.float64),
                      torch.from_numpy(pos).double()[:, None] * freq[None, :])
    zr = z * rot[:, None, :]
    want = torch.cat([zr.real, zr.imag], dim=-1).numpy()
    np.testing.assert_allclose(L.apply_rope(x, c, s), want, rtol=1e-10, atol=1e-12)


# ------------------------------------------------------- softmax / silu ----

def test_softmax_rows_sum_to_one_and_mask():
    s = rng.standard_normal((7, 33)) * 20
    s[:, 5] = -np.inf
    p = L.softmax(s)
    np.testing.assert_allclose(p.sum(-1), 1.0, atol=1e-12)
    assert np.all(p[:, 5] == 0.0)
    np.testing.assert_allclose(L.softmax(s + 123.0), p, rtol=1e-12)


def test_silu_special_values_and_torch():
    assert L.silu(np.array([0.0]))[0] == 0.0
    z = np.linspace(-30, 30, 301)
    np.testing.assert_allclose(L.silu(z), F.silu(torch.from_numpy(z)).numpy(), rtol=1e-13, atol=1e-15)
    assert abs(L.silu(np.array([-40.0]))[0]) < 1e-15


# ------------------------------------------------------------- attention ----

def _brute_attention(q, K, V, q_pos):
    T, n_q, d = q.shape
    n_kv = K.shape[0]
    out = np.zeros_like(q)
    for t in range(T):
        for j in range(n_q):
            g = j // (n_q // n_kv)
            sc = [sum(q[t, j, i] * K[g, s, i] for i in range(d)) / math.sqrt(d)
                  for s in range(q_pos[t] + 1)]
            m = max(sc)
            e = [math.exp(v - m) for v in sc]
            z = sum(e)
            for i in range(d):
                out[t, j, i] = sum(e[s] * V[g, s, i] for s in range(len(e))) / z
    return out


def test_attention_brute_force_tiny():
    q = rng.standard_normal((3, 4, 4))
    K = rng.standard_normal((2, 6, 4))
    V = rng.standard_normal((2, 6, 4))
    pos = np.array([2, 3, 5])
    np.testing.assert_allclose(L.causal_gqa_attention(q, K, V, pos),
                               _brute_attention(q, K, V, pos), rtol=1e-12, atol=1e-13)


def test_attention_single_key_returns_value_exactly():
    q = rng.standard_normal((1, 2, 8))
    K = rng.standard_normal((1, 4, 8))
    V = rng.standard_normal((1, 4, 8))
    out = L.causal_gqa_attention(q, K, V, np.array([0]))
    assert np.array_equal(out[0, 0], V[0, 0]) and np.array_equal(out[0, 1], V[0, 0])


def test_gqa_equals_mha_with_repeated_kv_heads_sdpa():
    T, n_q, n_kv, d = 9, 8, 2, 16
    q = rng.standard_normal((T, n_q, d))
    K = rng.standard_normal((n_kv, T, d))
    V = rng.standard_normal((n_kv, T, d))
    got = L.causal_gqa_attention(q, K, V, np.arange(T))
    Kr = np.repeat(K, n_q // n_kv, axis=0)                # head j -> kv head j // group
    Vr = np.repeat(V, n_q // n_kv, axis=0)
    want = F.scaled_dot_product_attention(
        torch.from_numpy(q.transpose(1, 0, 2)), torch.from_numpy(Kr), torch.from_numpy(Vr),
        is_causal=True).numpy().transpose(1, 0, 2)
    np.testing.assert_allclose(got, want, rtol=1e-10, atol=1e-12)
    # n_kv = n_q is plain multi-head attention
    Kf = rng.standard_normal((n_q, T, d))
    Vf = rng.standard_normal((n_q, T, d))
    want = F.scaled_dot_product_attention(
        torch.from_numpy(q.transpose(1, 0, 2)), torch.from_numpy(Kf), torch.from_numpy(Vf),
        is_causal=True).numpy().transpose(1, 0, 2)
    np.testing.assert_allclose(L.causal_gqa_attention(q, Kf, Vf, np.arange(T)), want,
                               rtol=1e-10, atol=1e-12)


def test_greedy_lowest_index_on_tie():
    x = np.array([0.1, 0.7, -2.0, 0.7, 0.3])
    assert L.greedy(x) == 1


# -------------------------------------------------------------- model ------

def _tiny_weights(cfg):
    return gen.make_weights(cfg)


def test_zero_layers_reduce_to_embedding_through_final_norm_and_head():
    cfg = gen.TINY
    w = _tiny_weights(cfg)
    for name in list(w):
        if name.startswith("layers.") and not name.endswith("norm"):
            w[name] = np.zeros_like(w[name])
    tok = 517
    m = oracle.OracleModel(cfg, w, max_tokens=4)
    logits, _ = m.prefill([tok])
    e = L.bf16_bits_to_f64(w["embed"][tok])
    h = e / math.sqrt(float(np.mean(e * e)) + cfg.rms_eps)
    want = L.bf16_bits_to_f64(w["lm_head"]) @ h
    np.testing.assert_allclose(logits, want, rtol=1e-12, atol=1e-14)


def test_incremental_decode_equals_full_causal_recompute():
    cfg = gen.TINY
    w = _tiny_weights(cfg)
    prompt = gen.make_prompt(cfg, 20, seed=1)
    extra = [5, 901, 77, 0, 1023]
    inc = oracle.OracleModel(cfg, w, max_tokens=32)
    inc.prefill(prompt)
    for t in extra:
        last, _ = inc.decode(t)
    full = oracle.OracleModel(cfg, w, max_tokens=32)
    want, _ = full.prefill(np.concatenate([prompt, extra]))
    np.testing.assert_allclose(last, want, rtol=1e-9, atol=1e-11)
    # chunked prefill (agentic turns) is the same computation
    ch = oracle.OracleModel(cfg, w, max_tokens=32)
    ch.prefill(prompt[:7])
    ch.prefill(prompt[7:])
    got, _ = ch.prefill(np.array(extra))
    np.testing.assert_allclose(got, want, rtol=1e-9, atol=1e-11)


def test_forced_decode_rows_equal_step_by_step_decode():
    # decode_forced feeds a known token sequence in one causal pass; each row must
    # be the logits that feeding the tokens one step at a time gives
    cfg = gen.TINY
    w = _tiny_weights(cfg)
    prompt = gen.make_prompt(cfg, 12, seed=1)
    forced = gen.make_prompt(cfg, 6, seed=9)
    step = oracle.OracleModel(cfg, w, max_tokens=32)
    step.prefill(prompt)
    want = [step.decode(int(t)) for t in forced]
    one = oracle.OracleModel(cfg, w, max_tokens=32)
    first, _ = one.prefill(prompt)
    rows = one.decode_forced(forced)
    assert rows.shape == (len(forced), cfg.vocab) and one.kv_len == step.kv_len
    for r, (logits, tok) in zip(rows, want):
        np.testing.assert_allclose(r, logits, rtol=1e-9, atol=1e-11)
        assert oracle.greedy(r) == tok
    # the last row of an all-rows pass is the ordinary last-position result
    a = oracle.OracleModel(cfg, w, max_tokens=32)
    b = oracle.OracleModel(cfg, w, max_tokens=32)
    np.testing.assert_allclose(a.forward(prompt, all_rows=True)[-1], b.forward(prompt), rtol=1e-12, atol=1e-13)


def _torch_restatement(cfg, w, tokens, mats=None):
    """The whole forward, written independently with torch library ops (fp64):
    F.rms_norm, complex-number RoPE, F.linear (with the QKV bias when present),
    F.scaled_dot_product_attention on repeated KV heads, F.silu.  `mats`, when
    given, supplies fp64 torch matrices that take the place of bf16 tensors."""
    def W(n):
        if mats is not None and n in mats:
            return mats[n]
        return torch.from_numpy((w[n].astype(np.uint32) << 16).view(np.float32)).double()

    def B(n):
        return W(n)[0] if cfg.qkv_bias else None

    T = len(tokens)
    d, nq, nkv = cfg.head_dim, cfg.n_q_heads, cfg.n_kv_heads
    x = W("embed")[torch.from_numpy(np.asarray(tokens, np.int64))]
    pos = torch.arange(T, dtype=torch.float64)
    freq = cfg.rope_theta ** (-torch.arange(0, d, 2, dtype=torch.float64) / d)
    rot = torch.polar(torch.ones(T, d // 2, dtype=torch.float64), pos[:, None] * freq[None, :])

    def rope(t):                                               # [T, heads, d]
        z = torch.complex(t[..., : d // 2], t[..., d // 2:]) * rot[:, None, :]
        return torch.cat([z.real, z.imag], dim=-1)

    def bf16(t):
        return t.float().bfloat16().double()

    for l in range(cfg.n_layers):
        p = f"layers.{l}."
        h = F.rms_norm(x, (cfg.hidden,), W(p + "attn_norm")[0], eps=cfg.rms_eps)
        q = F.linear(h, W(p + "wq"), B(p + "bq")).view(T, nq, d)
        k = F.linear(h, W(p + "wk"), B(p + "bk")).view(T, nkv, d)
        if cfg.qk_norm:
            q = F.rms_norm(q, (d,), W(p + "q_norm")[0], eps=cfg.rms_eps)
            k = F.rms_norm(k, (d,), W(p + "k_norm")[0], eps=cfg.rms_eps)
        q = rope(q)
        k = bf16(rope(k))
        v = bf16(F.linear(h, W(p + "wv"), B(p + "bv")).view(T, nkv, d))
        k = k.repeat_interleave(nq // nkv, dim=1)
        v = v.repeat_interleave(nq // nkv, dim=1)
        o = F.scaled_dot_product_attention(q.transpose(0, 1), k.transpose(0, 1), v.transpose(0, 1),
                                           is_causal=True).transpose(0, 1).reshape(T, nq * d)
        x = x + o @ W(p + "wo").T
        h2 = F.rms_norm(x, (cfg.hidden,), W(p + "ffn_norm")[0], eps=cfg.rms_eps)
        x = x + (F.silu(h2 @ W(p + "wg").T) * (h2 @ W(p + "wu").T)) @ W(p + "wd").T
    hf = F.rms_norm(x[-1], (cfg.hidden,), W("final_norm")[0], eps=cfg.rms_eps)
    head = "embed" if cfg.tied_embeddings else "lm_head"
    return (W(head) @ hf).numpy()


def test_tiny_model_matches_independent_torch_restatement():
    cfg = gen.TINY
    w = _tiny_weights(cfg)
    prompt = gen.make_prompt(cfg, cfg.prompt_len, seed=1)
    m = oracle.OracleModel(cfg, w, max_tokens=64)
    got, tok = m.prefill(prompt)
    want = _torch_restatement(cfg, w, prompt)
    np.testing.assert_allclose(got, want, rtol=0, atol=1e-6)
    assert tok == int(np.argmax(want))


def test_one_wide_layer_matches_torch_restatement():
    # Llama-3.2-1B widths (GQA 32/8, d=64), one layer, short prompt, narrow vocab
    cfg = gen.LLAMA_1B.with_(name="1b-cut", n_layers=1, vocab=512, tied_embeddings=False)
    w = gen.make_weights(cfg)
    prompt = gen.make_prompt(cfg, 24, seed=1)
    got, _ = oracle.OracleModel(cfg, w, max_tokens=32).prefill(prompt)
    np.testing.assert_allclose(got, _torch_restatement(cfg, w, prompt), rtol=0, atol=1e-6)


TINY_QK = gen.TINY.with_(name="tiny-qk", qk_norm=True, rope_theta=1e6, rms_eps=1e-6)


def test_qk_norm_model_matches_independent_torch_restatement():
    cfg = TINY_QK
    w = _tiny_weights(cfg)
    assert "layers.0.q_norm" in w and w["layers.0.q_norm"].shape == (1, cfg.head_dim)
    prompt = gen.make_prompt(cfg, 24, seed=1)
    got, _ = oracle.OracleModel(cfg, w, max_tokens=32).prefill(prompt)
    want = _torch_restatement(cfg, w, prompt)
    np.testing.assert_allclose(got, want, rtol=1e-6, atol=1e-6)


def test_qk_norm_makes_logits_blind_to_the_scale_of_wq_and_wk():
    # per-head RMSNorm of q and k removes any scale of their projections (up to
    # eps and the bf16 rounding of the stored keys): Wq x 2 and Wk x 4 leave the
    # logits unchanged, while without the norms every score grows eightfold
    def run(cfg, w):
        return oracle.OracleModel(cfg, w, max_tokens=32).prefill(gen.make_prompt(cfg, 20, seed=3))[0]

    def rescaled(w, cfg):
        w = dict(w)
        for l in range(cfg.n_layers):
            for name, f in (("wq", 2.0), ("wk", 4.0)):
                v = L.bf16_bits_to_f64(w[f"layers.{l}.{name}"]) * f        # exact in bf16
                w[f"layers.{l}.{name}"] = (v.astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)
        return w

    w = _tiny_weights(TINY_QK)
    base, moved = run(TINY_QK, w), run(TINY_QK, rescaled(w, TINY_QK))
    scale = np.abs(base).max()
    np.testing.assert_allclose(moved, base, rtol=0, atol=2e-3 * scale)
    plain = gen.TINY.with_(name="tiny-qk-off", rope_theta=1e6, rms_eps=1e-6)
    wp = {k: v for k, v in w.items() if "q_norm" not in k and "k_norm" not in k}
    assert np.abs(run(plain, rescaled(wp, plain)) - run(plain, wp)).max() > 5e-2 * scale


def test_qkv_bias_is_added_before_rope():
    cfg = gen.TINY.with_(name="tiny-bias", qkv_bias=True, rope_theta=1e6, rms_eps=1e-6)
    w = gen.make_weights(cfg)
    prompt = gen.make_prompt(cfg, 12, seed=1)
    got, _ = oracle.OracleModel(cfg, w, max_tokens=16).prefill(prompt)
    np.testing.assert_allclose(got, _torch_restatement(cfg, w, prompt), rtol=0, atol=1e-6)


def test_tied_head_uses_the_embedding_table():
    cfg = gen.TINY.with_(name="tiny-tied", tied_embeddings=True)
    w = gen.make_weights(cfg)
    assert "lm_head" not in w
    prompt = gen.make_prompt(cfg, 10, seed=1)
    got, _ = oracle.OracleModel(cfg, w, max_tokens=16).prefill(prompt)
    np.testing.assert_allclose(got, _torch_restatement(cfg, w, prompt), rtol=0, atol=1e-6)


def test_kv_store_rounds_to_bf16_and_capacity_is_checked():
    cfg = gen.TINY
    m = oracle.OracleModel(cfg, _tiny_weights(cfg), max_tokens=8)
    m.prefill(gen.make_prompt(cfg, 8, seed=1))
    k = m.K[0][:, :8, :].astype(np.float64)
    assert np.array_equal(L.round_bf16(k), k)
    with pytest.raises(ValueError):
        m.decode(1)
