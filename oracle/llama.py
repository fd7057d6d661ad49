"""Plain fp64 CPU oracle of the batch-1 Llama-style decoder forward pass.

TEST INFRASTRUCTURE ONLY.  Nothing in the product path may import or call this
module; only `tests/`, `__graft_entry__.smoke()` and the CPU-baseline leg of
`bench.py` use it.  It shares no code with the CUDA path; the only common
input is the byte stream of the seeded generator in `gen/`.

What it computes.  The paper (WiCi, Sec. 3.3 Eq. 1) leaves `T_Local`, the time
for the GPU to produce one token, as the quantity its remoting layer preserves;
the GPU work behind it is llama.cpp's LLM inference (Sec. 1, Sec. 5.1): a
prefill over the prompt whose last position gives the first token (TTFT), then
one forward step per generated token, each step repeating the same computation
with only the input token and its position changing (Sec. 4.2.2, trace replay).
The paper prints no model equations, so the layer is the standard Llama decoder
named by the workload: RMSNorm, rotate-half RoPE, grouped-query causal softmax
attention over a bf16 KV cache, SwiGLU MLP, residual adds, final RMSNorm, LM
head and greedy argmax.  Every point the paper leaves open is decided as below
and listed with the same wording in the design notes:

  * RoPE pairs element i with i + d/2 (rotate-half); angle p * theta^(-2i/d),
    computed in double; no frequency scaling.
  * RMSNorm gains are whatever the weights hold (the synthetic models use 1.0).
  * K (after RoPE) and V are rounded to bf16 (round-to-nearest-even) when they
    are stored; everything else is fp64.  Optional `prefill_act_bf16` rounds the
    activations that feed a prefill matrix product (h, q, o, h2, m) to bf16,
    a diagnostic that isolates operand rounding from errors.
  * QKV bias (Qwen2.5 shape) is added before RoPE; no other biases.
  * Qwen3 block (`qk_norm`): each head of q and of k is RMS-normalised over
    head_dim with its own gain (q_norm, k_norm), after the projection and
    before RoPE.
  * Falcon block (`block == "falcon"`, the Falcon-40B model of Tab. 1; the
    block comes from the public model family, not from the paper): attention
    and MLP both read the same residual stream x, each through its own
    LayerNorm with weight and bias (ln_attn, ln_mlp), and both add to it:
    x + Wo attn(LN_attn(x)) + W_down gelu(W_up LN_mlp(x)); GELU with the
    exact erf; no biases in the matrices; a final LayerNorm with bias.
    LayerNorm uses the biased variance over the hidden axis.
  * Greedy token = argmax of the logits, lowest index on an exact tie.
  * Optional `q8_weights`: matrices in the 8-bit block format (oracle/q8.py)
    replace the bf16 tensors of the same name.

Parity pins for every function are in `tests/test_oracle_pins.py`.
"""
from __future__ import annotations

import numpy as np

# ---------------------------------------------------------------------------
# bf16 storage format (IEEE binary32 with the low 16 mantissa bits dropped)
# ---------------------------------------------------------------------------


def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact value of bf16 bit patterns (np.uint16) as float64."""
    return (np.asarray(bits, np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def round_bf16(x: np.ndarray) -> np.ndarray:
    """Nearest bf16 value to each float64 (ties to even), returned as float64.

    bf16 keeps 7 explicit mantissa bits; float64 keeps 52, so 45 bits are
    rounded off the binary64 pattern directly (one rounding, no detour through
    float32).  Inputs are finite and inside the bf16 normal range here.
    """
    x = np.asarray(x, np.float64)
    u = x.view(np.uint64)
    lsb = (u >> np.uint64(45)) & np.uint64(1)
    u = (u + np.uint64((1 << 44) - 1) + lsb) & ~np.uint64((1 << 45) - 1)
    return u.view(np.float64)


# ---------------------------------------------------------------------------
# layer pieces
# ---------------------------------------------------------------------------


def rmsnorm(x: np.ndarray, g: np.ndarray, eps: float) -> np.ndarray:
    """h = x / sqrt(mean(x^2) + eps) * g over the last axis."""
    ms = np.mean(x * x, axis=-1, keepdims=True)
    return x / np.sqrt(ms + eps) * g


def rope_cos_sin(positions: np.ndarray, head_dim: int, theta: float):
    """cos and sin of the angles p * theta^(-2i/d), i < d/2, shape [len(positions), d/2]."""
    i = np.arange(head_dim // 2, dtype=np.float64)
    freq = theta ** (-2.0 * i / head_dim)
    ang = np.asarray(positions, np.float64)[:, None] * freq[None, :]
    return np.cos(ang), np.sin(ang)


def apply_rope(x: np.ndarray, cos: np.ndarray, sin: np.ndarray) -> np.ndarray:
    """Rotate-half RoPE on x [T, heads, d] with cos/sin [T, d/2]:
    x'_i = x_i cos - x_{i+d/2} sin,  x'_{i+d/2} = x_{i+d/2} cos + x_i sin."""
    half = x.shape[-1] // 2
    a, b = x[..., :half], x[..., half:]
    c, s = cos[:, None, :], sin[:, None, :]
    return np.concatenate([a * c - b * s, b * c + a * s], axis=-1)


def silu(z: np.ndarray) -> np.ndarray:
    """silu(z) = z / (1 + exp(-z))."""
    return z / (1.0 + np.exp(-z))


def layernorm(x: np.ndarray, g: np.ndarray, b: np.ndarray, eps: float) -> np.ndarray:
    """(x - mean(x)) / sqrt(mean((x - mean(x))^2) + eps) * g + b over the last axis."""
    c = x - np.mean(x, axis=-1, keepdims=True)
    var = np.mean(c * c, axis=-1, keepdims=True)
    return c / np.sqrt(var + eps) * g + b


def gelu(z: np.ndarray) -> np.ndarray:
    """gelu(z) = z * Phi(z) = z / 2 * (1 + erf(z / sqrt(2))), with the exact erf."""
    from scipy.special import erf
    return 0.5 * z * (1.0 + erf(z / np.sqrt(2.0)))


def softmax(s: np.ndarray, axis: int = -1) -> np.ndarray:
    """exp(s - max s) / sum exp(s - max s); masked entries carry -inf."""
    m = np.max(s, axis=axis, keepdims=True)
    e = np.exp(s - m)
    return e / np.sum(e, axis=axis, keepdims=True)


def causal_gqa_attention(q: np.ndarray, K: np.ndarray, V: np.ndarray,
                         q_pos: np.ndarray) -> np.ndarray:
    """Causal grouped-query attention.

    q [T, n_q, d] at absolute positions q_pos [T]; K, V [n_kv, S, d] hold the
    cached keys/values of positions 0..S-1.  Query head j reads KV head
    floor(j / (n_q / n_kv)); query t sees keys s <= q_pos[t]:
        o_j[t] = softmax_s(q_j[t] . K_g[s] / sqrt(d)) V_g[s].
    """
    T, n_q, d = q.shape
    n_kv, S, _ = K.shape
    group = n_q // n_kv
    mask = np.arange(S)[None, :] > np.asarray(q_pos)[:, None]          # [T, S] future keys
    out = np.empty((T, n_q, d), np.float64)
    scale = 1.0 / np.sqrt(d)
    for j in range(n_q):
        g = j // group
        s = (q[:, j, :] @ K[g].T) * scale                                # [T, S]
        s[mask] = -np.inf
        out[:, j, :] = softmax(s, axis=-1) @ V[g]
    return out


def greedy(logits: np.ndarray) -> int:
    """argmax, lowest index on an exact tie."""
    return int(np.argmax(logits))


# ---------------------------------------------------------------------------
# the model
# ---------------------------------------------------------------------------


class OracleModel:
    """The decoder over bf16 weight bits (a dict name -> np.uint16 [rows, cols]).

    prefill(tokens) appends tokens at positions kv_len.. and returns the
    last-position logits and greedy token; decode(token) appends one token.
    Both are the same `forward`; decode is the one-token case.
    """

    def __init__(self, cfg, weights: dict, prefill_act_bf16: bool = False,
                 max_tokens: int | None = None, cache_bytes: float = 6e9, q8_weights: dict | None = None):
        self.cfg = cfg
        self.w = weights
        # matrices given in the 8-bit block format ({name: (codes, scales)}) take
        # the place of the bf16 tensors of the same name
        self.q8 = q8_weights or {}
        self.prefill_act_bf16 = prefill_act_bf16
        self._act_round = round_bf16
        self.max_tokens = max_tokens or cfg.total_tokens
        total = sum(v.size for v in weights.values()) * 8
        self._cache = {} if total <= cache_bytes else None
        n_kv, d = cfg.n_kv_heads, cfg.head_dim
        # cached K/V values are bf16-exact, so float32 storage is lossless
        self.K = [np.zeros((n_kv, self.max_tokens, d), np.float32) for _ in range(cfg.n_layers)]
        self.V = [np.zeros((n_kv, self.max_tokens, d), np.float32) for _ in range(cfg.n_layers)]
        self.kv_len = 0

    def reset(self):
        self.kv_len = 0

    def W(self, name: str) -> np.ndarray:
        if self._cache is not None and name in self._cache:
            return self._cache[name]
        if name in self.q8:
            from .q8 import q8_dequantize
            m = q8_dequantize(*self.q8[name])
        else:
            m = bf16_bits_to_f64(self.w[name])
        if self._cache is not None:
            self._cache[name] = m
        return m

    def _vec(self, name: str) -> np.ndarray:
        return self.W(name).reshape(-1)

    def forward(self, tokens, round_act: bool = False, all_rows: bool = False) -> np.ndarray:
        """Run tokens at positions kv_len..kv_len+T-1; return logits [V] of the last
        one, or with `all_rows` the logits [T, V] after every one of them."""
        cfg = self.cfg
        tokens = np.asarray(tokens, np.int64).reshape(-1)
        T, P = len(tokens), self.kv_len
        if P + T > self.max_tokens:
            raise ValueError("KV capacity exceeded")
        H, d, n_q, n_kv = cfg.hidden, cfg.head_dim, cfg.n_q_heads, cfg.n_kv_heads
        rnd = self._act_round if round_act else (lambda a: a)
        pos = np.arange(P, P + T)
        cos, sin = rope_cos_sin(pos, d, cfg.rope_theta)

        x = bf16_bits_to_f64(self.w["embed"][tokens])                  # [T, H]
        falcon = getattr(cfg, "block", "llama") == "falcon"
        for l in range(cfg.n_layers):
            p = f"layers.{l}."
            if falcon:
                x = self._falcon_layer(l, x, T, P, pos, cos, sin, rnd)
                continue
            h = rnd(rmsnorm(x, self._vec(p + "attn_norm"), cfg.rms_eps))
            q = h @ self.W(p + "wq").T
            k = h @ self.W(p + "wk").T
            v = h @ self.W(p + "wv").T
            if cfg.qkv_bias:
                q = q + self._vec(p + "bq")
                k = k + self._vec(p + "bk")
                v = v + self._vec(p + "bv")
            q, k = q.reshape(T, n_q, d), k.reshape(T, n_kv, d)
            if getattr(cfg, "qk_norm", False):
                # Qwen3 block: every head of q and of k RMS-normalised over head_dim
                q = rmsnorm(q, self._vec(p + "q_norm"), cfg.rms_eps)
                k = rmsnorm(k, self._vec(p + "k_norm"), cfg.rms_eps)
            q = apply_rope(q, cos, sin)
            k = apply_rope(k, cos, sin)
            v = v.reshape(T, n_kv, d)
            self.K[l][:, P:P + T, :] = round_bf16(k).transpose(1, 0, 2)
            self.V[l][:, P:P + T, :] = round_bf16(v).transpose(1, 0, 2)
            Kc = self.K[l][:, :P + T, :].astype(np.float64)
            Vc = self.V[l][:, :P + T, :].astype(np.float64)
            o = causal_gqa_attention(rnd(q), Kc, Vc, pos)
            x = x + rnd(o.reshape(T, n_q * d)) @ self.W(p + "wo").T
            h2 = rnd(rmsnorm(x, self._vec(p + "ffn_norm"), cfg.rms_eps))
            m = silu(h2 @ self.W(p + "wg").T) * (h2 @ self.W(p + "wu").T)
            x = x + rnd(m) @ self.W(p + "wd").T
        self.kv_len = P + T
        lm = "embed" if cfg.tied_embeddings else "lm_head"
        if falcon:
            final = lambda a: layernorm(a, self._vec("final_norm"), self._vec("final_norm_b"), cfg.rms_eps)  # noqa: E731
        else:
            final = lambda a: rmsnorm(a, self._vec("final_norm"), cfg.rms_eps)  # noqa: E731
        if all_rows:
            return final(x) @ self.W(lm).T
        return self.W(lm) @ final(x[-1])

    def _falcon_layer(self, l, x, T, P, pos, cos, sin, rnd):
        """One Falcon block: x + Wo attn(LN_attn(x)) + W_down gelu(W_up LN_mlp(x))."""
        cfg = self.cfg
        d, n_q, n_kv = cfg.head_dim, cfg.n_q_heads, cfg.n_kv_heads
        p = f"layers.{l}."
        ha = rnd(layernorm(x, self._vec(p + "ln_attn"), self._vec(p + "ln_attn_b"), cfg.rms_eps))
        hm = rnd(layernorm(x, self._vec(p + "ln_mlp"), self._vec(p + "ln_mlp_b"), cfg.rms_eps))
        q = apply_rope((ha @ self.W(p + "wq").T).reshape(T, n_q, d), cos, sin)
        k = apply_rope((ha @ self.W(p + "wk").T).reshape(T, n_kv, d), cos, sin)
        v = (ha @ self.W(p + "wv").T).reshape(T, n_kv, d)
        self.K[l][:, P:P + T, :] = round_bf16(k).transpose(1, 0, 2)
        self.V[l][:, P:P + T, :] = round_bf16(v).transpose(1, 0, 2)
        Kc = self.K[l][:, :P + T, :].astype(np.float64)
        Vc = self.V[l][:, :P + T, :].astype(np.float64)
        o = causal_gqa_attention(rnd(q), Kc, Vc, pos)
        attn = rnd(o.reshape(T, n_q * d)) @ self.W(p + "wo").T
        mlp = rnd(gelu(hm @ self.W(p + "w_up").T)) @ self.W(p + "w_down").T
        return x + attn + mlp

    def prefill(self, tokens):
        logits = self.forward(tokens, round_act=self.prefill_act_bf16)
        return logits, greedy(logits)

    def decode(self, token: int):
        logits = self.forward([token], round_act=False)
        return logits, greedy(logits)

    def decode_forced(self, tokens) -> np.ndarray:
        """Decode steps fed a known token sequence (teacher forcing), taken as one
        pass: appends the tokens and returns [T, V], whose row t is what
        decode(tokens[t]) would return at that point.  A causal pass over known
        tokens is the same computation as feeding them one at a time (the KV
        cache only ever holds earlier positions)."""
        return self.forward(tokens, round_act=False, all_rows=True)


def run_workload(cfg, weights, prompts, decode_steps: int, **kw):
    """Turns of (prefill prompt, then `decode_steps` greedy steps), each step
    feeding the previous greedy token.  Returns a list of (logits, token) per
    produced position: per turn 1 + decode_steps entries."""
    model = OracleModel(cfg, weights, **kw)
    out = []
    for prompt in prompts:
        logits, tok = model.prefill(prompt)
        out.append((logits, tok))
        for _ in range(decode_steps):
            logits, tok = model.decode(tok)
            out.append((logits, tok))
    return out
