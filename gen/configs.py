"""Model shapes and workloads of the five synthetic decoder configurations.

These are workload descriptions only (shapes, seeds, lengths); no arithmetic of
the forward pass lives here.  The paper evaluates llama.cpp inference on
Qwen3/Falcon GGUF models (Sec. 5.1, Tab. 1) without giving their internals, so
the shapes are the standard Llama-3 / Qwen2.5 ones with seeded random bf16
weights ~N(0, 0.02) and all RMSNorm gains equal to 1.
"""
from __future__ import annotations

from dataclasses import dataclass, field, replace


@dataclass(frozen=True)
class ModelConfig:
    name: str
    n_layers: int
    hidden: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    ffn_dim: int
    vocab: int
    rope_theta: float
    rms_eps: float = 1e-5
    tied_embeddings: bool = False
    qkv_bias: bool = False
    qk_norm: bool = False          # Qwen3 block: per-head RMSNorm of q and k before RoPE
    # "llama": sequential attention then SwiGLU MLP, RMSNorm; "falcon": Falcon-40B's
    # parallel attention and GELU MLP, each after its own LayerNorm (weight and bias)
    block: str = "llama"
    weight_std: float = 0.02
    weight_seed: int = 0
    # workload: `turns` rounds of (prompt_len-token chunk, then decode_steps greedy tokens)
    prompt_len: int = 32
    decode_steps: int = 16
    turns: int = 1
    prompt_seeds: tuple = (1,)
    max_chunk: int = 2048
    page_tokens: int = 16
    extra: dict = field(default_factory=dict, compare=False)

    @property
    def q_dim(self) -> int:
        return self.n_q_heads * self.head_dim

    @property
    def kv_dim(self) -> int:
        return self.n_kv_heads * self.head_dim

    @property
    def total_tokens(self) -> int:
        return self.turns * (self.prompt_len + self.decode_steps)

    def with_(self, **kw) -> "ModelConfig":
        return replace(self, **kw)


TINY = ModelConfig(
    name="tiny", n_layers=2, hidden=256, n_q_heads=4, n_kv_heads=2, head_dim=64,
    ffn_dim=688, vocab=1024, rope_theta=10000.0, rms_eps=1e-5,
    prompt_len=32, decode_steps=16)

LLAMA_1B = ModelConfig(
    name="llama3.2-1b", n_layers=16, hidden=2048, n_q_heads=32, n_kv_heads=8, head_dim=64,
    ffn_dim=8192, vocab=128256, rope_theta=500000.0, rms_eps=1e-5, tied_embeddings=True,
    prompt_len=512, decode_steps=128)

LLAMA_8B = ModelConfig(
    name="llama3-8b", n_layers=32, hidden=4096, n_q_heads=32, n_kv_heads=8, head_dim=128,
    ffn_dim=14336, vocab=128256, rope_theta=500000.0, rms_eps=1e-5,
    prompt_len=1024, decode_steps=256)

LLAMA_8B_AGENTIC = LLAMA_8B.with_(
    name="llama3-8b-agentic", prompt_len=2048, decode_steps=64, turns=4,
    prompt_seeds=(1, 2, 3, 4))

QWEN_14B = ModelConfig(
    name="qwen2.5-14b", n_layers=48, hidden=5120, n_q_heads=40, n_kv_heads=8, head_dim=128,
    ffn_dim=13824, vocab=152064, rope_theta=1000000.0, rms_eps=1e-6, qkv_bias=True,
    prompt_len=2048, decode_steps=256)

# The paper's headline model family (Qwen3, Tab. 1) at the 8B shape: the Llama
# block plus a per-head RMSNorm of q and k before RoPE, no QKV bias, untied.
QWEN3_8B = ModelConfig(
    name="qwen3-8b", n_layers=36, hidden=4096, n_q_heads=32, n_kv_heads=8, head_dim=128,
    ffn_dim=12288, vocab=151936, rope_theta=1000000.0, rms_eps=1e-6, qk_norm=True,
    prompt_len=1024, decode_steps=256)

# The paper's largest evaluated model (Falcon-40B, Tab. 1): the Falcon block of
# the public model family (parallel attention and MLP from one residual stream,
# two LayerNorms per layer, a 4H GELU MLP, 128 query / 8 KV heads of 64,
# rotate-half RoPE, tied embeddings), and a two-layer stand-in for the pins.
FALCON_40B = ModelConfig(
    name="falcon-40b", n_layers=60, hidden=8192, n_q_heads=128, n_kv_heads=8, head_dim=64,
    ffn_dim=32768, vocab=65024, rope_theta=10000.0, rms_eps=1e-5, tied_embeddings=True,
    block="falcon", prompt_len=1024, decode_steps=256)

FALCON_TINY = FALCON_40B.with_(
    name="falcon-tiny", n_layers=2, hidden=256, n_q_heads=8, n_kv_heads=2, head_dim=32,
    ffn_dim=1024, vocab=1024, prompt_len=32, decode_steps=16)

CONFIGS = {c.name: c for c in (TINY, LLAMA_1B, LLAMA_8B, LLAMA_8B_AGENTIC, QWEN_14B, QWEN3_8B, FALCON_TINY,
                               FALCON_40B)}


def tensor_specs(cfg: ModelConfig):
    """Canonical tensor list: (name, (rows, cols), kind) with kind 'normal', 'ones'
    or 'gain' (1 + 0.25 N(0, 1): the per-head q/k norm gains and the Falcon
    LayerNorm weights, not all one).

    The position of a tensor in this list is its generator tag.  All matrices
    are row-major [out, in]; y = W x.
    """
    H, d = cfg.hidden, cfg.head_dim
    if cfg.block == "falcon":
        return _falcon_specs(cfg)
    specs = [("embed", (cfg.vocab, H), "normal")]
    for l in range(cfg.n_layers):
        p = f"layers.{l}."
        specs.append((p + "attn_norm", (1, H), "ones"))
        specs.append((p + "wq", (cfg.n_q_heads * d, H), "normal"))
        specs.append((p + "wk", (cfg.n_kv_heads * d, H), "normal"))
        specs.append((p + "wv", (cfg.n_kv_heads * d, H), "normal"))
        if cfg.qkv_bias:
            specs.append((p + "bq", (1, cfg.n_q_heads * d), "normal"))
            specs.append((p + "bk", (1, cfg.n_kv_heads * d), "normal"))
            specs.append((p + "bv", (1, cfg.n_kv_heads * d), "normal"))
        if cfg.qk_norm:
            specs.append((p + "q_norm", (1, d), "gain"))
            specs.append((p + "k_norm", (1, d), "gain"))
        specs.append((p + "wo", (H, cfg.n_q_heads * d), "normal"))
        specs.append((p + "ffn_norm", (1, H), "ones"))
        specs.append((p + "wg", (cfg.ffn_dim, H), "normal"))
        specs.append((p + "wu", (cfg.ffn_dim, H), "normal"))
        specs.append((p + "wd", (H, cfg.ffn_dim), "normal"))
    specs.append(("final_norm", (1, H), "ones"))
    if not cfg.tied_embeddings:
        specs.append(("lm_head", (cfg.vocab, H), "normal"))
    return specs


def _falcon_specs(cfg: ModelConfig):
    """Falcon block: per layer a LayerNorm (weight ln_attn, bias ln_attn_b) for the
    attention branch and one (ln_mlp, ln_mlp_b) for the MLP branch, no biases in
    the matrices; MLP w_up [F, H], w_down [H, F]; a final LayerNorm."""
    H, d = cfg.hidden, cfg.head_dim
    specs = [("embed", (cfg.vocab, H), "normal")]
    for l in range(cfg.n_layers):
        p = f"layers.{l}."
        specs.append((p + "ln_attn", (1, H), "gain"))
        specs.append((p + "ln_attn_b", (1, H), "normal"))
        specs.append((p + "ln_mlp", (1, H), "gain"))
        specs.append((p + "ln_mlp_b", (1, H), "normal"))
        specs.append((p + "wq", (cfg.n_q_heads * d, H), "normal"))
        specs.append((p + "wk", (cfg.n_kv_heads * d, H), "normal"))
        specs.append((p + "wv", (cfg.n_kv_heads * d, H), "normal"))
        specs.append((p + "wo", (H, cfg.n_q_heads * d), "normal"))
        specs.append((p + "w_up", (cfg.ffn_dim, H), "normal"))
        specs.append((p + "w_down", (H, cfg.ffn_dim), "normal"))
    specs.append(("final_norm", (1, H), "gain"))
    specs.append(("final_norm_b", (1, H), "normal"))
    if not cfg.tied_embeddings:
        specs.append(("lm_head", (cfg.vocab, H), "normal"))
    return specs


Q8_LAYER_MATRICES = ("wq", "wk", "wv", "wo", "wg", "wu", "wd", "w_up", "w_down")


def decode_bytes_per_token(cfg: ModelConfig, ctx: int, q8: bool = False) -> int:
    """Algorithmic HBM bytes one decode step must read: every weight once plus
    the K and V of `ctx` cached positions (bf16).  With `q8` the per-layer
    matrices whose input width is a whole number of 32-blocks are in the 8-bit
    block format: 1 byte per code plus a 2-byte scale per 32 (17/16 bytes per
    parameter); everything else stays bf16."""
    n = 0.0
    for name, (r, c), _ in tensor_specs(cfg):
        if name == "embed":
            n += 2 * cfg.hidden            # one embedding row is gathered
        elif q8 and name.split(".")[-1] in Q8_LAYER_MATRICES and c % 32 == 0:
            n += r * c * 17 / 16
        else:
            n += 2 * r * c
    if cfg.tied_embeddings:
        n += 2 * cfg.vocab * cfg.hidden    # the LM head reads the (shared) embedding table
    return int(n) + cfg.n_layers * 2 * cfg.kv_dim * 2 * ctx


def prefill_flops(cfg: ModelConfig, T: int, P: int = 0) -> float:
    """Algorithmic FLOPs of a T-token prefill appended after P cached tokens:
    2*T*(per-layer linear params)*L + causal attention (unmasked pairs only,
    QK^T and PV) + the LM head on the last row."""
    H, d = cfg.hidden, cfg.head_dim
    mlp = (2 if cfg.block == "falcon" else 3) * H * cfg.ffn_dim     # GELU: up, down; SwiGLU: gate, up, down
    lin = H * (cfg.q_dim + 2 * cfg.kv_dim) + cfg.q_dim * H + mlp
    pairs = T * P + T * (T + 1) // 2
    attn = cfg.n_q_heads * d * 4 * pairs
    return float(2 * T * lin * cfg.n_layers + attn * cfg.n_layers + 2 * cfg.vocab * H)
