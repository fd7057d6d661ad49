"""GPU parity of the Qwen3 block (the paper's evaluated family, Sec. 5.1, Tab. 1):
the Llama block plus a per-head RMSNorm of q and of k (own gains) before RoPE.
Decode finishes q and the new key inside the attention phase; prefill runs a
per-(token, head) norm + RoPE kernel after the QKV GEMM.  Checked against the
fp64 oracle with the parity rules of tests/parity.py, in bf16 and in the 8-bit
block format (the paper's Qwen-8B-GGUF is a block-quantised Qwen3-8B)."""
import numpy as np
import pytest

import gen
import oracle
from gen import q8 as gq
from tests.parity import run_teacher_forced

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2608_24204_gb300 import WiciModel, wici  # noqa: E402

TINY_QK = gen.TINY.with_(name="tiny-qk", qk_norm=True, rope_theta=1e6, rms_eps=1e-6, ffn_dim=768)


def _workload(cfg, q8=False, max_chunk=None, turns=1, page_perm_seed=None, cache_bytes=6e9):
    w = gen.make_weights(cfg)
    q8w = gq.make_q8_weights(cfg) if q8 else None
    prompts = [gen.make_prompt(cfg, cfg.prompt_len, seed=s) for s in range(1, turns + 1)]
    max_tokens = turns * (cfg.prompt_len + cfg.decode_steps)
    model = WiciModel(cfg, max_tokens=max_tokens, max_chunk=max_chunk, q8=q8).load(w, q8w)
    if page_perm_seed is not None:
        n = (max_tokens + 15) // 16
        wici.wici_set_page_table(model.ctx, np.random.default_rng(page_perm_seed).permutation(n))
    ref = oracle.OracleModel(cfg, w, max_tokens=max_tokens, q8_weights=q8w, cache_bytes=cache_bytes)
    stats = {}
    run_teacher_forced(model, ref, prompts, cfg.decode_steps, stats)
    model.close()
    return stats


def test_qk_norm_tiny_workload_matches_oracle():
    stats = _workload(TINY_QK)
    assert max(stats["max_abs"]) < 1e-3


def test_qk_norm_tiny_chunked_turns_permuted_pages():
    _workload(TINY_QK.with_(prompt_len=29, decode_steps=5), max_chunk=8, turns=3, page_perm_seed=11)


def test_qwen3_8b_width_two_layers_ragged_prompt():
    _workload(gen.QWEN3_8B.with_(name="qwen3-8b-2l", n_layers=2, prompt_len=93, decode_steps=5))


def test_qwen3_8b_width_two_layers_chunked_turns():
    _workload(gen.QWEN3_8B.with_(name="qwen3-8b-2l", n_layers=2, prompt_len=150, decode_steps=4), max_chunk=64,
              turns=2)


def test_qwen3_8b_width_two_layers_in_the_8bit_format():
    _workload(gen.QWEN3_8B.with_(name="qwen3-8b-q8-2l", n_layers=2, prompt_len=70, decode_steps=5), q8=True)


@pytest.mark.slow
def test_qwen3_8b_full_depth_full_prompt():
    # 36 layers, the 1024-token prompt, then 2 decode steps, bf16
    stats = _workload(gen.QWEN3_8B.with_(decode_steps=2), max_chunk=1024, cache_bytes=0)
    assert len(stats["max_abs"]) == 3


@pytest.mark.slow
def test_qwen3_8b_full_depth_in_the_8bit_format():
    # the paper's Qwen-8B-GGUF analogue: every layer matrix in the 8-bit block format
    stats = _workload(gen.QWEN3_8B.with_(decode_steps=2), q8=True, max_chunk=1024, cache_bytes=0)
    assert len(stats["max_abs"]) == 3
