"""GPU parity of the 8-bit block weight format (GGUF-style int8 codes with one
fp16 scale per 32 input columns; the paper's models are GGUF files, Sec. 5.1,
Tab. 1): the CUDA path through the C ABI against the fp64 oracle run with the
same codes and scales (`OracleModel(..., q8_weights=...)`), same rules as the
bf16 parity tests.  Decode streams the codes and scales and converts them in
registers; prefill dequantises each matrix into three exact bf16 terms for the
tensor cores."""
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

# the tiny shape with an FFN width that is a whole number of 256-column groups
TINY_Q8 = gen.TINY.with_(name="tiny-q8", ffn_dim=768)


def _q8_workload(cfg, max_chunk=None, turns=1, page_perm_seed=None, cache_bytes=6e9):
    w = gen.make_weights(cfg)
    q8 = gq.make_q8_weights(cfg)
    assert len(q8) == 7 * cfg.n_layers
    seeds = list(range(1, turns + 1))
    prompts = [gen.make_prompt(cfg, cfg.prompt_len, seed=s) for s in seeds]
    max_tokens = turns * (cfg.prompt_len + cfg.decode_steps)
    model = WiciModel(cfg, max_tokens=max_tokens, max_chunk=max_chunk, q8=True).load(w, q8)
    if page_perm_seed is not None:
        n = (max_tokens + 15) // 16
        wici.wici_set_page_table(model.ctx, np.random.default_rng(page_perm_seed).permutation(n))
    ref = oracle.OracleModel(cfg, w, max_tokens=max_tokens, q8_weights=q8, cache_bytes=cache_bytes)
    stats = {}
    run_teacher_forced(model, ref, prompts, cfg.decode_steps, stats)
    model.close()
    return stats


def test_q8_tiny_workload_matches_oracle():
    stats = _q8_workload(TINY_Q8)
    assert len(stats["max_abs"]) == 1 + TINY_Q8.decode_steps
    assert max(stats["max_abs"]) < 1e-3


def test_q8_tiny_chunked_turns_permuted_pages():
    _q8_workload(TINY_Q8.with_(prompt_len=37, decode_steps=5), max_chunk=16, turns=3, page_perm_seed=5)


def test_q8_llama8b_width_two_layers_ragged_prompt():
    _q8_workload(gen.LLAMA_8B.with_(name="8b-q8-2l", n_layers=2, prompt_len=77, decode_steps=4))


def test_q8_on_device_decode_matches_stepwise_decode():
    cfg = gen.LLAMA_8B.with_(name="8b-q8-2l", n_layers=2, prompt_len=40, decode_steps=6)
    w = gen.make_weights(cfg)
    q8 = gq.make_q8_weights(cfg)
    prompt = gen.make_prompt(cfg, cfg.prompt_len, seed=1)
    model = WiciModel(cfg, max_tokens=64, q8=True).load(w, q8)
    model.prefill(prompt)
    on_device = model.decode(cfg.decode_steps)
    model.reset()
    model.prefill(prompt)
    stepwise = [model.decode_step(-1) for _ in range(cfg.decode_steps)]
    model.close()
    assert list(on_device) == stepwise


def test_q8_rejects_bf16_matrices_and_q8_for_a_bf16_context():
    cfg = TINY_Q8
    w = gen.make_weights(cfg)
    q8 = gq.make_q8_weights(cfg)
    model = WiciModel(cfg, max_tokens=64, q8=True)
    with pytest.raises(wici.WiciError) as e:
        model.load({"layers.0.wq": w["layers.0.wq"]})
    assert e.value.status == wici.WICI_E_ARG
    with pytest.raises(wici.WiciError) as e:
        model.prefill(gen.make_prompt(cfg, 4))            # nothing loaded yet
    assert e.value.status == wici.WICI_E_STATE
    model.close()
    bf = WiciModel(cfg, max_tokens=64)
    with pytest.raises(wici.WiciError) as e:
        wici.wici_load_weights_q8(bf.ctx, [("layers.0.wq",) + q8["layers.0.wq"]])
    assert e.value.status == wici.WICI_E_ARG
    bf.close()


@pytest.mark.slow
def test_q8_llama3_8b_full_depth_full_prompt():
    # the headline shape in the 8-bit format: 32 layers, the 1024-token prompt, then 2 decode steps
    stats = _q8_workload(gen.LLAMA_8B.with_(name="8b-q8", decode_steps=2), max_chunk=1024, cache_bytes=0)
    assert len(stats["max_abs"]) == 3
