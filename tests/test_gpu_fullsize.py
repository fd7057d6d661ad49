"""Full-size parity: the configurations at their real widths, depths and prompt
lengths, in the launch configuration the benchmark times (one prefill of the
whole prompt, then captured-graph decode steps), against the fp64 oracle.
The oracle recomputes every compared logits vector itself; decode is sampled
to a few steps because each oracle step streams the whole model on the CPU."""
import numpy as np
import pytest

import gen
import oracle
from tests.parity import run_teacher_forced

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2608_24204_gb300 import WiciModel  # noqa: E402


def _full(cfg, decode_steps, max_chunk=None):
    w = gen.make_weights(cfg)
    prompt = gen.make_prompt(cfg, cfg.prompt_len, seed=1)
    max_tokens = cfg.prompt_len + decode_steps + 16
    model = WiciModel(cfg, max_tokens=max_tokens, max_chunk=max_chunk or cfg.prompt_len).load(w)
    ref = oracle.OracleModel(cfg, w, max_tokens=max_tokens, cache_bytes=0)
    stats = {}
    run_teacher_forced(model, ref, [prompt], decode_steps, stats)
    model.close()
    return stats


def test_llama3_8b_shape_bench_launch_configuration():
    stats = _full(gen.LLAMA_8B, decode_steps=3)
    assert len(stats["max_abs"]) == 4


def test_llama32_1b_shape_full_prompt():
    stats = _full(gen.LLAMA_1B, decode_steps=8)
    assert len(stats["max_abs"]) == 9


def test_qwen25_14b_shape_full_prompt():
    # the deepest config: 48 layers, a 2048-token prompt, then one decode step
    stats = _full(gen.QWEN_14B, decode_steps=1)
    assert len(stats["max_abs"]) == 2
