"""GPU parity: the CUDA path through the C ABI against the CPU oracle on the
same seeded inputs (gpu-marked; run on a GB300)."""
import numpy as np
import pytest

import gen
import oracle
from tests.parity import check_step, run_teacher_forced

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2608_24204_gb300 import WiciModel, wici  # noqa: E402

_weights_cache = {}


def weights(cfg):
    if cfg not in _weights_cache:
        _weights_cache.clear()
        _weights_cache[cfg] = gen.make_weights(cfg)
    return _weights_cache[cfg]


def _workload(cfg, max_chunk=None, page_perm_seed=None, turns=None):
    w = weights(cfg)
    turns = turns or cfg.turns
    seeds = list(cfg.prompt_seeds) + list(range(len(cfg.prompt_seeds) + 1, turns + 1))
    prompts = [gen.make_prompt(cfg, cfg.prompt_len, seed=s) for s in seeds[:turns]]
    max_tokens = turns * (cfg.prompt_len + cfg.decode_steps)
    model = WiciModel(cfg, max_tokens=max_tokens, max_chunk=max_chunk).load(w)
    if page_perm_seed is not None:
        n = (max_tokens + 15) // 16
        wici.wici_set_page_table(model.ctx, np.random.default_rng(page_perm_seed).permutation(n))
    ref = oracle.OracleModel(cfg, w, max_tokens=max_tokens)
    stats = {}
    run_teacher_forced(model, ref, prompts, cfg.decode_steps, stats)
    model.close()
    return stats


def test_tiny_workload_matches_oracle():
    stats = _workload(gen.TINY)
    assert len(stats["max_abs"]) == 1 + gen.TINY.decode_steps
    assert max(stats["max_abs"]) < 1e-3


def test_tiny_chunked_prefill_and_permuted_pages():
    _workload(gen.TINY.with_(name="tiny-turns", turns=3, prompt_len=21, decode_steps=5),
              max_chunk=8, page_perm_seed=3)


def test_llama1b_width_two_layers():
    _workload(gen.LLAMA_1B.with_(name="1b-2l", n_layers=2, prompt_len=64, decode_steps=6))


def test_llama8b_width_two_layers_ragged_prompt():
    _workload(gen.LLAMA_8B.with_(name="8b-2l", n_layers=2, prompt_len=77, decode_steps=4))


def test_qwen14b_width_two_layers_bias_group5():
    _workload(gen.QWEN_14B.with_(name="14b-2l", n_layers=2, prompt_len=50, decode_steps=4))


def test_agentic_turns_two_layers_chunked():
    cfg = gen.LLAMA_8B_AGENTIC.with_(name="agentic-2l", n_layers=2, prompt_len=300, decode_steps=6, turns=3,
                                     prompt_seeds=(1, 2, 3))
    _workload(cfg, max_chunk=128)


def test_agentic_long_context_two_layers():
    # past 2048 cached tokens the flash-decode splits hold more pages than its ring
    cfg = gen.LLAMA_8B_AGENTIC.with_(name="agentic-long-2l", n_layers=2, prompt_len=1100, decode_steps=4, turns=2,
                                     prompt_seeds=(1, 2))
    _workload(cfg, max_chunk=512)


def _tiny_model(max_tokens=64, **kw):
    cfg = gen.TINY
    return cfg, WiciModel(cfg, max_tokens=max_tokens, **kw).load(weights(cfg))


def test_reset_rerun_is_bit_identical_and_page_table_is_transparent():
    cfg, m = _tiny_model()
    prompt = gen.make_prompt(cfg, 20, seed=1)
    a, t = m.prefill(prompt, logits=True)
    a2, _ = m.decode_step(t, logits=True)
    m.reset()
    assert m.kv_len == 0
    b, _ = m.prefill(prompt, logits=True)
    b2, _ = m.decode_step(t, logits=True)
    assert np.array_equal(a, b) and np.array_equal(a2, b2)
    m.reset()
    wici.wici_set_page_table(m.ctx, np.arange(4)[::-1].copy())
    c, _ = m.prefill(prompt, logits=True)
    c2, _ = m.decode_step(t, logits=True)
    assert np.array_equal(a, c) and np.array_equal(a2, c2)
    m.close()


def test_on_device_decode_matches_stepwise_decode():
    cfg, m = _tiny_model()
    prompt = gen.make_prompt(cfg, 16, seed=2)
    t0 = m.prefill(prompt)
    steps = [m.decode_step()]
    for _ in range(9):
        steps.append(m.decode_step())
    m.reset()
    assert m.prefill(prompt) == t0
    toks = m.decode(10)
    assert list(toks) == steps
    assert m.kv_len == 16 + 10
    m.close()


def test_error_codes_and_state_preservation():
    cfg, m = _tiny_model(max_tokens=40)
    L = wici.lib()
    with pytest.raises(wici.WiciError) as e:
        m.decode_step()
    assert e.value.status == wici.WICI_E_STATE
    with pytest.raises(wici.WiciError) as e:
        m.prefill(np.array([0, cfg.vocab], np.int32))
    assert e.value.status == wici.WICI_E_ARG
    assert L.wici_prefill(m.ctx, None, 0, None, None) == wici.WICI_E_ARG
    prompt = gen.make_prompt(cfg, 30, seed=1)
    a, t = m.prefill(prompt, logits=True)
    with pytest.raises(wici.WiciError) as e:
        m.prefill(np.zeros(11, np.int32))                      # 30 + 11 > 40
    assert e.value.status == wici.WICI_E_CAPACITY
    assert m.kv_len == 30
    with pytest.raises(wici.WiciError) as e:
        m.decode(11)
    assert e.value.status == wici.WICI_E_CAPACITY
    assert m.kv_len == 30
    with pytest.raises(wici.WiciError) as e:
        wici.wici_set_page_table(m.ctx, np.arange(5))          # 40 tokens need 3 pages
    assert e.value.status == wici.WICI_E_ARG
    with pytest.raises(wici.WiciError) as e:
        wici.wici_set_page_table(m.ctx, np.arange(3))          # right length, but tokens are cached
    assert e.value.status == wici.WICI_E_STATE
    # the context still produces the same continuation after the rejected calls
    ref = oracle.OracleModel(cfg, weights(cfg), max_tokens=40)
    want, wt = ref.prefill(prompt)
    check_step(a, t, want, wt, "prefill")
    want, wt2 = ref.decode(wt)
    got, gt = m.decode_step(wt, logits=True)
    check_step(got, gt, want, wt2, "after errors")
    m.close()


def test_weights_must_be_loaded_and_names_checked():
    cfg = gen.TINY
    m = WiciModel(cfg, max_tokens=32)
    with pytest.raises(wici.WiciError) as e:
        m.prefill(np.array([1, 2, 3], np.int32))
    assert e.value.status == wici.WICI_E_STATE
    w = weights(cfg)
    with pytest.raises(wici.WiciError) as e:
        wici.wici_load_weights(m.ctx, [("layers.9.wq", w["layers.0.wq"], 256, 256)])
    assert e.value.status == wici.WICI_E_ARG
    with pytest.raises(wici.WiciError) as e:
        wici.wici_load_weights(m.ctx, [("layers.0.wq", w["layers.0.wk"], 128, 256)])
    assert e.value.status == wici.WICI_E_ARG
    m.close()


def test_bounded_wait_gives_up_and_context_stays_usable():
    st = torch.cuda.current_stream().cuda_stream
    assert wici.wici_check_bounded_wait(st, 2_000_000) == wici.WICI_E_TIMEOUT
    cfg, m = _tiny_model()
    t = m.prefill(gen.make_prompt(cfg, 8, seed=1))
    assert 0 <= m.decode_step(t) < cfg.vocab
    m.close()


def test_device_weights_load_like_host_weights():
    cfg = gen.TINY
    w = weights(cfg)
    a = WiciModel(cfg, max_tokens=32).load(w)
    b = WiciModel(cfg, max_tokens=32)
    dev = {k: torch.from_numpy(v.view(np.int16)).cuda() for k, v in w.items()}
    wici.wici_load_weights(b.ctx, [(k, (t.data_ptr(), 1), *t.shape) for k, t in dev.items()])
    prompt = gen.make_prompt(cfg, 12, seed=4)
    la, _ = a.prefill(prompt, logits=True)
    lb, _ = b.prefill(prompt, logits=True)
    assert np.array_equal(la, lb)
    a.close()
    b.close()


def test_multi_launch_decode_path_when_query_width_differs_from_hidden():
    # 8 query heads x 64 = 512 != hidden 256: the decode step runs as one launch per
    # layer operation (QKV, attention, O, gate/up, down) instead of the persistent kernel
    cfg = gen.TINY.with_(name="tiny-wideq", n_q_heads=8, decode_steps=6)
    _workload(cfg)
