"""The allocation-free LM-head entry point (wici_lm_head_argmax_noalloc).

It serves callers that cannot allocate device memory themselves (their device
memory belongs to another engine's pool, or allocation on their thread is not
allowed): they pass inputs and outputs, and the kernel's scratch is a fixed
array inside the library.

Checked through the C ABI in two ways:
  * against the fp64 oracle (final RMSNorm with a non-unit gain, then the bf16
    head, then greedy) on seeded random hidden vectors, two calls in a row that
    share the scratch, with a vocabulary that is not a multiple of the grid and
    one smaller than the SM count;
  * bit for bit against the LM head that wici_prefill runs, on a model whose
    layers are all zero (the hidden vector reaching the head is then exactly
    the token's embedding row): each row's reduction order does not depend on
    the grid, so the two must agree exactly.
This file sorts last so that a run stopping at the first failure has already
run every other test."""
import numpy as np
import pytest

import gen
import oracle
from tests.parity import check_step

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2608_24204_gb300 import WiciModel, wici  # noqa: E402


def _dev(bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).cuda()


def _bf16_bits(values):
    return (np.asarray(values, np.float32).view(np.uint32) >> 16).astype(np.uint16)


def _noalloc(lm, gain, x, hidden, vocab, eps):
    logits = torch.full((vocab,), float("nan"), dtype=torch.float32, device="cuda")
    token = torch.full((1,), -2, dtype=torch.int32, device="cuda")
    wici.wici_lm_head_argmax_noalloc(torch.cuda.current_stream().cuda_stream, lm.data_ptr(), gain.data_ptr(),
                                     x.data_ptr(), hidden, vocab, eps, logits.data_ptr(), token.data_ptr())
    torch.cuda.synchronize()
    return logits.cpu().numpy(), int(token.item())


def test_no_alloc_lm_head_matches_oracle_on_random_hidden_vectors():
    cfg = gen.TINY
    H = cfg.hidden
    lm_bits = gen.make_tensor(cfg, "lm_head")                                   # [1024, 256]
    # a non-unit final-norm gain, exact in bf16
    gain_bits = _bf16_bits(oracle.round_bf16(1.0 + 0.25 * gen.normal_f64(7, 1, H)))
    lm, gain = _dev(lm_bits), _dev(gain_bits)
    nsm = torch.cuda.get_device_properties(0).multi_processor_count
    for call, vocab in enumerate((cfg.vocab, 100, cfg.vocab)):   # 1024 % 152 != 0; 100 < the SM count
        assert vocab < nsm or vocab % nsm != 0
        x = (3.0 * gen.normal_f64(11, call, H)).astype(np.float32)
        h = oracle.rmsnorm(x.astype(np.float64), oracle.bf16_bits_to_f64(gain_bits), cfg.rms_eps)
        want = oracle.bf16_bits_to_f64(lm_bits[:vocab]) @ h
        got, tok = _noalloc(lm, gain, torch.from_numpy(x).cuda(), H, vocab, cfg.rms_eps)
        assert tok >= 0, "a bounded device wait gave up"
        check_step(got, tok, want, oracle.greedy(want), f"no-alloc head, call {call}, vocab {vocab}")


def test_no_alloc_lm_head_is_bit_identical_to_the_prefill_head():
    cfg = gen.TINY
    w = gen.make_weights(cfg)
    for name in list(w):
        if name.startswith("layers.") and not name.endswith("norm"):
            w[name] = np.zeros_like(w[name])
    model = WiciModel(cfg, max_tokens=8).load(w)
    lm, gain = _dev(w["lm_head"]), _dev(w["final_norm"])
    for tok in (517, 3):                       # two calls in a row share the scratch
        model.reset()
        want, want_tok = model.prefill(np.array([tok], np.int32), logits=True)
        x = torch.from_numpy((w["embed"][tok].astype(np.uint32) << 16).view(np.float32)).cuda()
        got, got_tok = _noalloc(lm, gain, x, cfg.hidden, cfg.vocab, cfg.rms_eps)
        assert got_tok == want_tok
        np.testing.assert_array_equal(got, want)
    model.close()


def test_no_alloc_lm_head_rejects_sizes_beyond_its_limits():
    z = torch.zeros(16, dtype=torch.float32, device="cuda")
    p = z.data_ptr()
    s = torch.cuda.current_stream().cuda_stream
    with pytest.raises(wici.WiciError) as e:
        wici.wici_lm_head_argmax_noalloc(s, p, p, p, 16392, 4, 1e-5, p, p)
    assert e.value.status == wici.WICI_E_ARG and "hidden" in str(e.value)
    with pytest.raises(wici.WiciError) as e:
        wici.wici_lm_head_argmax_noalloc(s, p, p, p, 12, 4, 1e-5, p, p)
    assert e.value.status == wici.WICI_E_ARG
