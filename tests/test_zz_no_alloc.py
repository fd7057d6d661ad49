"""The allocation-free LM-head entry point (wici_lm_head_argmax_noalloc).

It serves callers that cannot allocate device memory themselves (their device
memory belongs to another engine's pool, or allocation on their thread is not
allowed): they pass inputs and outputs, and the kernel's scratch is a fixed
array inside the library.  Checked through the C ABI against the existing
entry point, wici_prefill, on a model whose layers are all zero, so that the
hidden vector reaching the LM head is exactly the token's embedding row.
This file sorts last so that a run stopping at the first failure has already
run every other test."""
import numpy as np
import pytest

import gen
from tests.parity import check_step

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2608_24204_gb300 import WiciModel, wici  # noqa: E402


def _zero_layer_tiny():
    cfg = gen.TINY
    w = gen.make_weights(cfg)
    for name in list(w):
        if name.startswith("layers.") and not name.endswith("norm"):
            w[name] = np.zeros_like(w[name])
    return cfg, w


def test_no_alloc_lm_head_matches_prefill_twice_in_a_row():
    cfg, w = _zero_layer_tiny()
    model = WiciModel(cfg, max_tokens=8).load(w)
    dev = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).cuda()  # noqa: E731
    lm = dev(w["lm_head"])
    gain = dev(w["final_norm"])
    stream = torch.cuda.current_stream()
    for tok in (517, 3):                       # two calls in a row share the scratch
        model.reset()
        want, want_tok = model.prefill(np.array([tok], np.int32), logits=True)
        x = torch.from_numpy((w["embed"][tok].astype(np.uint32) << 16).view(np.float32)).cuda()
        logits = torch.full((cfg.vocab,), float("nan"), dtype=torch.float32, device="cuda")
        token = torch.full((1,), -1, dtype=torch.int32, device="cuda")
        wici.wici_lm_head_argmax_noalloc(stream.cuda_stream, lm.data_ptr(), gain.data_ptr(), x.data_ptr(),
                                         cfg.hidden, cfg.vocab, cfg.rms_eps, logits.data_ptr(), token.data_ptr())
        torch.cuda.synchronize()
        got = logits.cpu().numpy()
        check_step(got, int(token.item()), want, want_tok, f"no-alloc head, token {tok}")
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
