"""Two tenants on one GPU (the paper's two-client microbenchmark, Sec. 5.4, and
its task-scheduling discussion, Sec. 7): two contexts with different models,
each given an SM share (wici_config.max_sms) so that both persistent decode
grids are resident at once, each on its own stream with its own priority.

  * interleaved, teacher-forced steps of both tenants match their oracles;
  * greedy decode run by two host threads at the same time gives each tenant
    exactly the tokens it gives when it runs alone."""
import threading

import numpy as np
import pytest

import gen
import oracle
from tests.parity import check_step

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2608_24204_gb300 import WiciModel  # noqa: E402

SMALL = gen.LLAMA_1B.with_(name="1b-2l", n_layers=2, prompt_len=48, decode_steps=6)
LARGE = gen.LLAMA_8B.with_(name="8b-2l", n_layers=2, prompt_len=40, decode_steps=6)


def _shares():
    nsm = torch.cuda.get_device_properties(0).multi_processor_count
    small = max(8, nsm // 4)
    return small, nsm - small


def _tenant(cfg, share, priority, max_tokens=128):
    stream = torch.cuda.Stream(priority=priority)
    w = gen.make_weights(cfg)
    return WiciModel(cfg, max_tokens=max_tokens, stream=stream, max_sms=share).load(w), w


def test_two_tenants_interleaved_steps_match_their_oracles():
    s_small, s_large = _shares()
    lo, hi = 0, -1                            # CUDA stream priorities: lower is more urgent
    a, wa = _tenant(SMALL, s_small, hi)       # the small model's client gets the higher priority
    b, wb = _tenant(LARGE, s_large, lo)
    ra = oracle.OracleModel(SMALL, wa, max_tokens=128)
    rb = oracle.OracleModel(LARGE, wb, max_tokens=128)
    pa = gen.make_prompt(SMALL, SMALL.prompt_len, seed=1)
    pb = gen.make_prompt(LARGE, LARGE.prompt_len, seed=2)
    stats = {}
    want_a, ta = ra.prefill(pa)
    want_b, tb = rb.prefill(pb)
    got_a, ga = a.prefill(pa, logits=True)
    got_b, gb = b.prefill(pb, logits=True)
    check_step(got_a, ga, want_a, ta, "tenant A prefill", stats)
    check_step(got_b, gb, want_b, tb, "tenant B prefill", stats)
    for s in range(SMALL.decode_steps):
        fa, fb = ta, tb
        want_a, ta = ra.decode(fa)
        want_b, tb = rb.decode(fb)
        got_a, ga = a.decode_step(fa, logits=True)
        got_b, gb = b.decode_step(fb, logits=True)
        check_step(got_a, ga, want_a, ta, f"tenant A step {s}", stats)
        check_step(got_b, gb, want_b, tb, f"tenant B step {s}", stats)
    a.close()
    b.close()


def test_two_tenants_decoding_concurrently_give_their_solo_tokens():
    s_small, s_large = _shares()
    a, _ = _tenant(SMALL, s_small, -1, max_tokens=256)
    b, _ = _tenant(LARGE, s_large, 0, max_tokens=256)
    pa = gen.make_prompt(SMALL, SMALL.prompt_len, seed=1)
    pb = gen.make_prompt(LARGE, LARGE.prompt_len, seed=2)
    n = 96

    def solo(m, p):
        m.reset()
        m.prefill(p)
        return m.decode(n)

    alone_a, alone_b = solo(a, pa), solo(b, pb)
    for m, p in ((a, pa), (b, pb)):
        m.reset()
        m.prefill(p)
    out = {}

    def run(key, m):
        out[key] = m.decode(n)

    threads = [threading.Thread(target=run, args=("a", a)), threading.Thread(target=run, args=("b", b))]
    for t in threads:
        t.start()
    for t in threads:
        t.join()
    np.testing.assert_array_equal(out["a"], alone_a)
    np.testing.assert_array_equal(out["b"], alone_b)
    a.close()
    b.close()
