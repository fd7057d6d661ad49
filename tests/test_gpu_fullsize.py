"""Full-size parity: the configurations at their real widths, depths and prompt
lengths, in the launch configuration the benchmark times (one prefill per
chunk, then captured-graph decode steps), against the fp64 oracle.

The Llama-3-8B request (64 and all 256 decode steps), the agentic workload
and the Llama-3.2-1B request (all 128 of its decode steps) are compared with
oracle records stored under tests/golden/ (written by make_fullsize_golden.py, which
runs only the oracle): every decode step is teacher-forced with the record's
seeded tokens through `token_in`, and every produced logits vector is compared,
in full at the recorded positions and at 1024 fixed sample indices plus the
oracle's 8 largest entries everywhere else.  The 1B and 14B shapes recompute
the oracle on the fly; their decode is sampled to a few steps because each
oracle step streams the whole model on the CPU."""
import os

import numpy as np
import pytest

import gen
import oracle
from tests.parity import MAX_ABS, NEAR_TIE, REL_L2, check_step, run_teacher_forced

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2608_24204_gb300 import WiciModel  # noqa: E402

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
_weights = {}


def _weights_of(cfg):
    key = tuple(gen.tensor_specs(cfg))          # configs of one shape share their weights
    if key not in _weights:
        _weights.clear()
        _weights[key] = gen.make_weights(cfg)
    return _weights[key]


def _check_sampled(got, got_tok, rec, t, p, where, stats):
    """max-abs over the sample indices and the oracle's top entries, rel-L2 over
    the sample indices, and the token rule with the recorded top-2 gap."""
    got = np.asarray(got, np.float64)
    assert np.all(np.isfinite(got)), f"{where}: non-finite logits"
    ws = rec["sampled"][t, p].astype(np.float64)
    gs = got[rec["sample_idx"]]
    err = max(float(np.abs(gs - ws).max()),
              float(np.abs(got[rec["top_idx"][t, p]] - rec["top_val"][t, p]).max()))
    rel = float(np.linalg.norm(gs - ws) / np.linalg.norm(ws))
    stats.setdefault("max_abs", []).append(err)
    stats.setdefault("rel_l2", []).append(rel)
    assert err <= MAX_ABS, f"{where}: logits max-abs {err:.3e} > {MAX_ABS}"
    assert rel <= REL_L2, f"{where}: logits rel-L2 {rel:.3e} > {REL_L2}"
    want_tok = int(rec["tokens"][t, p])
    if got_tok != want_tok:
        gap = float(rec["gaps"][t, p])
        assert gap < NEAR_TIE, f"{where}: token {got_tok} != oracle {want_tok} with top-2 gap {gap:.3e}"
        stats["near_ties"] = stats.get("near_ties", 0) + 1


def _replay(name, max_tokens, max_chunk):
    rec = np.load(os.path.join(GOLDEN, f"fullsize_{name}.npz"))
    cfg = gen.CONFIGS[str(rec["config"])]
    turns, steps, plen = int(rec["turns"]), int(rec["steps"]), int(rec["prompt_len"])
    full = {(int(t), int(p)): i for i, (t, p) in enumerate(rec["full_where"])}
    model = WiciModel(cfg, max_tokens=max_tokens, max_chunk=max_chunk).load(_weights_of(cfg))
    stats, full_stats = {}, {}

    def compare(got, gtok, t, p, where):
        if (t, p) in full:
            want = rec["full"][full[(t, p)]]
            check_step(got, gtok, want, int(rec["tokens"][t, p]), where + " (whole vector)", full_stats)
        _check_sampled(got, gtok, rec, t, p, where, stats)

    for t in range(turns):
        prompt = gen.make_prompt(cfg, plen, seed=int(rec["prompt_seeds"][t]))
        got, gtok = model.prefill(prompt, logits=True)
        compare(got, gtok, t, 0, f"{name} turn {t} prefill (kv {model.kv_len})")
        for s in range(steps):
            got, gtok = model.decode_step(int(rec["forced"][t, s]), logits=True)
            compare(got, gtok, t, 1 + s, f"{name} turn {t} step {s} (kv {model.kv_len})")
    assert model.kv_len == turns * (plen + steps)
    model.close()
    print(f"\n{name}: {len(stats['max_abs'])} positions; sampled max-abs {max(stats['max_abs']):.3e}, "
          f"rel-L2 {max(stats['rel_l2']):.3e}; whole vectors ({len(full_stats['max_abs'])}) max-abs "
          f"{max(full_stats['max_abs']):.3e}, rel-L2 {max(full_stats['rel_l2']):.3e}; "
          f"near ties {stats.get('near_ties', 0)}")
    return stats


def test_llama3_8b_request_64_decode_steps_against_stored_oracle():
    # the bench's launch configuration: 1024-token prompt in one chunk, room for 256 steps
    stats = _replay("llama3-8b", max_tokens=1024 + 256 + 16, max_chunk=1024)
    assert len(stats["max_abs"]) == 65


def test_llama3_8b_request_all_256_decode_steps_against_stored_oracle():
    # the bench's whole request: 1024-token prompt, then all 256 decode steps
    stats = _replay("llama3-8b-256", max_tokens=1024 + 256 + 16, max_chunk=1024)
    assert len(stats["max_abs"]) == 257


def test_agentic_full_depth_four_turns_against_stored_oracle():
    # 32 layers, 4 x (2048-token chunk + 64 decode steps), 8448 cached at the end
    stats = _replay("llama3-8b-agentic", max_tokens=8448, max_chunk=2048)
    assert len(stats["max_abs"]) == 4 * 65
    _weights.clear()


def test_llama32_1b_request_128_decode_steps_against_stored_oracle():
    # the 1B configuration's whole request: 512-token prompt, then 128 decode steps
    stats = _replay("llama3.2-1b", max_tokens=512 + 128 + 16, max_chunk=512)
    assert len(stats["max_abs"]) == 129
    _weights.clear()


def _full(cfg, decode_steps, max_chunk=None):
    w = gen.make_weights(cfg)
    prompt = gen.make_prompt(cfg, cfg.prompt_len, seed=1)
    max_tokens = cfg.prompt_len + decode_steps + 16
    model = WiciModel(cfg, max_tokens=max_tokens, max_chunk=max_chunk or cfg.prompt_len).load(w)
    ref = oracle.OracleModel(cfg, w, max_tokens=max_tokens, cache_bytes=0)
    stats = {}
    run_teacher_forced(model, ref, [prompt], decode_steps, stats)
    model.close()
    print(f"\n{cfg.name}: {len(stats['max_abs'])} positions; max-abs {max(stats['max_abs']):.3e} "
          f"(prefill {stats['max_abs'][0]:.3e}), rel-L2 {max(stats['rel_l2']):.3e}; near ties {stats.get('near_ties', 0)}")
    return stats


def test_llama32_1b_shape_full_prompt():
    stats = _full(gen.LLAMA_1B, decode_steps=8)
    assert len(stats["max_abs"]) == 9


def test_qwen25_14b_shape_full_prompt():
    # the deepest config: 48 layers, a 2048-token prompt, then one decode step
    stats = _full(gen.QWEN_14B, decode_steps=1)
    assert len(stats["max_abs"]) == 2
