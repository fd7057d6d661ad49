"""Comparison rules between the CUDA path and the CPU oracle.

Logits: max-abs error <= 2e-2 and relative L2 error <= 1e-2 at every compared
position.  Greedy tokens: identical unless the oracle's top-2 logit gap is
below 1e-3.  The GPU is fed the oracle's tokens (teacher forcing through
`token_in`), so an accepted near-tie never carries into later steps; no oracle
input ever comes from the GPU.
"""
from __future__ import annotations

import numpy as np

MAX_ABS = 2e-2
REL_L2 = 1e-2
NEAR_TIE = 1e-3


def top2_gap(logits: np.ndarray) -> float:
    s = np.partition(np.asarray(logits, np.float64), -2)[-2:]
    return float(s[1] - s[0])


def check_step(got_logits, got_tok, want_logits, want_tok, where: str, stats: dict | None = None):
    got = np.asarray(got_logits, np.float64)
    want = np.asarray(want_logits, np.float64)
    assert np.all(np.isfinite(got)), f"{where}: non-finite logits"
    err = float(np.abs(got - want).max())
    rel = float(np.linalg.norm(got - want) / np.linalg.norm(want))
    if stats is not None:
        stats.setdefault("max_abs", []).append(err)
        stats.setdefault("rel_l2", []).append(rel)
    assert err <= MAX_ABS, f"{where}: logits max-abs {err:.3e} > {MAX_ABS}"
    assert rel <= REL_L2, f"{where}: logits rel-L2 {rel:.3e} > {REL_L2}"
    if got_tok != want_tok:
        gap = top2_gap(want)
        assert gap < NEAR_TIE, f"{where}: token {got_tok} != oracle {want_tok} with top-2 gap {gap:.3e}"
        if stats is not None:
            stats["near_ties"] = stats.get("near_ties", 0) + 1


def run_teacher_forced(model, ref, prompts, decode_steps: int, stats: dict | None = None):
    """Each turn: prefill the prompt, then `decode_steps` steps fed with the
    oracle's greedy tokens; every produced logits vector is compared."""
    n = 0
    for ti, prompt in enumerate(prompts):
        want, wtok = ref.prefill(prompt)
        got, gtok = model.prefill(prompt, logits=True)
        check_step(got, gtok, want, wtok, f"turn {ti} prefill", stats)
        n += 1
        for s in range(decode_steps):
            feed = wtok
            want, wtok = ref.decode(feed)
            got, gtok = model.decode_step(feed, logits=True)
            check_step(got, gtok, want, wtok, f"turn {ti} step {s}", stats)
            n += 1
    assert model.kv_len == ref.kv_len
    return n
