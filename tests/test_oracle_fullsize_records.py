"""Consistency of the stored full-size oracle records (tests/golden/fullsize_*.npz,
written by make_fullsize_golden.py from the oracle alone): the forced tokens are
the seeded draws the script names, every recorded token, top-2 gap, sample and
top-8 entry agrees with the whole logits vectors where those are kept, and the
shapes match the workload.  No GPU and no oracle run needed."""
import os

import numpy as np
import pytest

import gen

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
RECORDS = {"llama3-8b": (1, 1024, 64), "llama3-8b-agentic": (4, 2048, 64), "llama3.2-1b": (1, 512, 128),
           "llama3-8b-256": (1, 1024, 256)}


@pytest.mark.parametrize("name", sorted(RECORDS))
def test_fullsize_record_is_self_consistent(name):
    path = os.path.join(GOLDEN, f"fullsize_{name}.npz")
    if not os.path.exists(path):
        pytest.skip(f"{path} not written yet")
    rec = np.load(path)
    turns, plen, steps = RECORDS[name]
    cfg = gen.CONFIGS[str(rec["config"])]
    assert (int(rec["turns"]), int(rec["prompt_len"]), int(rec["steps"])) == (turns, plen, steps)
    assert cfg.prompt_len == plen and cfg.turns == turns
    assert list(rec["prompt_seeds"]) == list(cfg.prompt_seeds[:turns])
    for t in range(turns):
        np.testing.assert_array_equal(rec["forced"][t], gen.make_prompt(cfg, steps, seed=101 + t))
    idx = rec["sample_idx"]
    assert len(idx) == 1024 and np.all(np.diff(idx) > 0) and idx[-1] < cfg.vocab
    assert rec["tokens"].shape == rec["gaps"].shape == (turns, 1 + steps)
    assert np.all(rec["gaps"] >= 0)
    # every turn keeps its prefill and its last step whole
    where = {tuple(w) for w in rec["full_where"]}
    assert all((t, 0) in where and (t, steps) in where for t in range(turns))
    for (t, p), full in zip(rec["full_where"], rec["full"]):
        full = full.astype(np.float64)
        assert int(np.argmax(full)) == rec["tokens"][t, p]
        top2 = np.sort(full)[-2:]
        assert abs((top2[1] - top2[0]) - rec["gaps"][t, p]) < 1e-5
        np.testing.assert_array_equal(rec["sampled"][t, p], full[idx].astype(np.float32))
        np.testing.assert_array_equal(rec["top_val"][t, p], full[rec["top_idx"][t, p]].astype(np.float32))
    # the top-8 lists are sorted and start at the recorded token
    assert np.all(rec["top_idx"][:, :, 0] == rec["tokens"])
    assert np.all(np.diff(rec["top_val"], axis=-1) <= 0)
