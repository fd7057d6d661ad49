"""The comparison rules themselves (tests/parity.py), on CPU with made-up
vectors: what passes, what fails, and the near-tie exception for tokens."""
import numpy as np
import pytest

from tests.parity import MAX_ABS, NEAR_TIE, REL_L2, check_step, top2_gap

r = np.random.default_rng(12)


def _want():
    w = r.standard_normal(1000) * 3
    w[17] = w.max() + 1.0             # a clear winner
    return w


def test_exact_and_within_tolerance_pass():
    w = _want()
    stats = {}
    check_step(w, 17, w, 17, "exact", stats)
    check_step(w + 0.9 * MAX_ABS, 17, w, 17, "shifted", stats)
    assert stats["max_abs"][0] == 0.0 and abs(stats["max_abs"][1] - 0.9 * MAX_ABS) < 1e-12


def test_max_abs_and_rel_l2_limits_fail():
    w = _want()
    bump = w.copy()
    bump[3] += 1.01 * MAX_ABS
    with pytest.raises(AssertionError, match="max-abs"):
        check_step(bump, 17, w, 17, "one element off")
    small = np.full(1000, 1e-3)
    small[17] = 1.0
    noisy = small + 1.5 * REL_L2 * np.linalg.norm(small) / np.sqrt(1000) * np.sign(r.standard_normal(1000))
    assert np.abs(noisy - small).max() <= MAX_ABS
    with pytest.raises(AssertionError, match="rel-L2"):
        check_step(noisy, 17, small, 17, "spread error")


def test_non_finite_logits_fail():
    w = _want()
    bad = w.copy()
    bad[5] = np.nan
    with pytest.raises(AssertionError, match="non-finite"):
        check_step(bad, 17, w, 17, "nan")


def test_token_rule_near_tie_only():
    w = _want()
    with pytest.raises(AssertionError, match="top-2 gap"):
        check_step(w, 3, w, 17, "clear winner missed")
    tie = w.copy()
    tie[400] = tie[17] - 0.5 * NEAR_TIE          # runner-up within the near-tie gap
    assert top2_gap(tie) < NEAR_TIE
    stats = {}
    check_step(tie, 400, tie, 17, "near tie", stats)
    assert stats["near_ties"] == 1
