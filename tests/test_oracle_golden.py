"""Regression pin: the oracle's tiny-configuration output equals the stored
record written by tests/golden/make_golden.py (which calls only oracle/ and gen/)."""
import json
import os

import numpy as np

from tests.golden.make_golden import tiny_record

HERE = os.path.dirname(os.path.abspath(__file__))


def test_tiny_oracle_matches_stored_record():
    with open(os.path.join(HERE, "golden", "tiny_oracle.json")) as f:
        want = json.load(f)
    got = tiny_record()
    assert got["prompt"] == want["prompt"]
    for g, w in zip(got["steps"], want["steps"], strict=True):
        assert g["token"] == w["token"]
        assert [i for i, _ in g["top5"]] == [i for i, _ in w["top5"]]
        np.testing.assert_allclose([v for _, v in g["top5"]], [v for _, v in w["top5"]],
                                   rtol=0, atol=1e-9)
        np.testing.assert_allclose([g["sum"], g["sumsq"]], [w["sum"], w["sumsq"]], rtol=1e-9)
