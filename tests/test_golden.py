"""The oracle reproduces the values stored in tests/golden/oracle_tiny.json
(written by tests/golden/make_golden.py from the oracle itself; see the
README there: they guard against unintended changes of the oracle)."""

import json
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.join(HERE, "golden"))

import make_golden  # noqa: E402


def test_oracle_reproduces_golden_values():
    with open(os.path.join(HERE, "golden", "oracle_tiny.json")) as f:
        stored = json.load(f)
    now = make_golden.golden()
    assert now["workload"] == stored["workload"]
    for r, steps in stored["rows"].items():
        for s, (a, b) in enumerate(zip(steps, now["rows"][r])):
            assert a["kept_positions"] == b["kept_positions"], (r, s)
            for key in ("o_row0", "Hq", "feat_first4", "score_first8"):
                np.testing.assert_allclose(np.array(b[key]), np.array(a[key]), rtol=1e-12, atol=1e-15, err_msg=key)
    for a, b in zip(stored["pl_logz"], now["pl_logz"]):
        assert b["logz"] == a["logz"] or abs(b["logz"] - a["logz"]) <= 1e-12 * abs(a["logz"])
    assert now["gumbel_top7"] == stored["gumbel_top7"]
