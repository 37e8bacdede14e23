"""Fixtures under tests/golden/.

- table5_cross_family_handoff.txt: the handoff and native-prefill times the paper prints for
  Qwen2.5-1.5B -> Gemma-2-2B (Table 5).  The printed reductions are 1 - handoff / native,
  rounded to two decimals; at 4K that is 67.04% (the abstract's 67.05% rounds differently).
- oracle_regression.json: sampled oracle outputs written by make_oracle_golden.py (oracle
  only).  A change to the oracle's arithmetic changes them; such a change must cite the
  passage that justifies it, and the fixture is then rewritten by that script.
"""
import json
import os

import numpy as np

from golden.make_oracle_golden import CASES, build, key

HERE = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def test_table5_reductions_are_one_minus_the_time_ratio():
    rows = [ln.split() for ln in open(os.path.join(HERE, "table5_cross_family_handoff.txt"))
            if ln.strip() and not ln.startswith("#")]
    assert [int(r[0]) for r in rows] == [128, 1024, 4096]
    for _, handoff, native, printed in rows:
        red = 100.0 * (1.0 - float(handoff) / float(native))
        assert round(red, 2) == float(printed), (red, printed)
    assert abs(100.0 * (1.0 - 59.897 / 181.706) - 67.036) < 1e-3     # not 67.05


def test_oracle_matches_its_regression_fixture():
    want = json.load(open(os.path.join(HERE, "oracle_regression.json")))
    got = build()
    assert set(got) == set(want) == {key(*c) for c in CASES}
    for k in want:
        w, g = want[k], got[k]
        assert g["index"] == w["index"] and g["layer_map"] == w["layer_map"]
        assert g["span_lo"] == w["span_lo"] and g["span_hi"] == w["span_hi"]
        # fp64 oracle; libm may differ in the last bits between machines
        np.testing.assert_allclose(g["k"], w["k"], rtol=1e-12, atol=1e-12)
        np.testing.assert_allclose(g["v"], w["v"], rtol=1e-12, atol=1e-12)
