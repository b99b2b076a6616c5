"""Regression of the oracle against the committed golden fixture.

The fixture is written by tests/golden/make_golden.py from the oracle alone;
this test catches an unintended change of the oracle's arithmetic.
"""

import json
import os
import sys

import numpy as np

from oracle import JacapParams, oracle_unit

HERE = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
sys.path.insert(0, HERE)
from make_golden import tiny_inputs  # noqa: E402


def test_oracle_matches_golden_fixture():
    with open(os.path.join(HERE, "tiny_units.json")) as f:
        doc = json.load(f)
    for case in doc["cases"]:
        Q, K, V, tau, budget = tiny_inputs(case["case"])
        out = oracle_unit(Q, K, V, budget, JacapParams(tau=tau))
        np.testing.assert_allclose(out["w"], case["w"], rtol=1e-12, atol=0)
        np.testing.assert_allclose(out["scores"], case["scores"], rtol=1e-12, atol=0)
        assert out["idx"].tolist() == case["idx"]
        assert out["kept"] == case["kept"]
