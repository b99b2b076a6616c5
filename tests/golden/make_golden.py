"""Writes tests/golden/tiny_units.json from the float64 oracle alone.

The inputs are small integers divided by powers of two (exact in bf16, fp32
and fp64), so the fixture can feed any implementation bit-for-bit. Every
expected value comes from ``oracle.oracle_unit`` (Algorithm 1, Sec. 3.4;
Eqs. 8-10). Re-run after a deliberate, paper-justified oracle change:

    python tests/golden/make_golden.py
"""

import json
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))

from oracle import JacapParams, oracle_unit  # noqa: E402


def tiny_inputs(case: int):
    """Deterministic dyadic inputs for case ``case`` (no RNG library state)."""
    n, d, G, w = [(24, 8, 2, 3), (17, 8, 1, 4), (40, 16, 4, 2)][case]
    idx = np.arange(n * d).reshape(n, d)
    K = (((idx * 37 + 11 * case) % 29) - 14) / 8.0
    V = (((idx * 53 + 7 * case) % 31) - 15) / 16.0
    qi = np.arange(G * w * d).reshape(G, w, d)
    Q = (((qi * 41 + 5 * case) % 23) - 11) / 4.0
    tau = [1.0, 10.0, 0.5][case]
    budget = [5, 20, 9][case]
    return Q, K, V, tau, budget


def main():
    cases = []
    for c in range(3):
        Q, K, V, tau, budget = tiny_inputs(c)
        out = oracle_unit(Q, K, V, budget, JacapParams(tau=tau))
        cases.append({
            "case": c,
            "tau": tau,
            "budget": budget,
            "w": [float(x) for x in out["w"]],
            "scores": [float(x) for x in out["scores"]],
            "idx": [int(x) for x in out["idx"]],
            "kept": int(out["kept"]),
        })
    doc = {
        "source": "oracle.oracle_unit (Algorithm 1, Sec. 3.4; Eqs. 8-10), float64",
        "inputs": "tests/golden/make_golden.py:tiny_inputs",
        "cases": cases,
    }
    with open(os.path.join(HERE, "tiny_units.json"), "w") as f:
        json.dump(doc, f, indent=1)


if __name__ == "__main__":
    main()
