"""Run the float64 oracle on many sampled units in parallel (test helper).

Full-size parity samples units of caches with up to 131072 tokens, where the
oracle takes seconds per unit. The units' exact host copies (float32, which
holds bf16 and float32 caches exactly) go to a pool of spawned processes (a
pool forked after CUDA was initialised could hang); each runs the oracle's
steps in the oracle's order (Algorithm 1: weights, scores, TOP-B) and returns
the scores and the TOP-B sets for the requested budgets.
"""

from __future__ import annotations

import multiprocessing as mp
import os

import numpy as np


def oracle_scores(q, K, V, budgets, tau):
    from oracle import JacapParams
    from oracle import jacap_oracle as J

    params = JacapParams(tau=tau)
    w = J.unit_weights(np.asarray(K, np.float64), np.asarray(q, np.float64), params)
    scores = J.jacap_scores(np.asarray(V, np.float64), w, params.ridge)
    return scores, {b: J.select_topb(scores, b)[0] for b in budgets}


def run_units(units, budgets, tau=10.0, processes=None):
    """units: list of (q [G,w,d], K [n,d], V [n,d]) float32 arrays. Returns
    [(scores, {budget: idx})] in the same order."""
    processes = processes or max(1, min(len(units), (os.cpu_count() or 2) // 2, 8))
    # one BLAS thread per worker: the pool supplies the parallelism
    saved = {k: os.environ.get(k) for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS")}
    os.environ["OMP_NUM_THREADS"] = os.environ["OPENBLAS_NUM_THREADS"] = "1"
    try:
        with mp.get_context("spawn").Pool(processes) as pool:
            return pool.starmap(oracle_scores, [(q, K, V, tuple(budgets), tau) for (q, K, V) in units])
    finally:
        for k, v in saved.items():
            if v is None:
                os.environ.pop(k, None)
            else:
                os.environ[k] = v
