"""Float64 CPU oracle for decoding-stage eviction.

TEST INFRASTRUCTURE, under the same rules as ``jacap_oracle``: only
``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU legs may import
it; the CUDA path never calls it and it never imports the CUDA path.

The paper also evaluates Jacap while the model generates (Sec. 4, the
decoding-eviction experiments, whose budget is a number of reserved tokens)
and says that mu_Q and Lambda_Q are then estimated from the queries observed
so far (Sec. 3.4, last paragraph). It gives no schedule. Reading R16:

* the statistics of a (request, layer, query head) use every query observed
  for it: the prefill window's w queries, then one query per decode step;
  mu_Q is their mean and the diagonal Lambda_Q their per-channel variance
  (divide by the count n; by n - 1 with ``cov_unbiased``) -- reading R4 with
  the window grown to the whole history;
* a decode step first appends its token's (k, v) to the cache and its query
  to the history; then, if the cache holds at least B + Delta tokens, it runs
  Algorithm 1 steps 1-5 (``jacap_oracle.oracle_unit``) on the whole cache with
  those statistics and keeps the B best tokens in their cache order.
  Delta >= 1 is the eviction interval.

The oracle keeps the whole query history and recomputes the statistics from
it at every eviction: the definition, not a running update.
"""

from __future__ import annotations

import numpy as np

from .jacap_oracle import JacapParams, oracle_unit


def decode_run(q_prefill, K0, V0, steps, budget: int, interval: int, params: JacapParams = JacapParams()):
    """Decoding-stage eviction of one unit (request, layer, KV head).

    q_prefill  (G, w, d): the prefill window queries of the G query heads.
    K0, V0     (n0, d): the cache when decoding starts; its tokens get ids
               0 .. n0 - 1 and decode step t adds id n0 + t.
    steps      sequence of (q (G, d), k (d,), v (d,)) per decode step.
    Returns (events, ids, K, V): every eviction as a dict {step, ids (the cache
    before it, in cache order), mu, lam, scores, idx, kept_ids}, and the final
    cache ids and rows.
    """
    if budget < 1 or interval < 1:
        raise ValueError("budget and interval must be >= 1")
    hist = [np.asarray(q, dtype=np.float64) for q in np.asarray(q_prefill, dtype=np.float64).transpose(1, 0, 2)]
    K = [np.asarray(r) for r in np.asarray(K0)]
    V = [np.asarray(r) for r in np.asarray(V0)]
    ids = list(range(len(K)))
    next_id = len(K)
    events = []
    for t, (q, k, v) in enumerate(steps):
        K.append(np.asarray(k))
        V.append(np.asarray(v))
        ids.append(next_id)
        next_id += 1
        hist.append(np.asarray(q, dtype=np.float64))
        if len(K) >= budget + interval:
            q_group = np.stack(hist, axis=1)  # (G, n_q, d): the whole history
            ora = oracle_unit(q_group, np.stack(K), np.stack(V), budget, params)
            sel = [int(i) for i in ora["idx"][: ora["kept"]]]
            events.append({"step": t, "ids": np.array(ids), "mu": ora["mu"], "lam": ora["lam"],
                           "scores": ora["scores"], "idx": ora["idx"], "kept_ids": np.array([ids[i] for i in sel])})
            K = [K[i] for i in sel]
            V = [V[i] for i in sel]
            ids = [ids[i] for i in sel]
    return events, np.array(ids), np.stack(K), np.stack(V)
