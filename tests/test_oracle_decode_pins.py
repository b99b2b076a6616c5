"""Pins of the decoding-stage eviction oracle (reading R16).

Each fact is reached without the oracle's own bookkeeping: the eviction steps
from a closed form, the statistics from numpy over an independently built
history, the kept set from a construction whose scores are ordered by the
value norms alone.
"""

import numpy as np
import pytest

from oracle.decode_oracle import decode_run
from oracle.jacap_oracle import JacapParams


def _steps(r, T, G, d, K=None, V=None):
    out = []
    for t in range(T):
        k = r.normal(size=d) if K is None else K[t]
        v = r.normal(size=d) if V is None else V[t]
        out.append((r.normal(size=(G, d)), k, v))
    return out


def test_no_eviction_while_the_cache_stays_below_budget_plus_interval():
    r = np.random.default_rng(1)
    G, d, w, n0, T, B, D = 2, 8, 3, 5, 4, 8, 2  # at most 9 < B + D tokens
    events, ids, K, V = decode_run(r.normal(size=(G, w, d)), r.normal(size=(n0, d)), r.normal(size=(n0, d)),
                                   _steps(r, T, G, d), B, D)
    assert events == []
    assert list(ids) == list(range(n0 + T))
    assert K.shape == (n0 + T, d)


@pytest.mark.parametrize("n0", [3, 6, 8])
def test_evictions_happen_every_interval_once_the_cache_is_full(n0):
    # from n0 <= B + D - 1 tokens the cache first reaches B + D at step
    # B + D - n0 - 1 and then every D steps: t_k = B + (k + 1) D - n0 - 1
    r = np.random.default_rng(2)
    G, d, w, T, B, D = 1, 8, 4, 25, 6, 3
    events, ids, _, _ = decode_run(r.normal(size=(G, w, d)), r.normal(size=(n0, d)), r.normal(size=(n0, d)),
                                   _steps(r, T, G, d), B, D)
    expect = [B + (k + 1) * D - n0 - 1 for k in range(T) if B + (k + 1) * D - n0 - 1 < T]
    assert [e["step"] for e in events] == expect
    assert all(len(e["ids"]) == B + D and len(e["kept_ids"]) == B for e in events)
    last = expect[-1]
    assert len(ids) == B + (T - 1 - last)


def test_a_cache_longer_than_the_threshold_is_evicted_at_the_first_step():
    r = np.random.default_rng(3)
    G, d, w, n0, B, D = 1, 8, 4, 20, 6, 3
    events, _, _, _ = decode_run(r.normal(size=(G, w, d)), r.normal(size=(n0, d)), r.normal(size=(n0, d)),
                                 _steps(r, 4, G, d), B, D)
    assert events[0]["step"] == 0 and len(events[0]["ids"]) == n0 + 1


@pytest.mark.parametrize("order", ["newest", "oldest"])
def test_identical_keys_keep_the_largest_orthogonal_values(order):
    # identical keys give every token the same pool attention and the same
    # kappa, hence one weight w; with orthogonal values A is diagonal in their
    # basis and r_i = w s_i^2 / (1 + w s_i^2) grows with the value norm s_i.
    # Norms growing with the token id keep the B newest tokens; norms
    # shrinking with it keep the first B tokens for good.
    r = np.random.default_rng(4)
    G, d, w, n0, T, B, D = 2, 64, 5, 6, 40, 6, 3
    key = r.normal(size=d)
    n_all = n0 + T

    def value(i):
        s = 1.0 + 0.1 * i if order == "newest" else 10.0 - 0.1 * i
        return s * np.eye(d)[i]

    Vs = np.stack([value(i) for i in range(n_all)])
    Ks = np.tile(key, (n_all, 1))
    steps = _steps(r, T, G, d, K=Ks[n0:], V=Vs[n0:])
    events, ids, _, V = decode_run(r.normal(size=(G, w, d)), Ks[:n0], Vs[:n0], steps, B, D)
    assert len(events) > 5
    for e in events:
        want = e["ids"][-B:] if order == "newest" else np.arange(B)
        assert list(e["kept_ids"]) == list(want)
    np.testing.assert_array_equal(V, Vs[ids])


@pytest.mark.parametrize("unbiased", [False, True])
def test_statistics_are_the_moments_of_the_whole_query_history(unbiased):
    r = np.random.default_rng(5)
    G, d, w, n0, T, B, D = 2, 8, 4, 10, 30, 8, 4
    qp = r.normal(size=(G, w, d))
    steps = _steps(r, T, G, d)
    events, _, _, _ = decode_run(qp, r.normal(size=(n0, d)), r.normal(size=(n0, d)), steps, B, D,
                                 JacapParams(cov_unbiased=unbiased))
    assert len(events) >= 4
    for e in events:
        t = e["step"]
        for h in range(G):
            hist = np.concatenate([qp[h], np.stack([steps[j][0][h] for j in range(t + 1)])])
            np.testing.assert_allclose(e["mu"][h], np.mean(hist, axis=0), rtol=1e-12, atol=1e-14)
            np.testing.assert_allclose(e["lam"][h], np.var(hist, axis=0, ddof=1 if unbiased else 0), rtol=1e-12)
            # not the statistics of the last w queries only
            assert not np.allclose(e["mu"][h], np.mean(hist[-w:], axis=0))


def test_kept_tokens_ascend_and_evicted_tokens_never_return():
    r = np.random.default_rng(6)
    G, d, w, n0, T, B, D = 4, 16, 8, 12, 60, 10, 5
    events, ids, _, _ = decode_run(r.normal(size=(G, w, d)), r.normal(size=(n0, d)) * 2,
                                   r.normal(size=(n0, d)), _steps(r, T, G, d), B, D)
    gone = set()
    for e in events:
        kept = list(e["kept_ids"])
        assert kept == sorted(kept) and len(set(kept)) == B
        assert set(kept) <= set(e["ids"])
        assert not (set(e["ids"]) & gone)
        gone |= set(e["ids"]) - set(kept)
    assert list(ids) == sorted(ids) and not (set(ids) & gone)
