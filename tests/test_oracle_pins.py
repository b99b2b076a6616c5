"""Pins of the float64 oracle against facts the paper and mathematics fix.

No test here retypes the oracle's own formula: each one reaches the same
number by another route (a closed form, a library routine, an identity, a
limit, or brute force), chosen so that a dropped term, a wrong sign, a wrong
power, a transposed operand or a wrong normaliser fails at least one pin.
"""

import itertools
import math

import numpy as np
import pytest
from scipy.special import expit, softmax

from oracle import jacap_oracle as J
from oracle import theory as T


def rng(seed=0):
    return np.random.default_rng(seed)


# ---------------------------------------------------------------- step 1 ----
def test_window_stats_two_queries_closed_form():
    r = rng(1)
    q = r.normal(size=(2, 7))
    mu, lam = J.window_stats(q)
    np.testing.assert_allclose(mu, 0.5 * (q[0] + q[1]), rtol=1e-15)
    np.testing.assert_allclose(lam, (0.5 * (q[0] - q[1])) ** 2, rtol=1e-13)
    _, lam_u = J.window_stats(q, cov_unbiased=True)
    np.testing.assert_allclose(lam_u, 0.5 * (q[0] - q[1]) ** 2, rtol=1e-13)


def test_window_stats_match_numpy_moments():
    q = rng(2).normal(size=(32, 128))
    mu, lam = J.window_stats(q)
    np.testing.assert_allclose(mu, np.mean(q, axis=0), rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(lam, np.var(q, axis=0, ddof=0), rtol=1e-12)
    _, lam_u = J.window_stats(q, cov_unbiased=True)
    np.testing.assert_allclose(lam_u, np.var(q, axis=0, ddof=1), rtol=1e-12)


def test_window_of_one_query_has_zero_variance():
    mu, lam = J.window_stats(rng(3).normal(size=(1, 5)))
    assert np.all(lam == 0.0)
    with pytest.raises(ValueError):
        J.window_stats(np.ones((1, 5)), cov_unbiased=True)


# ---------------------------------------------------------------- step 2 ----
def test_pool_attention_two_tokens_is_logistic():
    r = rng(4)
    d, tau = 16, 3.0
    K = r.normal(size=(2, d)) * 4
    mu = r.normal(size=d)
    a = J.pool_attention(K, mu, tau)
    z = (K[0] - K[1]) @ mu / (tau * math.sqrt(d))
    np.testing.assert_allclose(a[0], expit(z), rtol=1e-14)
    np.testing.assert_allclose(a[1], expit(-z), rtol=1e-14)


def test_pool_attention_matches_scipy_softmax_with_temperature():
    r = rng(5)
    n, d, tau = 300, 64, 10.0
    K = r.normal(size=(n, d)) * 3
    mu = r.normal(size=d) * 2
    a = J.pool_attention(K, mu, tau)
    np.testing.assert_allclose(a, softmax(K @ mu / (tau * 8.0)), rtol=1e-12)
    assert abs(a.sum() - 1.0) < 1e-14


def test_pool_attention_limits():
    r = rng(6)
    K = r.normal(size=(50, 8))
    mu = r.normal(size=8)
    np.testing.assert_allclose(J.pool_attention(K, mu, 1e12), np.full(50, 1 / 50), rtol=1e-9)
    same = np.tile(r.normal(size=8), (50, 1))
    np.testing.assert_allclose(J.pool_attention(same, mu, 0.1), np.full(50, 1 / 50), rtol=1e-13)


# ---------------------------------------------------------------- step 3 ----
def _diagonal_covariance_window(mu, spread):
    """2d queries mu +- s_c e_c: empirical mean mu, covariance Diag(s_c^2 / d)."""
    d = mu.shape[0]
    Q = np.tile(mu, (2 * d, 1))
    for c in range(d):
        Q[2 * c, c] += spread[c]
        Q[2 * c + 1, c] -= spread[c]
    return Q


def test_kappa_is_the_variance_of_the_key_response():
    # Sec. 3.4: kappa_i is the variance of the logit k_i^T q under the query
    # perturbations. For a window whose empirical covariance is diagonal this
    # is the population variance of k_i^T q_j over the window.
    r = rng(7)
    d, n = 12, 40
    mu = r.normal(size=d)
    Q = _diagonal_covariance_window(mu, r.uniform(0.5, 3.0, size=d))
    K = r.normal(size=(n, d)) * r.uniform(0.2, 5, size=d)
    _, lam = J.window_stats(Q)
    kappa = J.response_variance(K, lam)
    np.testing.assert_allclose(kappa, np.var(Q @ K.T, axis=0, ddof=0), rtol=1e-12)


def test_rho_extremes_and_peak():
    rho = J.sensitivity(np.array([0.0, 0.5, 1.0, 0.25]))
    np.testing.assert_allclose(rho, [0.0, 0.25, 0.0, 0.1875])


# ---------------------------------------------------------------- step 4 ----
def test_weight_is_diagonal_of_the_linearised_channel():
    # App. B.1: with S_C -> D = Diag(rho) and K Lam K^T -> its diagonal, the
    # channel matrix J Lam J^T = (1/d) U D K Lam K^T D U^T reduces to
    # U Diag(w) U^T, so w is the diagonal of (1/d) D (K Lam K^T) D.
    r = rng(8)
    n, d, tau = 30, 16, 2.0
    K = r.normal(size=(n, d)) * 2
    Qw = r.normal(size=(8, d)) + r.normal(size=d)
    mu, lam = J.window_stats(Qw)
    a = softmax(K @ mu / (tau * math.sqrt(d)))
    D = np.diag(a * (1 - a))
    full = D @ (K @ np.diag(lam) @ K.T) @ D / d
    w = J.head_weight(K, mu, lam, J.JacapParams(tau=tau))
    np.testing.assert_allclose(w, np.diag(full), rtol=1e-12)


def test_weight_channel_identity_with_orthogonal_keys():
    # Keys along distinct axes make K Lam K^T exactly diagonal; then the
    # diagonal-S channel U D K Lam K^T D U^T / d equals U Diag(w) U^T exactly.
    r = rng(9)
    d, n, tau = 10, 6, 1.0
    K = np.zeros((n, d))
    for i in range(n):
        K[i, i] = r.uniform(0.5, 3.0) * (-1) ** i
    U = r.normal(size=(n, d))
    Qw = r.normal(size=(5, d))
    mu, lam = J.window_stats(Qw)
    a = softmax(K @ mu / math.sqrt(d))
    JD = U.T @ np.diag(a * (1 - a)) @ K / math.sqrt(d)  # Lemma 1 with S -> Diag(rho)
    w = J.head_weight(K, mu, lam, J.JacapParams(tau=tau))
    np.testing.assert_allclose(JD @ np.diag(lam) @ JD.T, U.T @ np.diag(w) @ U, rtol=1e-11, atol=1e-15)


def test_uniform_keys_closed_form():
    # All keys equal: alpha = 1/n, rho = (n-1)/n^2, kappa = c^2 sum(lam).
    n, d, c = 37, 8, 1.5
    K = np.full((n, d), c)
    Qw = rng(10).normal(size=(4, d))
    mu, lam = J.window_stats(Qw)
    w = J.head_weight(K, mu, lam)
    expected = ((n - 1) / n**2) ** 2 * c * c * lam.sum() / d
    np.testing.assert_allclose(w, expected, rtol=1e-13)
    w_nodiv = J.head_weight(K, mu, lam, J.JacapParams(weight_div_dk=False))
    np.testing.assert_allclose(w_nodiv, expected * d, rtol=1e-13)


def test_gqa_weights_are_the_sum_over_the_group_and_map_h_over_G():
    # Reading R5 through the cache layout: a G=2 cache equals the sum of two
    # one-head caches whose KV planes repeat the shared head.
    r = rng(11)
    L, Hkv, G, n, d, w = 1, 2, 2, 20, 8, 3
    k = r.normal(size=(L, Hkv, n, d))
    v = r.normal(size=(L, Hkv, n, d))
    q = r.normal(size=(1, L, Hkv * G, w, d))
    cu = np.array([0, n])
    gqa = J.oracle_pass(q, k, v, cu, Hkv * G, Hkv, budget=5)
    k_rep = np.repeat(k, G, axis=1)
    v_rep = np.repeat(v, G, axis=1)
    mha = J.oracle_pass(q, k_rep, v_rep, cu, Hkv * G, Hkv * G, budget=5)
    for g in range(Hkv):
        expect = sum(mha[(0, 0, g * G + j)]["w"] for j in range(G))
        np.testing.assert_allclose(gqa[(0, 0, g)]["w"], expect, rtol=1e-13)


# ------------------------------------------------------------ steps 5-6 ----
def test_scores_equal_ridge_leverage_from_the_svd():
    r = rng(12)
    n, d = 200, 16
    V = r.normal(size=(n, d))
    w = r.uniform(0, 0.2, size=n)
    s = J.jacap_scores(V, w)
    P, sig, _ = np.linalg.svd(np.sqrt(w)[:, None] * V, full_matrices=False)
    ridge = sig**2 / (1 + sig**2)
    np.testing.assert_allclose(s, (P**2) @ ridge, rtol=1e-11)
    np.testing.assert_allclose(s.sum(), ridge.sum(), rtol=1e-12)
    assert np.all(s >= 0) and np.all(s < 1)


def test_ridge_free_leverage_sums_to_rank():
    r = rng(13)
    n, d = 60, 8
    w = r.uniform(0.1, 1, size=n)
    V = r.normal(size=(n, d))
    s = J.jacap_scores(V, w, ridge=False)
    assert abs(s.sum() - d) < 1e-9
    assert np.all(s > -1e-12) and np.all(s <= 1 + 1e-12)
    V[:, 5:] = 0.0  # rank 5
    s = J.jacap_scores(V, w, ridge=False)
    assert abs(s.sum() - 5) < 1e-9


def test_leave_one_out_determinant_identity():
    # App. B.1 (matrix determinant lemma): w_i u_i^T A^-1 u_i = 1 - det(A_-i)/det(A).
    r = rng(14)
    n, d = 12, 5
    V = r.normal(size=(n, d))
    w = r.uniform(0, 2, size=n)
    s = J.jacap_scores(V, w)
    full = np.linalg.slogdet(np.eye(d) + (V * w[:, None]).T @ V)[1]
    for i in range(n):
        keep = np.arange(n) != i
        part = np.linalg.slogdet(np.eye(d) + (V[keep] * w[keep, None]).T @ V[keep])[1]
        np.testing.assert_allclose(s[i], 1 - math.exp(part - full), rtol=1e-10, atol=1e-14)


def test_one_channel_closed_form():
    r = rng(15)
    v = r.normal(size=(9, 1))
    w = r.uniform(0, 1, size=9)
    s = J.jacap_scores(v, w)
    np.testing.assert_allclose(s, w * v[:, 0] ** 2 / (1 + np.sum(w * v[:, 0] ** 2)), rtol=1e-13)


def test_scores_use_values_not_keys():
    # u_i = v_i (Sec. 3.4). V with a single live channel makes A diagonal.
    r = rng(16)
    n, d = 25, 6
    K = r.normal(size=(n, d))
    V = np.zeros((n, d))
    V[:, 2] = r.normal(size=n)
    Q = r.normal(size=(1, 4, d))
    out = J.oracle_unit(Q, K, V, budget=3)
    w = out["w"]
    np.testing.assert_allclose(out["scores"], w * V[:, 2] ** 2 / (1 + np.sum(w * V[:, 2] ** 2)), rtol=1e-12)


def test_permutation_equivariance():
    r = rng(17)
    n, d = 80, 16
    K = r.normal(size=(n, d)) * 2
    V = r.normal(size=(n, d))
    Q = r.normal(size=(2, 6, d))
    p = r.permutation(n)
    a = J.oracle_unit(Q, K, V, budget=10, params=J.JacapParams(tau=0.5))
    b = J.oracle_unit(Q, K[p], V[p], budget=10, params=J.JacapParams(tau=0.5))
    np.testing.assert_allclose(b["scores"], a["scores"][p], rtol=1e-10)
    np.testing.assert_allclose(b["w"], a["w"][p], rtol=1e-12)
    assert set(p[b["idx"]].tolist()) == set(a["idx"].tolist())


def test_orthogonal_values_topb_is_the_brute_force_optimum():
    # With mutually orthogonal u_i the approximated capacity separates into
    # sum_C 1/2 log(1 + w_i |u_i|^2) and r_i is increasing in w_i |u_i|^2, so
    # Jacap's TOP-B maximises the approximated objective (App. B.1).
    r = rng(18)
    n, d, B = 11, 16, 4
    Qo, _ = np.linalg.qr(r.normal(size=(d, d)))
    V = Qo[:n] * r.uniform(0.5, 2.0, size=(n, 1))
    K = r.normal(size=(n, d)) * 3
    Q = r.normal(size=(1, 5, d))
    out = J.oracle_unit(Q, K, V, budget=B, params=J.JacapParams(tau=0.3))
    best, args = T.brute_force_best(n, B, lambda C: T.approx_capacity(V[list(C)], out["w"][list(C)]))
    assert tuple(out["idx"].tolist()) in [tuple(c) for c in args]


# ---------------------------------------------------------------- step 7 ----
def test_select_hand_cases():
    idx, kept = J.select_topb(np.array([0.5, 0.9, 0.5, 0.1, 0.9]), 3)
    assert idx.tolist() == [0, 1, 4] and kept == 3
    idx, kept = J.select_topb(np.array([0.5, 0.5, 0.5, 0.5]), 2)
    assert idx.tolist() == [0, 1]
    idx, kept = J.select_topb(np.array([0.2, 0.3]), 4)
    assert idx.tolist() == [0, 1, -1, -1] and kept == 2
    idx, kept = J.select_topb(np.array([0.0, 3.0, 2.0]), 1)
    assert idx.tolist() == [1]


def test_select_matches_brute_force_with_ties():
    r = rng(19)
    for trial in range(40):
        n = int(r.integers(1, 10))
        B = int(r.integers(1, 6))
        s = r.integers(0, 4, size=n) / 4.0  # dyadic values: exact ties
        idx, kept = J.select_topb(s, B)
        if n <= B:
            assert idx[:n].tolist() == list(range(n))
            continue
        cands = list(itertools.combinations(range(n), B))
        best = max(sum(s[list(c)]) for c in cands)
        winners = sorted(c for c in cands if sum(s[list(c)]) == best)
        assert tuple(idx.tolist()) == winners[0]


def test_compact_is_a_bitwise_row_gather():
    r = rng(20)
    K = r.normal(size=(10, 4)).astype(np.float32)
    V = r.normal(size=(10, 4)).astype(np.float32)
    idx = np.array([1, 4, 7, -1])
    k_out, v_out = J.compact(K, V, idx, 3)
    assert k_out.tobytes() == np.concatenate([K[1:2], K[4:5], K[7:8]]).tobytes()
    assert v_out.tobytes() == np.concatenate([V[1:2], V[4:5], V[7:8]]).tobytes()


def test_window_of_one_gives_zero_scores_and_first_b():
    # Reading R12: w = 1 => lambda = 0 => every weight and score is 0.
    r = rng(21)
    out = J.oracle_unit(r.normal(size=(1, 1, 8)), r.normal(size=(30, 8)), r.normal(size=(30, 8)), budget=7)
    assert np.all(out["scores"] == 0.0)
    assert out["idx"].tolist() == list(range(7))


# ----------------------------------------------------------------- theory ---
def test_lemma1_jacobian_matches_finite_differences():
    r = rng(22)
    n, d = 9, 6
    U = r.normal(size=(n, 4))
    K = r.normal(size=(n, d)) * 2
    mu = r.normal(size=d)
    Jm = T.retained_jacobian(U, K, mu)
    h = 1e-5
    fd = np.zeros_like(Jm)
    for c in range(d):
        e = np.zeros(d)
        e[c] = h
        fd[:, c] = (T.retained_map(U, K, mu + e) - T.retained_map(U, K, mu - e)) / (2 * h)
    np.testing.assert_allclose(Jm, fd, rtol=1e-7, atol=1e-9)


def test_theorem1_objective_of_the_jacap_set_is_reported():
    # Jacap is a heuristic for Theorem 1's objective: the paper claims no
    # optimality, so only the ordering <= optimum is asserted.
    r = rng(23)
    n, d, B = 10, 6, 3
    K = r.normal(size=(n, d)) * 2
    V = r.normal(size=(n, d))
    Q = r.normal(size=(1, 6, d))
    out = J.oracle_unit(Q, K, V, budget=B, params=J.JacapParams(tau=1.0))
    mu, lam = J.window_stats(Q[0])

    def obj(C):
        C = list(C)
        return T.jacobian_capacity(V[C], K[C], mu, lam)

    best, _ = T.brute_force_best(n, B, obj)
    got = obj(out["idx"])
    assert got <= best + 1e-12
    assert got > 0


def test_theorem1_capacity_two_tokens_scalar_closed_form():
    # d_k = d_o = 1, two tokens: S = a1 a2 [[1, -1], [-1, 1]], so
    # J = a1 a2 (u1 - u2)(k1 - k2) and the capacity is
    # 1/2 log(1 + lambda J^2 / sigma^2), with a1 = logistic((k1 - k2) mu).
    k1, k2, u1, u2, mu, lam, sig2 = 1.3, -0.4, 0.7, -1.1, 0.8, 2.5, 0.6
    a1 = expit((k1 - k2) * mu)
    jac = a1 * (1 - a1) * (u1 - u2) * (k1 - k2)
    want = 0.5 * math.log1p(lam * jac * jac / sig2)
    got = T.jacobian_capacity(np.array([[u1], [u2]]), np.array([[k1], [k2]]), np.array([mu]), np.array([lam]),
                              noise=np.array([[sig2]]))
    assert got == pytest.approx(want, rel=1e-13)


def test_theorem1_capacity_is_the_gaussian_channel_information():
    # Theorem 1's objective is the mutual information of y = J q + e with
    # q ~ N(mu, Lambda) and e ~ N(0, Sigma): 1/2 [logdet(J Lambda J^T + Sigma)
    # - logdet(Sigma)]. J comes here from central differences of Eq. 3, with
    # d_o != d_k and a non-identity Sigma, so a transposed Jacobian, a dropped
    # 1/2 or Sigma applied on the wrong side all fail.
    r = rng(29)
    n, dk, do = 6, 5, 3
    K = r.normal(size=(n, dk))
    U = r.normal(size=(n, do))
    mu = r.normal(size=dk)
    lam = r.uniform(0.5, 2.0, size=dk)
    A = r.normal(size=(do, do))
    Sig = A @ A.T + 0.5 * np.eye(do)
    h = 1e-5
    Jfd = np.zeros((do, dk))
    for c in range(dk):
        e = np.zeros(dk)
        e[c] = h
        Jfd[:, c] = (T.retained_map(U, K, mu + e) - T.retained_map(U, K, mu - e)) / (2 * h)
    want = 0.5 * (np.linalg.slogdet(Jfd @ np.diag(lam) @ Jfd.T + Sig)[1] - np.linalg.slogdet(Sig)[1])
    got = T.jacobian_capacity(U, K, mu, lam, noise=Sig)
    assert got == pytest.approx(want, rel=1e-7)
