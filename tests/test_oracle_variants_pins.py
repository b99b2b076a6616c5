"""Pins of the oracle's variants against facts fixed by the paper and mathematics.

R13 linear weighting (S_C = I), R14 full-covariance Lambda_Q, and the greedy
log-determinant reference selection. As in test_oracle_pins.py, each value is
reached by a route other than the oracle's own formula.
"""

import itertools
import math

import numpy as np

from oracle import jacap_oracle as J


def rng(seed=0):
    return np.random.default_rng(seed)


LIN = J.JacapParams(linear_weighting=True)
FULL = J.JacapParams(full_covariance=True)


# ------------------------------------------------------------- R13 linear ----
def test_linear_weights_are_the_jacobian_channel_with_identity_sensitivity():
    # App. B.1: w = diag((1/d) D K Lambda K^T D) with D = Diag(rho); with
    # S_C = I (the linear surrogate) D = I, so w = diag(K Lambda K^T) / d.
    r = rng(1)
    n, d, G, wq = 40, 16, 3, 9
    K = r.normal(size=(n, d)) * r.lognormal(size=d)
    q = r.normal(size=(G, wq, d))
    w = J.unit_weights(K, q, LIN)
    ref = np.zeros(n)
    for h in range(G):
        Lam = np.diag(np.var(q[h], axis=0))
        ref += np.diag(K @ Lam @ K.T) / d
    np.testing.assert_allclose(w, ref, rtol=1e-12)


def test_linear_weights_ignore_the_query_mean_jacobian_weights_do_not():
    # shifting every window query by one vector leaves Lambda_Q unchanged and
    # moves mu_Q: only the softmax-aware weight may change
    r = rng(2)
    n, d, wq = 64, 8, 6
    K = r.normal(size=(n, d)) * 3
    q = r.normal(size=(1, wq, d))
    shift = r.normal(size=d) * 5
    np.testing.assert_allclose(J.unit_weights(K, q + shift, LIN), J.unit_weights(K, q, LIN), rtol=1e-12)
    assert not np.allclose(J.unit_weights(K, q + shift), J.unit_weights(K, q), rtol=1e-3)


def test_linear_weight_of_a_single_token_scales_with_tau_free_kappa():
    # n = 1: alpha = 1 so the Jacobian weight vanishes (saturation, App. A),
    # while the linear weight is kappa / d for any tau
    r = rng(3)
    d = 5
    K = r.normal(size=(1, d))
    q = r.normal(size=(1, 4, d))
    assert J.unit_weights(K, q)[0] == 0.0
    lam = np.var(q[0], axis=0)
    for tau in (0.1, 10.0):
        w = J.unit_weights(K, q, J.JacapParams(tau=tau, linear_weighting=True))
        np.testing.assert_allclose(w[0], (K[0] ** 2) @ lam / d, rtol=1e-13)


# ---------------------------------------------------- R14 full covariance ----
def test_full_covariance_kappa_is_the_window_variance_of_the_logits():
    # k^T Lambda_Q k with the full covariance equals the variance, over the
    # window, of the logits q_j . k (no diagonal assumption)
    r = rng(4)
    n, d, wq = 30, 12, 7
    K = r.normal(size=(n, d))
    C = r.normal(size=(d, d))
    q = r.normal(size=(wq, d)) @ C  # strongly correlated channels
    Lam = J.window_covariance(q)
    kappa = J.response_variance_full(K, Lam)
    np.testing.assert_allclose(kappa, np.var(q @ K.T, axis=0, ddof=0), rtol=1e-11)
    kappa_u = J.response_variance_full(K, J.window_covariance(q, cov_unbiased=True))
    np.testing.assert_allclose(kappa_u, np.var(q @ K.T, axis=0, ddof=1), rtol=1e-11)


def test_full_covariance_matches_numpy_cov():
    q = rng(5).normal(size=(9, 6)) @ rng(6).normal(size=(6, 6))
    np.testing.assert_allclose(J.window_covariance(q), np.cov(q, rowvar=False, ddof=0), rtol=1e-12)
    np.testing.assert_allclose(J.window_covariance(q, True), np.cov(q, rowvar=False, ddof=1), rtol=1e-12)


def test_full_and_diagonal_kappa_agree_for_uncorrelated_channels():
    # each window query deviates from a common base along one channel only,
    # in +/- pairs: the covariance is exactly diagonal, so both estimators
    # give the same kappa, and it equals diag(2 x_c^2 / w)
    r = rng(7)
    d, n = 6, 25
    b = r.normal(size=d)
    x = r.random(d) * 3 + 0.5
    q = np.stack([b + s * x[c] * np.eye(d)[c] for c in range(d) for s in (1.0, -1.0)])
    w = q.shape[0]
    Lam = J.window_covariance(q)
    np.testing.assert_allclose(Lam, np.diag(2 * x * x / w), rtol=1e-12, atol=1e-15)
    K = r.normal(size=(n, d))
    np.testing.assert_allclose(J.response_variance_full(K, Lam),
                               J.response_variance(K, J.window_stats(q)[1]), rtol=1e-12)


def test_full_covariance_weight_counts_cross_channel_terms():
    # two channels moving together: k = (1, -1) sees no variance with the full
    # covariance but twice the channel variance with the diagonal one
    q = np.array([[[1.0, 1.0]], [[-1.0, -1.0]]]).reshape(1, 2, 2)
    K = np.array([[1.0, -1.0], [1.0, 1.0]])
    Lam = J.window_covariance(q[0])
    kf = J.response_variance_full(K, Lam)
    kd = J.response_variance(K, J.window_stats(q[0])[1])
    np.testing.assert_allclose(kf, [0.0, 4.0], atol=1e-15)
    np.testing.assert_allclose(kd, [2.0, 2.0], rtol=1e-15)


# ------------------------------------------------------ greedy log-det ----
def _objective(U, w, C):
    A = np.eye(U.shape[1]) + sum((w[i] * np.outer(U[i], U[i]) for i in C), np.zeros((U.shape[1],) * 2))
    return np.linalg.slogdet(A)[1]


def test_greedy_first_pick_maximises_w_norm2():
    # with A = I the gain log(1 + w ||u||^2) is monotone in w ||u||^2
    r = rng(8)
    U = r.normal(size=(20, 4))
    w = r.random(20)
    idx, _ = J.greedy_logdet_select(U, w, 1)
    assert idx[0] == int(np.argmax(w * (U * U).sum(axis=1)))


def test_greedy_objective_increments_follow_the_determinant_lemma():
    r = rng(9)
    U = r.normal(size=(15, 5))
    w = r.random(15) * 2
    idx, obj = J.greedy_logdet_select(U, w, 6)
    for k in range(len(idx)):
        np.testing.assert_allclose(obj[k], _objective(U, w, idx[: k + 1]), rtol=1e-10, atol=1e-12)


def test_greedy_is_optimal_for_orthogonal_values():
    # orthogonal u: the objective is sum log(1 + w_i ||u_i||^2) over C, so the
    # best set is the B largest w ||u||^2 -- brute force agrees
    r = rng(10)
    d = n = 6
    Q, _ = np.linalg.qr(r.normal(size=(d, d)))
    U = Q * r.random(n)[:, None] * 3
    w = r.random(n)
    for B in (1, 2, 3):
        idx, obj = J.greedy_logdet_select(U, w, B)
        best = max(_objective(U, w, C) for C in itertools.combinations(range(n), B))
        np.testing.assert_allclose(obj[-1], best, rtol=1e-12)
        assert set(idx) == set(np.argsort(-(w * (U * U).sum(axis=1)))[:B])


def test_greedy_never_beats_brute_force_and_reaches_a_known_bound():
    # submodular maximisation: greedy >= (1 - 1/e) * optimum gain over I
    r = rng(11)
    n, d, B = 9, 3, 4
    U = r.normal(size=(n, d))
    w = r.random(n) * 3
    _, obj = J.greedy_logdet_select(U, w, B)
    best = max(_objective(U, w, C) for C in itertools.combinations(range(n), B))
    assert obj[-1] <= best + 1e-12
    assert obj[-1] >= (1 - 1 / math.e) * best - 1e-12


def test_greedy_tie_goes_to_the_lower_index():
    U = np.eye(3)[[0, 0, 1]]
    w = np.ones(3)
    idx, _ = J.greedy_logdet_select(U, w, 2)
    assert list(idx) == [0, 2]


def test_full_covariance_unit_weight_composes_rho_and_logit_variance():
    # Eq. 8 with R14: w_i = (1/d) sum_h rho_h,i^2 var_j(q_h,j . k_i), the pool
    # attention taken from scipy's softmax at temperature tau sqrt(d)
    from scipy.special import softmax

    r = rng(12)
    n, d, G, wq, tau = 50, 8, 2, 5, 2.0
    K = r.normal(size=(n, d)) * 2
    q = r.normal(size=(G, wq, d)) @ r.normal(size=(d, d))
    ref = np.zeros(n)
    for h in range(G):
        a = softmax(K @ q[h].mean(axis=0) / (tau * math.sqrt(d)))
        ref += (a * (1 - a)) ** 2 * np.var(q[h] @ K.T, axis=0) / d
    w = J.unit_weights(K, q, J.JacapParams(tau=tau, full_covariance=True))
    np.testing.assert_allclose(w, ref, rtol=1e-11)
    assert FULL.full_covariance and not FULL.linear_weighting


# -------------------------------------------------- R15 output directions ----
def _unit(seed, n=60, d=16, G=2, wq=6):
    r = rng(seed)
    K = r.normal(size=(n, d)) * 2
    V = r.normal(size=(n, d)) * r.lognormal(size=d)
    q = r.normal(size=(G, wq, d))
    return K, V, q


def test_output_directions_reduce_to_a_d_by_d_problem():
    # push-through identity: with W = Q R (Q orthonormal columns),
    # u^T (I + sum w u u^T)^{-1} u = (R v)^T (I + R G R^T)^{-1} (R v), G = sum w v v^T,
    # i.e. the d_o x d_o problem equals a d x d one -- checked against the
    # oracle's explicit d_o-dimensional computation
    K, V, q = _unit(13)
    d, do = V.shape[1], 48
    W = rng(14).normal(size=(do, d))
    ora = J.oracle_unit(q, K, V, 8, out_proj=W)
    w = J.unit_weights(K, q)
    _, R = np.linalg.qr(W)
    G = (V * w[:, None]).T @ V
    M = np.eye(d) + R @ G @ R.T
    Lm = np.linalg.cholesky(M)
    Y = np.linalg.solve(Lm, R @ V.T)
    np.testing.assert_allclose(ora["scores"], w * (Y * Y).sum(axis=0), rtol=1e-9)
    assert ora["A"].shape == (do, do)


def test_orthonormal_output_map_leaves_scores_unchanged():
    # W with orthonormal columns (W^T W = I) is a rotation into a larger space:
    # the scores equal those of the u = v proxy
    K, V, q = _unit(15)
    Q, _ = np.linalg.qr(rng(16).normal(size=(40, V.shape[1])))
    np.testing.assert_allclose(J.oracle_unit(q, K, V, 8, out_proj=Q)["scores"],
                               J.oracle_unit(q, K, V, 8)["scores"], rtol=1e-10)


def test_scaled_identity_output_map_equals_scaled_values():
    # W = c I: u = c v, so the scores equal those computed on c V
    K, V, q = _unit(17)
    c = 2.5
    np.testing.assert_allclose(J.oracle_unit(q, K, V, 8, out_proj=c * np.eye(V.shape[1]))["scores"],
                               J.oracle_unit(q, K, c * V, 8)["scores"], rtol=1e-11)
