"""Float64 restatements of the paper's theory, used only to pin the oracle.

TEST INFRASTRUCTURE (same import rule as ``jacap_oracle``): only tests,
``__graft_entry__.smoke()`` and ``bench.py``'s CPU legs may use it.

* ``retained_map``       f_C(q) = U_C softmax(K_C q / sqrt(d_k))      (Eq. 3)
* ``retained_jacobian``  J_C = U_C S_C K_C / sqrt(d_k)                (Lemma 1, Eq. 6)
* ``jacobian_capacity``  1/2 logdet(I + Sigma^{-1} J_C Lambda J_C^T)  (Theorem 1, Eq. 7)
* ``approx_capacity``    1/2 logdet(I + sum_{i in C} w_i u_i u_i^T)   (App. B.1, the
                          objective left after both diagonal approximations)
* ``brute_force_best``   exhaustive maximisation over all subsets of size B.

Here the columns of U_C are output directions u_i (d_o each); the code keeps
tokens on the first axis, so ``U`` is (n, d_o) and ``K`` is (n, d_k).
"""

from __future__ import annotations

import itertools
import math

import numpy as np


def _f64(x):
    return np.asarray(x, dtype=np.float64)


def retained_map(U, K, q):
    """f_C(q) = U_C softmax(K_C q / sqrt(d_k)) (Eq. 3). Returns (d_o,)."""
    U, K, q = _f64(U), _f64(K), _f64(q)
    s = K @ q / math.sqrt(K.shape[1])
    a = np.exp(s - s.max())
    a = a / a.sum()
    return U.T @ a


def retained_jacobian(U, K, mu):
    """J_C = U_C S_C K_C / sqrt(d_k), S_C = Diag(a*) - a* a*^T (Lemma 1, Eq. 6)."""
    U, K, mu = _f64(U), _f64(K), _f64(mu)
    s = K @ mu / math.sqrt(K.shape[1])
    a = np.exp(s - s.max())
    a = a / a.sum()
    S = np.diag(a) - np.outer(a, a)
    return U.T @ S @ K / math.sqrt(K.shape[1])


def jacobian_capacity(U, K, mu, Lam, noise=None):
    """1/2 logdet(I + Sigma_noise^{-1} J_C Lambda_Q J_C^T) (Theorem 1, Eq. 7)."""
    J = retained_jacobian(U, K, mu)
    Lam = _f64(Lam)
    if Lam.ndim == 1:
        Lam = np.diag(Lam)
    d_o = J.shape[0]
    Sig = np.eye(d_o) if noise is None else _f64(noise)
    M = np.eye(d_o) + np.linalg.solve(Sig, J @ Lam @ J.T)
    sign, logdet = np.linalg.slogdet(M)
    assert sign > 0
    return 0.5 * logdet


def approx_capacity(U, w):
    """1/2 logdet(I + sum_i w_i u_i u_i^T) over the given rows (App. B.1)."""
    U, w = _f64(U), _f64(w)
    M = np.eye(U.shape[1]) + (U * w[:, None]).T @ U
    sign, logdet = np.linalg.slogdet(M)
    assert sign > 0
    return 0.5 * logdet


def brute_force_best(n: int, budget: int, objective):
    """Best subset of size ``budget`` of range(n) for ``objective(tuple)``.

    Returns (best_value, list of all subsets reaching it within 1e-12 relative).
    """
    best, arg = None, []
    for C in itertools.combinations(range(n), budget):
        val = objective(C)
        if best is None or val > best + 1e-12 * max(1.0, abs(best)):
            best, arg = val, [C]
        elif abs(val - best) <= 1e-12 * max(1.0, abs(best)):
            arg.append(C)
    return best, arg
