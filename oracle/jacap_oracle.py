"""Float64 CPU oracle for Jacap's prefill-time eviction pass.

TEST INFRASTRUCTURE. Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import this
module. The CUDA path never calls it, shares no code with it and does not
import it; the oracle never imports the CUDA path either.

It is a plain, slow, one-unit-at-a-time restatement of Algorithm 1 (Sec. 3.4)
in float64 numpy. A *unit* is one (request, layer, KV head). For a unit with
keys K (n x d), values V (n x d) and the window queries of the G query heads
that share its KV head, the pass computes, in the paper's order and notation:

1. query statistics mu_Q and a diagonal Lambda_Q for every query head
   (Sec. 3.4 last paragraph: estimated from observed queries; App. B.2:
   Lambda_Q is diagonal in practice);
2. the pool attention alpha_bar_i = softmax_i(k_i^T mu_Q / (tau sqrt(d_k)))
   over every cached token (Sec. 3.4, display after Algorithm 1; Alg. 1 step 1);
3. rho_i = alpha_bar_i (1 - alpha_bar_i) (Sec. 3.4 diagonal approximation of
   S_C) and kappa_i = k_i^T Lambda_Q k_i (Sec. 3.4, query-response variance);
4. w_i = rho_i^2 kappa_i / d_k (Eq. 8), summed over the G query heads of the
   group (reading R5, stated below);
5. A_Jac = I + sum_j w_j u_j u_j^T with u_j = v_j (Eq. 9; u = v proxy from the
   last paragraph of Sec. 3.4);
6. r_i = w_i u_i^T A_Jac^{-1} u_i (Eq. 10; Alg. 1 step 4);
7. the TOP-B indices by score (Alg. 1 step 5), and the retained cache
   Z_C = {(k_i, v_i)}_{i in C} (Sec. 3.1).

Readings of points where the paper is silent or inconsistent (each is a
switch so the alternatives stay testable):

* R1  the 1/d_k factor of Eq. 8 is kept (Alg. 1 step 2 omits it);
      ``weight_div_dk=False`` drops it.
* R2  the ridge I of Eq. 9 is kept; ``ridge=False`` uses the pseudo-inverse
      of sum_j w_j u_j u_j^T (used only by the rank pin).
* R3  logits are divided by tau * sqrt(d_k); default tau = 10 (Sec. 4.4
      ablation: best around 10).
* R4  mu_Q is the mean of the last w queries of each query head and Lambda_Q
      their per-channel population variance (divide by w);
      ``cov_unbiased=True`` divides by w - 1.
* R5  a KV head shared by G query heads (GQA) gets w_i = sum over the G heads
      of that head's Eq. 8 weight. Query head h belongs to KV head h // G.
* R6  the candidate pool is every cached token of the unit (no causal mask,
      no forced retention).
* R7  TOP-B orders by score descending, then by index ascending; the chosen
      indices are returned in ascending order.
* R8  when n <= B every token is kept (kept = n) and the index list is padded
      with -1 up to B.
* R10 Sigma_noise = I (isotropic noise with sigma^2 absorbed, App. B.1).
* R13 ``linear_weighting=True`` replaces S_C by the identity, the linear
      Gaussian surrogate the paper contrasts Jacap with (App. A, end of the
      discussion of S_C): rho_i = 1, so w_i = kappa_i / d_k.
* R14 ``full_covariance=True`` uses the full window covariance Lambda_Q (the
      O(N d^2) variant of App. B.2's complexity analysis) instead of its
      diagonal: kappa_i = k_i^T Lambda_Q k_i, Lambda_Q = (1/w) sum_j
      (q_j - mu)(q_j - mu)^T (1/(w-1) with ``cov_unbiased``).

* R15 true output directions (Sec. 3.1: u_i = W_O v_i; Sec. 3.4 uses v_i as a
      proxy): ``oracle_unit(..., out_proj=W)`` takes one output map W
      (d_o x d) per unit -- for a KV head shared by G query heads the caller
      chooses how the heads' W_O slices combine (e.g. stacked) -- and uses
      u_i = W v_i in A = I + sum_j w_j u_j u_j^T (d_o x d_o) and in the score.

Also here, as a quality reference only (no GPU counterpart):
``greedy_logdet_select`` picks B tokens one at a time, each maximising the
increase of the App. B.1 objective log det(I + sum_{i in C} w_i u_i u_i^T).
"""

from __future__ import annotations

import math
from dataclasses import dataclass

import numpy as np


@dataclass(frozen=True)
class JacapParams:
    """Switches for the readings R1-R4, R13, R14 above; defaults are the method's."""

    tau: float = 10.0
    weight_div_dk: bool = True
    ridge: bool = True
    cov_unbiased: bool = False
    linear_weighting: bool = False
    full_covariance: bool = False


def _f64(x) -> np.ndarray:
    return np.asarray(x, dtype=np.float64)


# --------------------------------------------------------------------------
# Step 1: query statistics (Sec. 3.4 last paragraph; App. B.2 diagonal Lambda_Q)
# --------------------------------------------------------------------------
def window_stats(q_win, cov_unbiased: bool = False):
    """Mean mu_Q and diagonal covariance lambda (the diagonal of Lambda_Q).

    ``q_win`` is (w, d): the last w queries of ONE query head. Reading R4.
    """
    q = _f64(q_win)
    w = q.shape[0]
    if w < 1 or (cov_unbiased and w < 2):
        raise ValueError("window too short for the requested estimator")
    mu = q.sum(axis=0) / w
    dev = q - mu
    denom = (w - 1) if cov_unbiased else w
    lam = (dev * dev).sum(axis=0) / denom
    return mu, lam


def window_covariance(q_win, cov_unbiased: bool = False):
    """Full Lambda_Q of one query head's window (reading R14): the covariance
    of the w window queries, (w, d) in, (d, d) out."""
    q = _f64(q_win)
    w = q.shape[0]
    if w < 1 or (cov_unbiased and w < 2):
        raise ValueError("window too short for the requested estimator")
    dev = q - q.sum(axis=0) / w
    return (dev.T @ dev) / ((w - 1) if cov_unbiased else w)


# --------------------------------------------------------------------------
# Step 2: pool attention (Sec. 3.4 display after Algorithm 1; Alg. 1 step 1)
# --------------------------------------------------------------------------
def pool_attention(K, mu, tau: float):
    """alpha_bar_i = exp(k_i.mu/(tau sqrt d)) / sum_j exp(k_j.mu/(tau sqrt d)).

    The softmax runs over every token of the unit (reading R6). The common
    factor exp(-max) cancels between numerator and denominator.
    """
    K = _f64(K)
    d = K.shape[1]
    logits = (K @ _f64(mu)) / (tau * math.sqrt(d))
    e = np.exp(logits - logits.max())
    return e / e.sum()


# --------------------------------------------------------------------------
# Step 3: diagonal softmax sensitivity and query-response variance (Sec. 3.4)
# --------------------------------------------------------------------------
def sensitivity(alpha_bar):
    """rho_i = alpha_bar_i (1 - alpha_bar_i): the diagonal of S_C (Sec. 3.4)."""
    a = _f64(alpha_bar)
    return a * (1.0 - a)


def response_variance(K, lam):
    """kappa_i = k_i^T Lambda_Q k_i with Lambda_Q = Diag(lam) (Sec. 3.4, App. B.2)."""
    K = _f64(K)
    return (K * K) @ _f64(lam)


def response_variance_full(K, Lam):
    """kappa_i = k_i^T Lambda_Q k_i for a full Lambda_Q (App. B.2, reading R14)."""
    K = _f64(K)
    return np.einsum("nc,cd,nd->n", K, _f64(Lam), K)


# --------------------------------------------------------------------------
# Step 4: Jacobian importance weight (Eq. 8), GQA sum (reading R5)
# --------------------------------------------------------------------------
def head_weight(K, mu, lam, params: JacapParams = JacapParams()):
    """w_i = rho_i^2 kappa_i / d_k for one query head (Eq. 8).

    ``lam`` is the diagonal of Lambda_Q, or the full (d, d) matrix when
    ``params.full_covariance`` (R14). With ``params.linear_weighting`` S_C is
    the identity and rho_i = 1 (R13)."""
    K = _f64(K)
    d = K.shape[1]
    if params.linear_weighting:
        rho = np.ones(K.shape[0])
    else:
        rho = sensitivity(pool_attention(K, mu, params.tau))
    kappa = response_variance_full(K, lam) if params.full_covariance else response_variance(K, lam)
    w = rho * rho * kappa
    if params.weight_div_dk:
        w = w / d
    return w


def unit_weights(K, q_group, params: JacapParams = JacapParams()):
    """Weights of one unit whose KV head serves the query heads in ``q_group``.

    ``q_group`` is (G, w, d): the window queries of the G query heads mapped
    to this KV head. Returns w (n,) = sum over heads of Eq. 8 (reading R5).
    """
    K = _f64(K)
    q_group = _f64(q_group)
    w = np.zeros(K.shape[0])
    for h in range(q_group.shape[0]):
        mu, lam = window_stats(q_group[h], params.cov_unbiased)
        if params.full_covariance:
            lam = window_covariance(q_group[h], params.cov_unbiased)
        w = w + head_weight(K, mu, lam, params)
    return w


# --------------------------------------------------------------------------
# Step 5: capacity matrix (Eq. 9) and step 6: score (Eq. 10)
# --------------------------------------------------------------------------
def capacity_matrix(U, w, ridge: bool = True):
    """A_Jac = I + sum_j w_j u_j u_j^T (Eq. 9), Sigma_noise = I (reading R10)."""
    U = _f64(U)
    w = _f64(w)
    d = U.shape[1]
    A = np.zeros((d, d))
    for j in range(U.shape[0]):
        A += w[j] * np.outer(U[j], U[j])
    if ridge:
        A += np.eye(d)
    return A


def jacap_scores(U, w, ridge: bool = True):
    """r_i = w_i u_i^T A_Jac^{-1} u_i (Eq. 10) for every token of the unit."""
    U = _f64(U)
    w = _f64(w)
    A = capacity_matrix(U, w, ridge)
    if ridge:
        X = np.linalg.solve(A, U.T)  # columns A^{-1} u_i
    else:
        X = np.linalg.pinv(A) @ U.T
    quad = np.einsum("ij,ji->i", U, X)  # u_i^T A^{-1} u_i
    return w * quad


# --------------------------------------------------------------------------
# Step 7: TOP-B selection (Alg. 1 step 5) and the retained cache (Sec. 3.1)
# --------------------------------------------------------------------------
def select_topb(scores, budget: int):
    """Indices of the B largest scores, ties to the lower index (R7), ascending.

    Returns (idx, kept): idx has length ``budget`` and is padded with -1 when
    the unit has fewer than ``budget`` tokens (reading R8).
    """
    s = _f64(scores)
    n = s.shape[0]
    order = sorted(range(n), key=lambda i: (-s[i], i))
    kept = min(n, budget)
    chosen = sorted(order[:kept])
    idx = np.full(budget, -1, dtype=np.int64)
    idx[:kept] = chosen
    return idx, kept


def compact(K, V, idx, kept: int):
    """Retained cache Z_C: the rows of K and V listed in idx (Sec. 3.1)."""
    sel = np.asarray(idx[:kept], dtype=np.int64)
    return np.asarray(K)[sel], np.asarray(V)[sel]


# --------------------------------------------------------------------------
# Quality reference: greedy log-determinant selection (App. B.1 objective)
# --------------------------------------------------------------------------
def greedy_logdet_select(U, w, budget: int):
    """Greedy maximiser of log det(I + sum_{i in C} w_i u_i u_i^T) over |C| = B.

    Each round adds the token with the largest gain log(1 + w_i u_i^T A^{-1} u_i)
    (matrix determinant lemma, App. B.1), A being I plus the chosen terms so far;
    ties go to the lower index. Returns the chosen indices in pick order and the
    objective after each pick. Plain float64; a reference for selection quality,
    not part of the GPU pass.
    """
    U = _f64(U)
    w = _f64(w)
    n, d = U.shape
    A = np.eye(d)
    chosen, objective = [], []
    free = np.ones(n, dtype=bool)
    for _ in range(min(budget, n)):
        Ainv = np.linalg.inv(A)
        gain = np.full(n, -np.inf)
        q = np.einsum("nc,cd,nd->n", U, Ainv, U)
        gain[free] = np.log1p(w[free] * q[free])
        i = int(np.argmax(gain))  # first maximum: the lower index on ties
        chosen.append(i)
        free[i] = False
        A = A + w[i] * np.outer(U[i], U[i])
        objective.append(float(np.linalg.slogdet(A)[1]))
    return np.array(chosen, dtype=np.int64), np.array(objective)


# --------------------------------------------------------------------------
# Whole unit and whole cache
# --------------------------------------------------------------------------
def oracle_unit(q_group, K, V, budget: int, params: JacapParams = JacapParams(), out_proj=None):
    """Algorithm 1 for one unit; returns every intermediate the GPU exposes.

    ``out_proj`` (d_o x d) gives the output directions u_i = W v_i (R15); by
    default u_i = v_i. "A" is then d_o x d_o."""
    K64 = _f64(K)
    V64 = _f64(V)
    U64 = V64 if out_proj is None else V64 @ _f64(out_proj).T
    q_group = _f64(q_group)
    G = q_group.shape[0]
    mus, lams, alphas = [], [], []
    for h in range(G):
        mu, lam = window_stats(q_group[h], params.cov_unbiased)
        mus.append(mu)
        lams.append(lam)  # the diagonal of Lambda_Q, also under R14
        alphas.append(pool_attention(K64, mu, params.tau))
    w = unit_weights(K64, q_group, params)
    scores = jacap_scores(U64, w, params.ridge)
    idx, kept = select_topb(scores, budget)
    k_out, v_out = compact(K, V, idx, kept)
    return {
        "mu": np.stack(mus),
        "lam": np.stack(lams),
        "alpha": np.stack(alphas),
        "w": w,
        "A": capacity_matrix(U64, w, params.ridge),
        "scores": scores,
        "idx": idx,
        "kept": kept,
        "k_out": k_out,
        "v_out": v_out,
    }


def unit_views(q_win, k, v, cu_seqlens, num_q_heads: int, num_kv_heads: int, s: int, layer: int, g: int):
    """Slices of one unit from the cache layout the library uses.

    k, v: (L, Hkv, N_tot, d); q_win: (S, L, Hq, w, d); cu_seqlens: (S + 1,).
    Query head h serves KV head h // G (reading R5).
    """
    G = num_q_heads // num_kv_heads
    a, b = int(cu_seqlens[s]), int(cu_seqlens[s + 1])
    return (
        np.asarray(q_win[s, layer, g * G:(g + 1) * G]),
        np.asarray(k[layer, g, a:b]),
        np.asarray(v[layer, g, a:b]),
    )


def oracle_pass(q_win, k, v, cu_seqlens, num_q_heads: int, num_kv_heads: int, budget: int,
                params: JacapParams = JacapParams(), units=None):
    """Run Algorithm 1 over the listed units (default: all) of a cache.

    Returns {(s, layer, g): oracle_unit(...)}.
    """
    S = len(cu_seqlens) - 1
    L = k.shape[0]
    if units is None:
        units = [(s, l, g) for l in range(L) for g in range(num_kv_heads) for s in range(S)]
    out = {}
    for (s, l, g) in units:
        qg, K, V = unit_views(q_win, k, v, cu_seqlens, num_q_heads, num_kv_heads, s, l, g)
        out[(s, l, g)] = oracle_unit(qg, K, V, budget, params)
    return out
