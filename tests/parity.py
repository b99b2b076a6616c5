"""Comparison rules between the CUDA path and the float64 oracle.

* scores (float32 on the GPU): |g - o| <= 1e-3 |o| + 1e-9 max_unit |o|; the
  floor keeps scores that underflow far below the unit's scale from failing.
* TOP-B index sets: the GPU set may differ from the oracle's only by tokens
  whose oracle score lies within rel 1e-5 of the oracle's B-th score (near
  ties decided by fp32 rounding); the GPU list must be ascending, unique and
  in range, and hold min(n, B) entries followed by -1.
* compacted K / V: bit-identical to the source rows at the GPU's positions.
"""

import numpy as np
import torch

SCORE_RTOL = 1e-3
SCORE_FLOOR = 1e-9
TIE_RTOL = 1e-5


def assert_scores_close(gpu, ora, what="scores"):
    gpu = np.asarray(gpu, dtype=np.float64)
    ora = np.asarray(ora, dtype=np.float64)
    assert gpu.shape == ora.shape, (gpu.shape, ora.shape)
    if ora.size == 0:
        return
    scale = np.max(np.abs(ora))
    tol = SCORE_RTOL * np.abs(ora) + SCORE_FLOOR * scale
    err = np.abs(gpu - ora)
    bad = np.nonzero(err > tol)[0]
    assert bad.size == 0, (
        f"{what}: {bad.size}/{ora.size} outside tolerance; worst rel "
        f"{np.max(err / np.maximum(np.abs(ora), 1e-300)):.3e} at {bad[:5]} gpu={gpu[bad[:5]]} ora={ora[bad[:5]]}")


def assert_selection(gpu_idx, n, budget, ora_scores, ora_idx):
    gpu_idx = np.asarray(gpu_idx)
    kept = min(n, budget)
    assert np.all(gpu_idx[kept:] == -1), "padding must be -1"
    sel = gpu_idx[:kept]
    assert np.all(sel >= 0) and np.all(sel < n), "indices out of range"
    assert np.all(np.diff(sel) > 0), "indices must be strictly ascending"
    ora_sel = np.asarray(ora_idx)[:kept]
    diff = set(sel.tolist()) ^ set(ora_sel.tolist())
    if not diff:
        return
    s = np.asarray(ora_scores, dtype=np.float64)
    b_th = np.sort(s)[::-1][kept - 1]
    for i in diff:
        assert abs(s[i] - b_th) <= TIE_RTOL * abs(b_th), (
            f"token {i} differs between GPU and oracle sets; oracle score {s[i]!r} vs B-th {b_th!r}")


def assert_rows_bitwise(src_rows: torch.Tensor, out_rows: torch.Tensor):
    a = src_rows.contiguous().view(torch.uint8).cpu().numpy()
    b = out_rows.contiguous().view(torch.uint8).cpu().numpy()
    assert a.shape == b.shape and np.array_equal(a, b), "compacted rows are not bit-identical"


def gpu_selection_properties(scores: torch.Tensor, idx: torch.Tensor, kept: torch.Tensor, seqlens, budget):
    """Full-size checks of the GPU's own selection against the GPU's scores.

    For every unit: chosen positions ascending and unique; every chosen score
    >= every other score; among tokens equal to the smallest chosen score the
    chosen ones are the lowest positions.
    """
    L, Hkv, N = scores.shape
    cu = np.concatenate([[0], np.cumsum(seqlens)])
    assert kept.cpu().tolist() == [min(n, budget) for n in seqlens]
    for s, n in enumerate(seqlens):
        k = min(n, budget)
        sc = scores[:, :, cu[s]:cu[s + 1]].reshape(L * Hkv, n)
        ix = idx[:, :, s, :].reshape(L * Hkv, budget).long()
        assert bool((ix[:, k:] == -1).all())
        sel = ix[:, :k]
        assert bool((sel >= 0).all()) and bool((sel < n).all())
        if k > 1:
            assert bool((sel[:, 1:] > sel[:, :-1]).all())
        if k == n:
            continue
        chosen = torch.gather(sc, 1, sel)
        thr = chosen.min(dim=1).values
        mask = torch.ones_like(sc, dtype=torch.bool)
        mask.scatter_(1, sel, False)
        other = torch.where(mask, sc, torch.full_like(sc, -1.0))
        assert bool((other.max(dim=1).values <= thr).all()), "a dropped token outscores a kept one"
        # ties at the threshold: kept ones must be the lowest positions
        pos = torch.arange(n, device=sc.device).expand_as(sc)
        tie_unkept = torch.where(mask & (sc == thr[:, None]), pos, torch.full_like(pos, n))
        tie_kept = torch.where(~mask & (sc == thr[:, None]), pos, torch.full_like(pos, -1))
        assert bool((tie_kept.max(dim=1).values < tie_unkept.min(dim=1).values).all())
