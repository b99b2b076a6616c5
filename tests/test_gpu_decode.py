"""GPU parity of decoding-stage eviction (reading R16) against the oracle.

A synthetic decode stream: the workload generator's cache rows n0 .. n0+T-1
of a request are the tokens its decode steps append, and its window queries
w .. w+T-1 are their queries (the first w are the prefill window). At every
eviction the slot is read back before the library touches it; the GPU's
scores and kept set are compared with ``oracle_unit`` on that exact cache
with the whole query history (so a near tie settled differently earlier
cannot make later comparisons fail), the in-place compaction bit for bit, the
running statistics with numpy moments of the history, and the eviction steps
with ``decode_run``'s schedule.
"""

import ctypes

import numpy as np
import pytest
import torch

from oracle import JacapParams, oracle_unit
from oracle.decode_oracle import decode_run
from paper_2609_08131_gb300 import jacap_params
from paper_2609_08131_gb300.api import Cache, DecodeEvictor, Evictor
from paper_2609_08131_gb300.workloads import Workload, generate

from parity import assert_rows_bitwise, assert_scores_close, assert_selection

pytestmark = pytest.mark.gpu

DEV = "cuda:0"

CASES = {
    # name: (layers, Hq, Hkv, prefill lengths, window, steps, budget, interval, dtype, params, seed, preserve_order)
    "bf16_gqa4": (2, 8, 2, (40, 63), 8, 70, 48, 16, "bf16", jacap_params(), 31, False),
    "bf16_gqa4_ordered": (2, 8, 2, (40, 63), 8, 70, 48, 16, "bf16", jacap_params(), 31, True),
    "bf16_gqa2_interval1": (1, 4, 2, (30,), 4, 12, 32, 1, "bf16", jacap_params(tau=2.0), 32, False),
    "f32_mha_unbiased": (1, 4, 4, (10, 24), 4, 30, 20, 5, "f32", jacap_params(cov_unbiased=1, tau=3.0), 33, False),
    "f32_mha_unbiased_ordered": (1, 4, 4, (10, 24), 4, 30, 20, 5, "f32", jacap_params(cov_unbiased=1, tau=3.0), 33,
                                 True),
    "bf16_gqa8_long_slot": (1, 8, 1, (700,), 16, 40, 512, 200, "bf16", jacap_params(), 34, False),
    "bf16_gqa8_long_slot_ordered": (1, 8, 1, (700,), 16, 40, 512, 200, "bf16", jacap_params(), 34, True),
    # Nemotron-7B's heads (28 q / 4 kv, G = 7), the paper's decoding-stage model
    "bf16_gqa7_nemotron_heads": (2, 28, 4, (50, 45), 8, 60, 40, 16, "bf16", jacap_params(), 35, False),
    "f32_gqa5_ordered": (1, 10, 2, (30,), 4, 25, 24, 8, "f32", jacap_params(tau=2.0), 36, True),
}


def _arrangement(gidx, B, preserve_order):
    """Slot row r after the compaction holds pre-compaction row out[r]."""
    kept = [int(x) for x in gidx[:B]]
    if preserve_order:
        return kept
    out = list(range(B))
    front = {x for x in kept if x < B}
    holes = [r for r in range(B) if r not in front]
    back = [x for x in kept if x >= B]
    assert len(holes) == len(back)
    for r, x in zip(holes, back):
        out[r] = x
    return out


def _oracle_params(p):
    return JacapParams(tau=p.tau, weight_div_dk=bool(p.weight_div_dk), cov_unbiased=bool(p.cov_unbiased),
                       linear_weighting=bool(p.linear_weighting))


@pytest.mark.parametrize("name", list(CASES))
def test_decode_evictions_match_the_oracle_event_by_event(name):
    L, Hq, Hkv, n0s, w, T, B, D, dtype, params, seed, ordered = CASES[name]
    S, G, cap = len(n0s), Hq // Hkv, B + D
    wl = Workload("decode stream", L, Hq, Hkv, tuple(n + T for n in n0s), w + T, B, dtype=dtype, seed=seed)
    t = generate(wl, DEV)
    cu = t.cu_seqlens.cpu().tolist()
    tdt = t.k.dtype
    k0 = torch.zeros((S, L, Hkv, max(n0s), 128), dtype=tdt, device=DEV)
    v0 = torch.zeros_like(k0)
    for s, n in enumerate(n0s):
        k0[s, :, :, :n] = t.k[:, :, cu[s]:cu[s] + n]
        v0[s, :, :, :n] = t.v[:, :, cu[s]:cu[s] + n]
    ev = DecodeEvictor(S, L, Hq, Hkv, B, D, dtype=tdt, params=params, device=DEV, preserve_order=ordered)
    ev.start(k0, v0, t.q_win[:, :, :, :w].contiguous(), list(n0s))
    q_all = t.q_win.double().cpu().numpy()  # [S, L, Hq, w + T, d]
    P = _oracle_params(params)
    event_steps = {s: [] for s in range(S)}
    for step in range(T):
        rows = [cu[s] + n0s[s] + step for s in range(S)]
        k_new = torch.stack([t.k[:, :, r] for r in rows])
        v_new = torch.stack([t.v[:, :, r] for r in rows])
        q_new = t.q_win[:, :, :, w + step].contiguous()
        for s in ev.append(k_new, v_new, q_new):
            event_steps[s].append(step)
            kb, vb, pb = ev.k[s].clone(), ev.v[s].clone(), ev.pos[s].cpu().numpy()
            nq = w + step + 1
            # running statistics = moments of the whole history
            stats = ev.stats[s].double().cpu().numpy()
            assert (ev.counts[s].cpu().numpy() == nq).all()
            hist = q_all[s, :, :, :nq]
            scale = np.abs(hist).max()
            np.testing.assert_allclose(stats[:, :, 0], hist.mean(axis=2), rtol=1e-4, atol=1e-5 * scale)
            np.testing.assert_allclose(stats[:, :, 1] / nq, hist.var(axis=2), rtol=1e-4, atol=1e-6 * scale * scale)
            ev.evict(s)
            ev.check()
            for layer in range(L):
                for g in range(Hkv):
                    K = kb[layer, g].double().cpu().numpy()
                    V = vb[layer, g].double().cpu().numpy()
                    ora = oracle_unit(hist[layer, g * G:(g + 1) * G], K, V, B, P)
                    assert_scores_close(ev.scores[layer, g].double().cpu().numpy(), ora["scores"],
                                        f"event {step} request {s} unit ({layer}, {g})")
                    gidx = ev.idx[layer, g, 0].cpu().numpy()
                    assert_selection(gidx, cap, B, ora["scores"], ora["idx"])
                    sel = torch.as_tensor(_arrangement(gidx, B, ordered), dtype=torch.long, device=DEV)
                    after_k, after_v = ev.k[s, layer, g], ev.v[s, layer, g]
                    assert_rows_bitwise(kb[layer, g][sel], after_k[:B])
                    assert_rows_bitwise(vb[layer, g][sel], after_v[:B])
                    assert_rows_bitwise(kb[layer, g][B:], after_k[B:])  # the free rows are left alone
                    assert_rows_bitwise(vb[layer, g][B:], after_v[B:])
                    np.testing.assert_array_equal(ev.pos[s, layer, g, :B].cpu().numpy(), pb[layer, g][sel.cpu().numpy()])
                    assert sorted(sel.tolist()) == [int(x) for x in gidx[:B]]
    # the schedule of every request is decode_run's (it does not depend on scores)
    for s in range(S):
        r = cu[s]
        Kr = t.k[0, 0, r:r + n0s[s] + T].double().cpu().numpy()
        Vr = t.v[0, 0, r:r + n0s[s] + T].double().cpu().numpy()
        steps = [(q_all[s, 0, :G, w + j], Kr[n0s[s] + j], Vr[n0s[s] + j]) for j in range(T)]
        events, ids, _, _ = decode_run(q_all[s, 0, :G, :w], Kr[:n0s[s]], Vr[:n0s[s]], steps, B, D, P)
        assert [e["step"] for e in events] == event_steps[s]
        assert ev.lengths[s] == len(ids)
    assert ev.events == sum(len(v) for v in event_steps.values()) > 0


@pytest.mark.parametrize("ordered", [False, True])
def test_requests_that_fill_together_are_evicted_in_one_pass(ordered):
    # three of four requests start with equal prefills, so they fill on the same
    # decode step; the neighbouring two of them (0, 1) share one pass, request
    # 3 gets its own, and request 2 fills alone five steps earlier. Every unit
    # of every request is checked against the oracle
    # on the exact slot contents before the eviction, and the tags move with
    # the rows.
    L, Hq, Hkv, B, D, w, T = 2, 12, 2, 40, 16, 8, 20
    n0s = (40, 40, 45, 40)
    S, G, cap = len(n0s), Hq // Hkv, B + D
    wl = Workload("decode batch", L, Hq, Hkv, tuple(n + T for n in n0s), w + T, B, seed=37)
    t = generate(wl, DEV)
    cu = t.cu_seqlens.cpu().tolist()
    k0 = torch.zeros((S, L, Hkv, max(n0s), 128), dtype=t.k.dtype, device=DEV)
    v0 = torch.zeros_like(k0)
    for s, n in enumerate(n0s):
        k0[s, :, :, :n] = t.k[:, :, cu[s]:cu[s] + n]
        v0[s, :, :, :n] = t.v[:, :, cu[s]:cu[s] + n]
    ev = DecodeEvictor(S, L, Hq, Hkv, B, D, dtype=t.k.dtype, device=DEV, preserve_order=ordered)
    ev.start(k0, v0, t.q_win[:, :, :, :w].contiguous(), list(n0s))
    q_all = t.q_win.double().cpu().numpy()
    P = JacapParams()
    batched = 0
    for step in range(T):
        rows = [cu[s] + n0s[s] + step for s in range(S)]
        k_new = torch.stack([t.k[:, :, r] for r in rows])
        v_new = torch.stack([t.v[:, :, r] for r in rows])
        full = ev.append(k_new, v_new, t.q_win[:, :, :, w + step].contiguous())
        if not full:
            continue
        before = {s: (ev.k[s].clone(), ev.v[s].clone(), ev.pos[s].clone()) for s in full}
        runs = []  # the groups evict_many forms: maximal runs of neighbouring requests
        for s in full:
            if runs and runs[-1][-1] == s - 1:
                runs[-1].append(s)
            else:
                runs.append([s])
        for run in runs:
            # one run per call, so the scores and positions of each pass can be read
            assert ev.evict_many(run) == [(run[0], run[-1] + 1)]
            a, b = run[0], run[-1] + 1
            ev.check()
            batched += b - a > 1
            for j, s in enumerate(range(a, b)):
                kb, vb, pb = before[s]
                hist = q_all[s, :, :, :w + step + 1]
                for layer in range(L):
                    for g in range(Hkv):
                        K = kb[layer, g].double().cpu().numpy()
                        V = vb[layer, g].double().cpu().numpy()
                        ora = oracle_unit(hist[layer, g * G:(g + 1) * G], K, V, B, P)
                        sc = ev.scores[layer, g, j * cap:(j + 1) * cap].double().cpu().numpy()
                        assert_scores_close(sc, ora["scores"], f"step {step} request {s} unit ({layer}, {g})")
                        gidx = ev.idx[layer, g, j].cpu().numpy()
                        assert_selection(gidx, cap, B, ora["scores"], ora["idx"])
                        sel = torch.as_tensor(_arrangement(gidx, B, ordered), dtype=torch.long, device=DEV)
                        assert_rows_bitwise(kb[layer, g][sel], ev.k[s, layer, g, :B])
                        assert_rows_bitwise(vb[layer, g][sel], ev.v[s, layer, g, :B])
                        assert torch.equal(pb[layer, g][sel], ev.pos[s, layer, g, :B])
    assert batched >= 1 and ev.events > ev.passes


def test_compaction_refuses_positions_that_do_not_ascend():
    # a hand-made index list with a repeat: the unit is left untouched and the
    # status word says invalid argument (no out-of-range access is possible:
    # the positions are checked before any row moves)
    from paper_2609_08131_gb300 import JACAP_ERR_INVALID_ARG, jacap_compact_inplace, jacap_device_status
    from paper_2609_08131_gb300.api import _ptr, _stream

    ev = DecodeEvictor(1, 1, 2, 2, 4, 4, dtype=torch.bfloat16, device=DEV)
    ev.k.normal_()
    ev.v.normal_()
    before = ev.k.clone()
    ev.idx[:] = torch.tensor([0, 2, 2, 5], dtype=torch.int32, device=DEV)
    for ordered in (0, 1):
        ev.ws.zero_()
        st = jacap_compact_inplace(ev.slot, _ptr(ev.k[0]), _ptr(ev.v[0]), _ptr(ev.pos[0]), _ptr(ev.idx), 4, ordered,
                                   _ptr(ev.ws), ev.ws.numel(), _stream())
        assert st == 0
        assert jacap_device_status(_ptr(ev.ws), _stream()) == JACAP_ERR_INVALID_ARG
        assert torch.equal(ev.k, before)


def test_host_evictor_matches_the_oracle():
    # a cache in pinned host memory, evicted through jacap_evict_host in layer
    # groups of 2 through two device buffers (the groups' copies overlap the
    # previous group's pass); positions and retained rows come back to the host
    from oracle import JacapParams as JP
    from paper_2609_08131_gb300.api import HostEvictor
    from paper_2609_08131_gb300.workloads import unit_arrays

    wl = Workload("host cache", 5, 8, 2, (900, 333), 16, 64, seed=41)
    t = generate(wl, DEV)
    he = HostEvictor(t.q_win.cpu().pin_memory(), t.k.cpu().pin_memory(), t.v.cpu().pin_memory(),
                     t.cu_seqlens, list(wl.seqlens), wl.num_q_heads, wl.budget, jacap_params(),
                     group_layers=2, device=DEV)
    first = None
    for _ in range(2):  # the second run reuses the buffers and must repeat the first bit for bit
        he.idx_h.fill_(-7)
        he.k_out_h.fill_(3)
        he.run()
        if first is None:
            first = (he.idx_h.clone(), he.k_out_h.clone(), he.v_out_h.clone())
    assert torch.equal(first[0], he.idx_h)
    assert_rows_bitwise(first[1], he.k_out_h)
    assert_rows_bitwise(first[2], he.v_out_h)
    cu = t.cu_seqlens.cpu().tolist()
    assert he.kept_h.tolist() == [min(n, wl.budget) for n in wl.seqlens]
    for layer in range(wl.num_layers):
        for g in range(wl.num_kv_heads):
            for s in range(len(wl.seqlens)):
                q, K, V = unit_arrays(t, wl.num_q_heads, s, layer, g)
                ora = oracle_unit(q, K, V, wl.budget, JP())
                gidx = he.idx_h[layer, g, s].numpy()
                assert_selection(gidx, cu[s + 1] - cu[s], wl.budget, ora["scores"], ora["idx"])
                kept = min(cu[s + 1] - cu[s], wl.budget)
                sel = torch.as_tensor(gidx[:kept], dtype=torch.long)
                assert_rows_bitwise(t.k[layer, g, cu[s]:cu[s + 1]].cpu()[sel], he.k_out_h[layer, g, s, :kept])
                assert_rows_bitwise(t.v[layer, g, cu[s]:cu[s + 1]].cpu()[sel], he.v_out_h[layer, g, s, :kept])
                assert bool((he.k_out_h[layer, g, s, kept:] == 0).all())


def test_host_evictor_positions_only_on_one_stream():
    # copy_rows off and a single stream (no copy stream): positions only, in order
    from paper_2609_08131_gb300 import jacap_evict_host
    from paper_2609_08131_gb300.api import HostEvictor, _ptr, _stream

    wl = Workload("host cache", 3, 12, 2, (500, 77, 640), 8, 48, seed=42)
    t = generate(wl, DEV)
    he = HostEvictor(t.q_win.cpu().pin_memory(), t.k.cpu().pin_memory(), t.v.cpu().pin_memory(),
                     t.cu_seqlens, list(wl.seqlens), wl.num_q_heads, wl.budget, jacap_params(tau=2.0),
                     group_layers=2, device=DEV, copy_rows=False)
    assert he.d2h_bytes == (he.idx_h.numel() + he.kept_h.numel()) * 4
    he.run()
    two = he.idx_h.clone()
    st = jacap_evict_host(he.lay, he.params, he.budget, he.gl, _ptr(he.q_h), _ptr(he.k_h), _ptr(he.v_h),
                          ctypes.c_void_p(0), _ptr(he.idx_h), _ptr(he.kept_h), ctypes.c_void_p(0),
                          ctypes.c_void_p(0), _ptr(he.dev_buf), he.dev_buf.numel(), _stream(), ctypes.c_void_p(0))
    assert st == 0
    assert torch.equal(two, he.idx_h)
    dev = Evictor(Cache(t.q_win, t.k, t.v, t.cu_seqlens, t.seqlens, wl.num_q_heads), wl.budget,
                  jacap_params(tau=2.0))
    dev.run()
    a, b = he.idx_h.reshape(-1, wl.budget).numpy(), dev.idx.cpu().reshape(-1, wl.budget).numpy()
    assert sum(len(np.setdiff1d(x, y)) for x, y in zip(a, b)) <= 2


def test_many_slots_fill_their_holes_with_the_small_selection_ctas():
    # an eviction of one request's slot covers 24 layers x 8 KV heads = 192
    # units (more than the SMs) of 200 tokens: the selection with the hole
    # filling runs 256-thread CTAs; each unit's compaction is checked against
    # the positions it selected
    L, Hq, Hkv, S, B, D = 24, 16, 8, 2, 160, 40
    wl = Workload("decode many", L, Hq, Hkv, (B + D,) * S, 8, B, seed=47)
    t = generate(wl, DEV)
    cu = t.cu_seqlens.cpu().tolist()
    ev = DecodeEvictor(S, L, Hq, Hkv, B, D, dtype=t.k.dtype, device=DEV)
    assert L * Hkv > torch.cuda.get_device_properties(0).multi_processor_count
    n0 = B + D - 1
    k0 = torch.stack([t.k[:, :, cu[s]:cu[s] + n0] for s in range(S)])
    v0 = torch.stack([t.v[:, :, cu[s]:cu[s] + n0] for s in range(S)])
    ev.start(k0, v0, t.q_win.contiguous(), [n0] * S)
    k_new = torch.stack([t.k[:, :, cu[s] + n0] for s in range(S)])
    v_new = torch.stack([t.v[:, :, cu[s] + n0] for s in range(S)])
    full = ev.append(k_new, v_new, t.q_win[:, :, :, -1].contiguous())
    assert sorted(full) == list(range(S))
    for s in range(S):
        kb, vb = ev.k[s].clone(), ev.v[s].clone()
        ev.evict(s)
        ev.check()
        for layer in (0, 5, 11, 23):
            for g in (0, 3, 7):
                gidx = ev.idx[layer, g, 0].cpu().numpy()
                assert list(gidx) == sorted(set(int(x) for x in gidx)) and 0 <= gidx[0] and gidx[-1] < B + D
                sel = torch.as_tensor(_arrangement(gidx, B, False), dtype=torch.long, device=DEV)
                assert_rows_bitwise(kb[layer, g][sel], ev.k[s, layer, g, :B])
                assert_rows_bitwise(vb[layer, g][sel], ev.v[s, layer, g, :B])
