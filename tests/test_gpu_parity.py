"""GPU parity of the CUDA eviction pass against the float64 oracle.

Every test calls the library through the C ABI (via the ctypes binding) and
compares with ``oracle.oracle_unit`` on the same bytes (the oracle reads the
device tensors back exactly). Small cases compare every unit and every
intermediate; the five evaluation configurations run at full size, in the
launch configuration bench.py times, with sampled units checked against the
oracle and size-independent properties checked on every unit.
"""

from dataclasses import replace

import numpy as np
import pytest
import torch

from oracle import JacapParams, oracle_unit
from paper_2609_08131_gb300 import jacap_params
from paper_2609_08131_gb300.api import Cache, Evictor, evict
from paper_2609_08131_gb300.workloads import Workload, config, generate, unit_arrays

from oracle_pool import run_units
from parity import assert_rows_bitwise, assert_scores_close, assert_selection, gpu_selection_properties

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


def make_cache(t, wl):
    return Cache(t.q_win, t.k, t.v, t.cu_seqlens, t.seqlens, wl.num_q_heads)


def check_unit(ev, t, wl, params, s, layer, g, check_w=True):
    q, K, V = unit_arrays(t, wl.num_q_heads, s, layer, g)
    ora = oracle_unit(q, K, V, ev.budget, JacapParams(tau=params.tau, weight_div_dk=bool(params.weight_div_dk),
                                                       cov_unbiased=bool(params.cov_unbiased),
                                                       linear_weighting=bool(params.linear_weighting),
                                                       full_covariance=bool(params.full_covariance)))
    cu = t.cu_seqlens.cpu().tolist()
    a, b = cu[s], cu[s + 1]
    n = b - a
    gs = ev.scores[layer, g, a:b].double().cpu().numpy()
    if check_w:
        gw = ev.intermediates()["weights"][layer, g, a:b].double().cpu().numpy()
        assert_scores_close(gw, ora["w"], "weights")
    assert_scores_close(gs, ora["scores"])
    gidx = ev.idx[layer, g, s].cpu().numpy()
    assert_selection(gidx, n, ev.budget, ora["scores"], ora["idx"])
    kept = min(n, ev.budget)
    sel = torch.as_tensor(gidx[:kept], dtype=torch.long, device=t.k.device)
    assert_rows_bitwise(t.k[layer, g, a:b][sel], ev.k_out[layer, g, s, :kept])
    assert_rows_bitwise(t.v[layer, g, a:b][sel], ev.v_out[layer, g, s, :kept])
    if kept < ev.budget:
        assert bool((ev.k_out[layer, g, s, kept:] == 0).all()) and bool((ev.v_out[layer, g, s, kept:] == 0).all())
    return ora


SMALL = {
    # name: (workload, params)
    "bf16_gqa4_ragged_tails": (Workload("t", 2, 8, 2, (1000, 300, 129), 16, 64, seed=11), jacap_params()),
    "bf16_mha_tau1": (Workload("t", 1, 4, 4, (777,), 8, 100, seed=12), jacap_params(tau=1.0)),
    "bf16_gqa2_peaky_tiny_seq": (Workload("t", 1, 4, 2, (500, 1, 2), 16, 32, seed=13), jacap_params(tau=0.3)),
    "bf16_gqa8_one_past_tile": (Workload("t", 1, 8, 1, (4101,), 32, 256, seed=14), jacap_params()),
    "bf16_sinks_unbiased_nodiv": (Workload("t", 1, 8, 2, (2048, 1500), 64, 200, seed=15, sink_tokens=4,
                                           sink_scale=4.0), jacap_params(tau=2.0, weight_div_dk=0, cov_unbiased=1)),
    "f32_outlier_mha": (Workload("t", 1, 4, 4, (1500, 2049), 32, 128, dtype="f32", dist="outlier", seed=16,
                                 outlier_channels=4, outlier_scale=8.0), jacap_params()),
    "f32_gqa4_peaky": (Workload("t", 2, 8, 2, (600, 130), 8, 50, dtype="f32", seed=17), jacap_params(tau=0.5)),
    "bf16_budget_exceeds_all": (Workload("t", 1, 4, 2, (100, 257), 8, 300, seed=18), jacap_params()),
    "bf16_gqa4_linear_weighting": (Workload("t", 2, 8, 2, (1500, 700), 16, 128, seed=19),
                                   jacap_params(linear_weighting=1)),
    # full-covariance kappa (App. B.2) on the tensor-core kernel
    "bf16_gqa4_full_cov_w32": (Workload("t", 2, 8, 2, (1300, 300), 32, 96, seed=22), jacap_params(full_covariance=1)),
    "bf16_gqa2_full_cov_w64_unbiased": (Workload("t", 1, 4, 2, (900, 129), 64, 64, seed=23),
                                        jacap_params(full_covariance=1, cov_unbiased=1, tau=2.0)),
    "bf16_gqa8_full_cov_w8": (Workload("t", 1, 8, 1, (700,), 8, 64, seed=24), jacap_params(full_covariance=1)),
    "bf16_gqa8_full_cov_w16": (Workload("t", 1, 16, 2, (1100, 40), 16, 64, seed=27), jacap_params(full_covariance=1)),
    # 8 centred queries per group: the image's zero padding rows
    "bf16_mha_full_cov_w8_tau1": (Workload("t", 2, 4, 4, (650, 3), 8, 32, seed=28),
                                  jacap_params(full_covariance=1, tau=1.0)),
    # ... and the CUDA-core kernel (w = 24; float32)
    "bf16_gqa4_full_cov_w24": (Workload("t", 1, 8, 2, (600, 200), 24, 64, seed=25), jacap_params(full_covariance=1)),
    "f32_gqa2_full_cov": (Workload("t", 1, 4, 2, (500,), 16, 32, dtype="f32", seed=26),
                          jacap_params(full_covariance=1)),
    "f32_mha_linear_weighting": (Workload("t", 1, 4, 4, (900,), 8, 64, dtype="f32", seed=20),
                                 jacap_params(linear_weighting=1, cov_unbiased=1)),
    # GQA ratios of the paper's other models: Qwen3-14B (40 q / 8 kv heads,
    # G = 5) and Nemotron-7B (28 q / 4 kv heads, G = 7), plus G = 3 and 6.
    # Odd G gives 8-byte aligned logits/kappa rows and 4-byte aligned kappa halves.
    "bf16_gqa5_qwen3_14b_heads": (Workload("t", 2, 40, 8, (1200, 333), 32, 128, seed=41), jacap_params()),
    "bf16_gqa7_nemotron_heads": (Workload("t", 2, 28, 4, (1500, 129), 32, 128, seed=42), jacap_params()),
    "bf16_gqa3_tau1": (Workload("t", 1, 6, 2, (800, 257), 16, 64, seed=43), jacap_params(tau=1.0)),
    "bf16_gqa6_unbiased": (Workload("t", 1, 12, 2, (700, 130), 16, 64, seed=44), jacap_params(cov_unbiased=1)),
    "bf16_gqa7_peaky_linear": (Workload("t", 1, 14, 2, (650, 3), 8, 40, seed=45), jacap_params(linear_weighting=1)),
    "f32_gqa5": (Workload("t", 1, 10, 2, (600, 77), 16, 64, dtype="f32", seed=46), jacap_params(tau=0.7)),
    "f32_gqa7": (Workload("t", 1, 14, 2, (500, 70), 8, 32, dtype="f32", seed=47), jacap_params()),
    # full covariance: tensor-core kernel with G w = 96, 80, 112 centred queries
    # (the last with a 32-row mu' image), CUDA-core kernel with G w = 192
    "bf16_gqa3_full_cov_w32": (Workload("t", 1, 6, 2, (900, 100), 32, 64, seed=48), jacap_params(full_covariance=1)),
    "bf16_gqa5_full_cov_w16": (Workload("t", 1, 10, 2, (700,), 16, 64, seed=49), jacap_params(full_covariance=1)),
    "bf16_gqa7_full_cov_w16": (Workload("t", 1, 14, 2, (640, 33), 16, 64, seed=50),
                               jacap_params(full_covariance=1, tau=2.0)),
    "bf16_gqa6_full_cov_w32_simt": (Workload("t", 1, 12, 2, (500,), 32, 64, seed=51),
                                    jacap_params(full_covariance=1)),
}


def with_schedule(p, schedule):
    return jacap_params(p.tau, p.weight_div_dk, p.ridge, p.cov_unbiased, p.linear_weighting, p.full_covariance,
                        schedule)


# every bf16 case under both schedules (separate kernels; the fused persistent
# launch); float32 caches always take the separate kernels
SMALL_RUNS = [(n, sch) for n in SMALL for sch in ((1, 2) if SMALL[n][0].dtype == "bf16" else (0,))]


@pytest.mark.parametrize("name,schedule", SMALL_RUNS, ids=[f"{n}-s{s}" for n, s in SMALL_RUNS])
def test_small_caches_every_unit(name, schedule):
    wl, params = SMALL[name]
    params = with_schedule(params, schedule)
    t = generate(wl, DEV)
    ev = evict(make_cache(t, wl), wl.budget, params)
    for s in range(len(wl.seqlens)):
        for layer in range(wl.num_layers):
            for g in range(wl.num_kv_heads):
                check_unit(ev, t, wl, params, s, layer, g)
    gpu_selection_properties(ev.scores, ev.idx, ev.kept, wl.seqlens, wl.budget)


@pytest.mark.parametrize("schedule", [1, 2])
def test_intermediates_match_the_oracle(schedule):
    wl = Workload("t", 2, 8, 2, (900, 333), 16, 64, seed=21)
    params = jacap_params(tau=1.5, schedule=schedule)
    t = generate(wl, DEV)
    ev = evict(make_cache(t, wl), wl.budget, params)
    inter = ev.intermediates()
    G = wl.num_q_heads // wl.num_kv_heads
    import oracle.jacap_oracle as O
    for s in range(2):
        for layer in range(2):
            for g in range(2):
                q, K, V = unit_arrays(t, wl.num_q_heads, s, layer, g)
                for j in range(G):
                    mu, lam = O.window_stats(q[j])
                    h = g * G + j
                    np.testing.assert_allclose(inter["mu_scaled"][s, layer, h].double().cpu().numpy(),
                                               mu / (params.tau * np.sqrt(128)), rtol=1e-5, atol=1e-7)
                    np.testing.assert_allclose(inter["lambda"][s, layer, h].double().cpu().numpy(), lam,
                                               rtol=1e-5, atol=1e-7)
                w = O.unit_weights(K, q, JacapParams(tau=params.tau))
                A = O.capacity_matrix(V, w)
                G_ora = A - np.eye(128)
                G_gpu = inter["gram"][layer, g, s].double().cpu().numpy()
                np.testing.assert_allclose(G_gpu, G_ora, rtol=1e-4, atol=1e-5 * np.abs(G_ora).max())
                Lc = np.linalg.cholesky(A)
                Minv = np.linalg.inv(Lc)
                np.testing.assert_allclose(inter["chol_inv"][layer, g, s].double().cpu().numpy(), Minv,
                                           rtol=1e-4, atol=1e-6)


def test_layer_groups_bound_the_workspace_and_match_the_oracle():
    # the pass over groups of 2 of 5 layers with a workspace sized for a group
    wl = Workload("t", 5, 12, 2, (900, 333), 16, 64, seed=31)
    t = generate(wl, DEV)
    whole = Evictor(make_cache(t, wl), wl.budget)
    ev = Evictor(make_cache(t, wl), wl.budget, layer_group=2)
    assert ev.ws.numel() < whole.ws.numel() and [n for _, n in ev.groups] == [2, 2, 1]
    ev.run()
    ev.check()
    for s in range(len(wl.seqlens)):
        for layer in range(wl.num_layers):
            for g in range(wl.num_kv_heads):
                check_unit(ev, t, wl, jacap_params(), s, layer, g, check_w=False)
    gpu_selection_properties(ev.scores, ev.idx, ev.kept, wl.seqlens, wl.budget)


@pytest.mark.parametrize("schedule", [1, 2])
def test_repeat_calls_are_bitwise_deterministic(schedule):
    wl = Workload("t", 2, 8, 2, (1500, 700), 16, 64, seed=22)
    t = generate(wl, DEV)
    ev = Evictor(make_cache(t, wl), wl.budget, jacap_params(schedule=schedule))
    ev.run()
    ev.check()
    s1, i1 = ev.scores.clone(), ev.idx.clone()
    ev.run()
    ev.check()
    assert torch.equal(ev.scores, s1) and torch.equal(ev.idx, i1)


def test_strided_cache_views():
    # K/V as views into a padded buffer (token stride 136) and a head-major
    # buffer; the TMA maps and the gather must follow the strides.
    wl = Workload("t", 2, 8, 2, (700, 260), 16, 64, seed=23)
    t = generate(wl, DEV)
    L, Hkv, N, d = t.k.shape
    kb = torch.zeros((Hkv, L, N, 136), dtype=t.k.dtype, device=DEV)
    vb = torch.zeros_like(kb)
    kb[..., :d] = t.k.transpose(0, 1)
    vb[..., :d] = t.v.transpose(0, 1)
    k2 = kb.transpose(0, 1)[..., :d]
    v2 = vb.transpose(0, 1)[..., :d]
    ev_ref = evict(make_cache(t, wl), wl.budget)
    t2 = replace(t, k=k2, v=v2)
    ev = evict(Cache(t.q_win, k2, v2, t.cu_seqlens, t.seqlens, wl.num_q_heads), wl.budget)
    assert torch.equal(ev.scores, ev_ref.scores)
    assert torch.equal(ev.idx, ev_ref.idx)
    assert torch.equal(ev.k_out, ev_ref.k_out) and torch.equal(ev.v_out, ev_ref.v_out)
    check_unit(ev, t2, wl, jacap_params(), 1, 1, 1)


@pytest.mark.parametrize("name", ["bf16_gqa4_ragged_tails", "bf16_gqa2_peaky_tiny_seq", "f32_gqa4_peaky",
                                  "bf16_budget_exceeds_all"])
def test_fused_select_compact_equals_the_two_calls(name):
    # jacap_select_compact (one launch) against jacap_select + jacap_compact on
    # the same scores: positions, kept counts and rows bit for bit
    wl, params = SMALL[name]
    t = generate(wl, DEV)
    ev = evict(make_cache(t, wl), wl.budget, params)  # the fused call
    sep = Evictor(make_cache(t, wl), wl.budget, params)
    sep.scores.copy_(ev.scores)
    sep.ws[:64].zero_()
    sep.k_out.fill_(7)  # the zero rows must be written, not left over
    sep.v_out.fill_(7)
    sep.select()
    sep.compact()
    sep.check()
    assert torch.equal(ev.idx, sep.idx) and torch.equal(ev.kept, sep.kept)
    assert_rows_bitwise(sep.k_out, ev.k_out)
    assert_rows_bitwise(sep.v_out, ev.v_out)


def test_fused_select_compact_zero_fills_a_malformed_request():
    # request 1 claims tokens 300 .. 599 of a 500-token cache: it is refused
    # (positions -1, zero rows, status invalid argument) and request 0 is served
    wl = Workload("t", 1, 4, 2, (300, 200), 8, 32, seed=25)
    t = generate(wl, DEV)
    bad = torch.tensor([0, 300, 600], dtype=torch.int32, device=DEV)
    ev = Evictor(Cache(t.q_win, t.k, t.v, bad, [300, 300], wl.num_q_heads), wl.budget)
    ev.scores.fill_(1.0)  # all equal: the first B positions are kept
    ev.k_out.fill_(7)
    ev.v_out.fill_(7)
    ev.ws[:64].zero_()
    ev.select_compact()
    assert ev.device_status() == 1  # JACAP_ERR_INVALID_ARG
    assert ev.kept.cpu().tolist() == [wl.budget, 0]
    assert bool((ev.idx[:, :, 1] == -1).all())
    assert bool((ev.k_out[:, :, 1] == 0).all()) and bool((ev.v_out[:, :, 1] == 0).all())
    assert ev.idx[0, 0, 0].cpu().tolist() == list(range(wl.budget))
    for g in range(wl.num_kv_heads):
        assert_rows_bitwise(t.k[0, g, :wl.budget], ev.k_out[0, g, 0])
        assert_rows_bitwise(t.v[0, g, :wl.budget], ev.v_out[0, g, 0])


def test_window_of_one_gives_zero_scores_and_first_positions():
    wl = Workload("t", 1, 4, 2, (600,), 1, 40, seed=24)
    t = generate(wl, DEV)
    ev = evict(make_cache(t, wl), wl.budget)
    assert bool((ev.scores == 0).all())
    assert ev.idx[0, 0, 0].cpu().tolist() == list(range(40))


def test_malformed_cu_seqlens_is_reported_on_the_device():
    wl = Workload("t", 1, 4, 2, (300, 200), 8, 32, seed=25)
    t = generate(wl, DEV)
    bad = torch.tensor([0, 300, 400], dtype=torch.int32, device=DEV)  # does not end at N_tot
    ev = Evictor(Cache(t.q_win, t.k, t.v, bad, [300, 100], wl.num_q_heads), wl.budget)
    ev.run()
    assert ev.device_status() == 1  # JACAP_ERR_INVALID_ARG


def test_nonfinite_input_is_reported_on_the_device():
    wl = Workload("t", 1, 4, 2, (300,), 8, 32, seed=26)
    t = generate(wl, DEV)
    t.k[0, 1, 17, 5] = float("nan")
    ev = Evictor(make_cache(t, wl), wl.budget)
    ev.run()
    assert ev.device_status() == 5  # JACAP_ERR_NONFINITE


def test_config1_every_unit():
    wl = config(1)
    t = generate(wl, DEV)
    ev = evict(make_cache(t, wl), wl.budget)
    for g in range(wl.num_kv_heads):
        check_unit(ev, t, wl, jacap_params(), 0, 0, g)
    gpu_selection_properties(ev.scores, ev.idx, ev.kept, wl.seqlens, wl.budget)


def _spread_units(wl, count):
    """`count` units (request, layer, KV head): the first and the last layer and
    KV head, the shortest and the longest request, the rest drawn with a fixed
    seed."""
    S, L, H = len(wl.seqlens), wl.num_layers, wl.num_kv_heads
    out = []

    def add(u):
        if u not in out:
            out.append(u)

    for s in dict.fromkeys([int(np.argmin(wl.seqlens)), int(np.argmax(wl.seqlens)), 0, S - 1]):
        add((s, 0, 0))
        add((s, L - 1, H - 1))
    add((0, 0, H - 1))
    add((0, L - 1, 0))
    r = np.random.default_rng(1000 + S * 100 + L)
    while len(out) < count:
        add((int(r.integers(S)), int(r.integers(L)), int(r.integers(H))))
    return out[:count]


def _check_sampled_units(t, wl, evs, units):
    """Scores, TOP-B sets (for every evictor's budget) and kept rows of `units`
    against the oracle, run on a pool of processes."""
    budgets = sorted({e.budget for e in evs})
    arrays = [tuple(x.astype(np.float32) for x in unit_arrays(t, wl.num_q_heads, s, layer, g))
              for (s, layer, g) in units]
    results = run_units(arrays, budgets)
    cu = t.cu_seqlens.cpu().tolist()
    for (s, layer, g), (ora_scores, ora_idx) in zip(units, results):
        a, b = cu[s], cu[s + 1]
        gs = evs[0].scores[layer, g, a:b].double().cpu().numpy()
        assert_scores_close(gs, ora_scores, f"scores of unit {(s, layer, g)}")
        for ev in evs:
            gidx = ev.idx[layer, g, s].cpu().numpy()
            assert_selection(gidx, b - a, ev.budget, ora_scores, ora_idx[ev.budget])
            kept = min(b - a, ev.budget)
            sel = torch.as_tensor(gidx[:kept], dtype=torch.long, device=t.k.device)
            assert_rows_bitwise(t.k[layer, g, a:b][sel], ev.k_out[layer, g, s, :kept])
            assert_rows_bitwise(t.v[layer, g, a:b][sel], ev.v_out[layer, g, s, :kept])


@pytest.mark.parametrize("index,samples", [(2, 8), (3, 8), (4, 16), (5, 16)])
def test_full_size_config(index, samples):
    wl = config(index)
    t = generate(wl, DEV)
    ev = evict(make_cache(t, wl), wl.budget)
    gpu_selection_properties(ev.scores, ev.idx, ev.kept, wl.seqlens, wl.budget)
    evs = [ev]
    if index == 2:
        # the other two budgets of the configuration: selection (and compaction)
        # on the same scores, as separate calls and as the fused call
        for b in (128, 2048):
            ev2 = Evictor(make_cache(t, wl), b)
            ev2.scores.copy_(ev.scores)
            ev2.ws[:64].zero_()  # status word: select honours the one jacap_score leaves
            ev2.select()
            ev2.compact()
            gpu_selection_properties(ev2.scores, ev2.idx, ev2.kept, wl.seqlens, b)
            k2, v2 = ev2.k_out.clone(), ev2.v_out.clone()
            ev2.select_compact()
            assert_rows_bitwise(k2, ev2.k_out)
            assert_rows_bitwise(v2, ev2.v_out)
            del k2, v2
            evs.append(ev2)
    _check_sampled_units(t, wl, evs, _spread_units(wl, samples))
    del ev, evs, t
    torch.cuda.empty_cache()


def _output_factors(wl, d_o, seed, device):
    """Synthetic output maps W (d_o x 128) per plane and their 128 x 128 factors
    F = R of W = Q R (float32 on the device); W stays on the host for the oracle."""
    r = np.random.default_rng(seed)
    L, Hkv = wl.num_layers, wl.num_kv_heads
    W = r.normal(size=(L, Hkv, d_o, 128)) / np.sqrt(128)
    F = np.stack([[np.linalg.qr(W[l, g])[1] for g in range(Hkv)] for l in range(L)])
    return W, torch.as_tensor(F, dtype=torch.float32, device=device).contiguous()


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_output_directions_every_unit(dtype):
    # u_i = W v_i (Sec. 3.1) through the reduced d x d form on the GPU vs the
    # oracle's explicit d_o-dimensional capacity matrix
    wl = Workload("t", 2, 8, 2, (1300, 400), 16, 96, dtype=dtype, seed=21)
    t = generate(wl, DEV)
    W, F = _output_factors(wl, 192, 5, DEV)
    params = jacap_params()
    ev = Evictor(make_cache(t, wl), wl.budget, params, out_factor=F)
    ev.run()
    ev.check()
    # the factors the GPU used, in float64, define the same W^T W as W up to rounding
    cu = t.cu_seqlens.cpu().tolist()
    for s in range(len(wl.seqlens)):
        for layer in range(wl.num_layers):
            for g in range(wl.num_kv_heads):
                q, K, V = unit_arrays(t, wl.num_q_heads, s, layer, g)
                Ff = F[layer, g].double().cpu().numpy()  # a d x d output map with the GPU's exact factor
                ora = oracle_unit(q, K, V, wl.budget, JacapParams(), out_proj=Ff)
                a, b = cu[s], cu[s + 1]
                assert_scores_close(ev.scores[layer, g, a:b].double().cpu().numpy(), ora["scores"])
                assert_selection(ev.idx[layer, g, s].cpu().numpy(), b - a, wl.budget, ora["scores"], ora["idx"])
                # and the explicit d_o-dimensional output map gives the same scores (push-through)
                ora_w = oracle_unit(q, K, V, wl.budget, JacapParams(), out_proj=W[layer, g])
                assert_scores_close(ev.scores[layer, g, a:b].double().cpu().numpy(), ora_w["scores"])


def test_pass_replays_from_a_cuda_graph():
    # the whole pass (scores, selection, compaction) captured once into a CUDA
    # graph and replayed gives the eager pass's results bit for bit
    wl, params = SMALL["bf16_gqa4_ragged_tails"]
    t = generate(wl, DEV)
    ev = evict(make_cache(t, wl), wl.budget, params)  # eager, also warms every kernel up
    ref = [x.clone() for x in (ev.scores, ev.idx, ev.kept, ev.k_out, ev.v_out)]
    for x in (ev.scores, ev.k_out, ev.v_out):
        x.zero_()
    ev.idx.fill_(-7)
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.stream(side):
        with torch.cuda.graph(g, stream=side, capture_error_mode="thread_local"):
            ev.run(side)
    torch.cuda.current_stream().wait_stream(side)
    for _ in range(2):
        g.replay()
        torch.cuda.synchronize()
        ev.check()
        got = (ev.scores, ev.idx, ev.kept, ev.k_out, ev.v_out)
        assert all(torch.equal(a, b) for a, b in zip(ref, got))


def test_a_wait_that_nothing_ends_expires_and_the_context_stays_usable():
    # failure detection without a fault: a bounded wait on an mbarrier that
    # nothing arrives on gives up after its limit, the status word says
    # timeout, and the next pass on the same workspace runs clean
    import time

    from paper_2609_08131_gb300 import JACAP_ERR_TIMEOUT, jacap_selftest_wait
    from paper_2609_08131_gb300.api import _ptr, _stream

    wl = Workload("t", 1, 4, 2, (700, 129), 8, 64, seed=29)
    t = generate(wl, DEV)
    ev = Evictor(make_cache(t, wl), wl.budget)
    t0 = time.time()
    assert jacap_selftest_wait(_ptr(ev.ws), ev.ws.numel(), 20_000_000, _stream()) == 0
    assert ev.device_status() == JACAP_ERR_TIMEOUT
    assert time.time() - t0 < 5.0
    ev.run()
    ev.check()
    for g in range(wl.num_kv_heads):
        check_unit(ev, t, wl, jacap_params(), 1, 0, g)


def test_host_cache_pass_with_output_directions_matches_the_device_pass():
    # HostEvictor hands each layer group its slice of the output factors: the
    # kept positions and rows equal those of the device-resident pass (both run
    # the same kernels on the same bytes; only the chunking of a group's
    # layout may differ, so positions may differ only at near ties)
    from paper_2609_08131_gb300.api import HostEvictor

    wl = Workload("t", 3, 8, 2, (900, 300), 16, 64, seed=44)
    t = generate(wl, DEV)
    _, F = _output_factors(wl, 160, 9, DEV)
    dev = Evictor(make_cache(t, wl), wl.budget, jacap_params(), out_factor=F)
    dev.run()
    dev.check()
    he = HostEvictor(t.q_win.cpu().pin_memory(), t.k.cpu().pin_memory(), t.v.cpu().pin_memory(), t.cu_seqlens,
                     list(wl.seqlens), wl.num_q_heads, wl.budget, jacap_params(), group_layers=2, device=DEV,
                     out_factor=F)
    he.run()
    a, b = he.idx_h.reshape(-1, wl.budget).numpy(), dev.idx.cpu().reshape(-1, wl.budget).numpy()
    differ = sum(len(np.setdiff1d(x, y)) for x, y in zip(a, b))
    assert differ <= 2, differ
    if differ == 0:
        assert_rows_bitwise(dev.k_out, he.k_out_h)
        assert_rows_bitwise(dev.v_out, he.v_out_h)


def test_many_short_units_take_the_small_selection_ctas():
    # more units than SMs and requests of at most 4096 tokens: the selection
    # runs 256-thread CTAs (four or more per SM); sampled units against the
    # oracle, every unit's selection properties, and the fused selection +
    # compaction against the two separate calls
    wl = Workload("t", 24, 16, 8, (1500, 700, 129), 16, 96, seed=46)  # 24 x 8 x 3 = 576 units
    assert wl.num_layers * wl.num_kv_heads * len(wl.seqlens) > torch.cuda.get_device_properties(0).multi_processor_count
    t = generate(wl, DEV)
    ev = evict(make_cache(t, wl), wl.budget)
    gpu_selection_properties(ev.scores, ev.idx, ev.kept, wl.seqlens, wl.budget)
    for (s, layer, g) in ((0, 0, 0), (1, 11, 5), (2, 23, 7), (0, 17, 3)):
        check_unit(ev, t, wl, jacap_params(), s, layer, g, check_w=False)
    sep = Evictor(make_cache(t, wl), wl.budget)
    sep.scores.copy_(ev.scores)
    sep.ws[:64].zero_()
    sep.select()
    sep.compact()
    sep.check()
    assert torch.equal(ev.idx, sep.idx) and torch.equal(ev.kept, sep.kept)
    assert_rows_bitwise(sep.k_out, ev.k_out)
    assert_rows_bitwise(sep.v_out, ev.v_out)


def test_full_size_full_covariance():
    # the K pass with the full-covariance kappa on the 32-layer 32K-token
    # cache (every CTA runs several units, one image per run): sampled units
    # against the oracle, every unit's selection properties
    wl = config(2)
    t = generate(wl, DEV)
    params = jacap_params(full_covariance=1)
    ev = evict(make_cache(t, wl), wl.budget, params)
    gpu_selection_properties(ev.scores, ev.idx, ev.kept, wl.seqlens, wl.budget)
    for (layer, g) in ((0, 0), (31, 7), (13, 4)):
        check_unit(ev, t, wl, params, 0, layer, g, check_w=False)
    del ev, t
    torch.cuda.empty_cache()
