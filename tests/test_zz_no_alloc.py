"""jacap_score_static: the scoring pass on the library's static scratch.

The GPU tests call it twice in a row through the C ABI and compare both
results with jacap_score on a caller-allocated workspace, bit for bit. The file is named to
be collected last, so the static scratch is first touched after every other
test has run; it passes alone as well. The host-side refusals need no GPU.
"""

import ctypes

import pytest
import torch

from paper_2609_08131_gb300 import (
    JACAP_ERR_INVALID_ARG,
    JACAP_ERR_WORKSPACE,
    JACAP_OK,
    JACAP_STATIC_SCRATCH_BYTES,
    jacap_device_status,
    jacap_params,
    jacap_score_static,
    jacap_select,
    jacap_workspace_size,
)
from paper_2609_08131_gb300.api import Cache, Evictor
from paper_2609_08131_gb300.workloads import Workload, generate

from parity import assert_scores_close

CASES = {
    # 41 MiB of scratch: ragged requests, GQA 4, two layers.
    "bf16_gqa4_two_requests": (Workload("t", 2, 32, 8, (3000, 1000), 32, 256, seed=21), jacap_params()),
    # The SIMT float32 path with a ragged tail.
    "f32_mha_tau2": (Workload("t", 1, 4, 4, (1500, 2049), 16, 128, dtype="f32", seed=22), jacap_params(tau=2.0)),
}


def _ptr(t):
    return ctypes.c_void_p(t.data_ptr())


def _cache(t, wl):
    return Cache(t.q_win, t.k, t.v, t.cu_seqlens, t.seqlens, wl.num_q_heads)


@pytest.mark.gpu
@pytest.mark.parametrize("name", list(CASES))
def test_static_scratch_matches_caller_workspace_twice(name):
    wl, params = CASES[name]
    t = generate(wl, "cuda:0")
    cache = _cache(t, wl)
    ev = Evictor(cache, wl.budget, params)
    assert jacap_workspace_size(ev.lay, wl.budget) <= JACAP_STATIC_SCRATCH_BYTES
    ev.score()
    ev.check()
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    ref = ev.scores.double().cpu().numpy()
    for call in range(2):
        out = torch.full_like(ev.scores, float("nan"))
        st, scratch = jacap_score_static(ev.lay, params, _ptr(t.q_win), _ptr(t.k), _ptr(t.v), _ptr(out), stream)
        assert st == JACAP_OK, (call, st)
        assert scratch != 0 and scratch % 256 == 0
        assert jacap_device_status(ctypes.c_void_p(scratch), stream) == JACAP_OK
        # same kernels on the same bytes with fixed-order reductions: the
        # scores are bit for bit those of the caller-workspace pass
        assert_scores_close(out.double().cpu().numpy(), ref, f"static scores, call {call}")
        assert torch.equal(out.view(torch.int32), ev.scores.view(torch.int32)), f"static scores, call {call}"
    # The returned scratch serves as the workspace of jacap_select.
    idx = torch.empty_like(ev.idx)
    kept = torch.empty_like(ev.kept)
    st = jacap_select(ev.lay, _ptr(out), wl.budget, _ptr(idx), _ptr(kept), ctypes.c_void_p(scratch),
                      JACAP_STATIC_SCRATCH_BYTES, stream)
    assert st == JACAP_OK
    assert jacap_device_status(ctypes.c_void_p(scratch), stream) == JACAP_OK
    assert torch.equal(kept.cpu(), torch.tensor([min(n, wl.budget) for n in wl.seqlens], dtype=torch.int32))


def test_oversized_and_invalid_layouts_are_refused_on_the_host():
    # 89 MiB of scratch needed: refused before any CUDA call, so no GPU needed.
    wl = Workload("t", 4, 32, 8, (4096, 4096), 32, 512, seed=3)
    t = generate(wl, "cpu")
    lay = _cache(t, wl).layout()
    assert jacap_workspace_size(lay, wl.budget) > JACAP_STATIC_SCRATCH_BYTES
    null = ctypes.c_void_p(0)
    st, scratch = jacap_score_static(lay, jacap_params(), null, null, null, null, null)
    assert (st, scratch) == (JACAP_ERR_WORKSPACE, 0)
    lay.window = 0
    st, scratch = jacap_score_static(lay, jacap_params(), null, null, null, null, null)
    assert (st, scratch) == (JACAP_ERR_INVALID_ARG, 0)
