"""The C-ABI library builds, loads, exports every declared symbol, and rejects
bad arguments on the host before touching a GPU. No compute call here."""

import ctypes
import os
import re

import pytest

import paper_2609_08131_gb300 as J
from paper_2609_08131_gb300 import _lib

HEADER = os.path.join(_lib.INCLUDE, "jacap.h")


def declared_symbols():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(jacap_[a-z_]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_symbols()
    for n in ["jacap_score", "jacap_select", "jacap_compact", "jacap_workspace_size", "jacap_device_status",
              "jacap_status_string", "jacap_workspace_offsets"]:
        assert n in names
    assert set(names) == set(_lib.EXPORTS)


def test_library_exports_every_declared_symbol(jacap_lib):
    for name in declared_symbols():
        assert hasattr(jacap_lib, name), name


def good_layout(**kw):
    lay = J.jacap_layout()
    lay.num_seqs = 2
    lay.cu_seqlens = 0x1000  # never dereferenced on the host
    lay.max_seqlen = 300
    lay.total_tokens = 500
    lay.num_layers = 2
    lay.num_q_heads = 8
    lay.num_kv_heads = 2
    lay.head_dim = 128
    lay.window = 16
    lay.dtype = J.JACAP_BF16
    lay.kv_stride_layer = 2 * 500 * 128
    lay.kv_stride_head = 500 * 128
    lay.kv_stride_token = 128
    lay.q_stride_seq = 2 * 8 * 16 * 128
    lay.q_stride_layer = 8 * 16 * 128
    lay.q_stride_head = 16 * 128
    lay.q_stride_pos = 128
    for k, v in kw.items():
        setattr(lay, k, v)
    return lay


def test_workspace_size_is_positive_and_monotone():
    a = J.jacap_workspace_size(good_layout(), 64)
    b = J.jacap_workspace_size(good_layout(total_tokens=5000, max_seqlen=4000,
                                           kv_stride_head=5000 * 128, kv_stride_layer=2 * 5000 * 128), 64)
    assert 0 < a < b
    assert a % 1024 == 0


@pytest.mark.parametrize("field,value,expect", [
    ("head_dim", 64, J.JACAP_ERR_UNSUPPORTED),
    ("num_q_heads", 7, J.JACAP_ERR_INVALID_ARG),       # not a multiple
    ("num_q_heads", 32, J.JACAP_ERR_UNSUPPORTED),      # G = 16
    ("window", 0, J.JACAP_ERR_INVALID_ARG),
    ("num_seqs", 0, J.JACAP_ERR_INVALID_ARG),
    ("total_tokens", 0, J.JACAP_ERR_INVALID_ARG),
    ("total_tokens", 1 << 31, J.JACAP_ERR_INVALID_ARG),
    ("max_seqlen", 0, J.JACAP_ERR_INVALID_ARG),
    ("kv_stride_token", 100, J.JACAP_ERR_INVALID_ARG),  # < head_dim
    ("kv_stride_token", 132, J.JACAP_ERR_INVALID_ARG),  # not 16-byte aligned rows (bf16)
    ("q_stride_pos", 130, J.JACAP_ERR_INVALID_ARG),
    ("dtype", 7, J.JACAP_ERR_INVALID_ARG),
    ("cu_seqlens", 0, J.JACAP_ERR_INVALID_ARG),
])
def test_invalid_layouts_are_rejected_on_the_host(field, value, expect):
    lay = good_layout(**{field: value})
    assert J.jacap_workspace_size(lay, 8) == 0
    p = ctypes.c_void_p(0x1000)
    st = J.jacap_score(lay, J.jacap_params(), p, p, p, p, p, 1 << 40, None)
    assert st == expect
    st = J.jacap_select(lay, p, 8, p, p, p, 1 << 40, None)
    assert st == expect
    st = J.jacap_compact(lay, p, p, p, 8, p, p, None)
    assert st == expect


@pytest.mark.parametrize("group", range(1, 9))
def test_every_gqa_ratio_up_to_eight_is_accepted(group):
    # Hq = G Hkv for G = 1 .. 8 (Qwen3-14B has G = 5, Nemotron-7B G = 7)
    lay = good_layout(num_q_heads=group * good_layout().num_kv_heads)
    assert J.jacap_workspace_size(lay, 8) > 0


def test_bad_params_and_buffers_are_rejected_on_the_host():
    lay = good_layout()
    p = ctypes.c_void_p(0x1000)
    big = J.jacap_workspace_size(lay, 8)
    assert J.jacap_score(lay, J.jacap_params(tau=0.0), p, p, p, p, p, big, None) == J.JACAP_ERR_INVALID_ARG
    assert J.jacap_score(lay, J.jacap_params(tau=float("nan")), p, p, p, p, p, big, None) == J.JACAP_ERR_INVALID_ARG
    assert J.jacap_score(lay, J.jacap_params(ridge=0), p, p, p, p, p, big, None) == J.JACAP_ERR_UNSUPPORTED
    assert J.jacap_score(lay, J.jacap_params(weight_div_dk=2), p, p, p, p, p, big, None) == J.JACAP_ERR_INVALID_ARG
    assert J.jacap_score(lay, J.jacap_params(linear_weighting=2), p, p, p, p, p, big, None) == J.JACAP_ERR_INVALID_ARG
    assert J.jacap_score(lay, J.jacap_params(full_covariance=3), p, p, p, p, p, big, None) == J.JACAP_ERR_INVALID_ARG
    assert J.jacap_score(lay, J.jacap_params(schedule=3), p, p, p, p, p, big, None) == J.JACAP_ERR_INVALID_ARG
    assert J.jacap_score(lay, J.jacap_params(schedule=-1), p, p, p, p, p, big, None) == J.JACAP_ERR_INVALID_ARG
    # the schedule query checks its arguments before it asks for a device
    assert J.jacap_schedule_info(lay, J.jacap_params(schedule=3))[0] == -J.JACAP_ERR_INVALID_ARG
    assert J.jacap_schedule_info(good_layout(head_dim=64), J.jacap_params())[0] == -J.JACAP_ERR_UNSUPPORTED
    lay1 = good_layout(window=1)
    assert J.jacap_score(lay1, J.jacap_params(cov_unbiased=1), p, p, p, p, p, big, None) == J.JACAP_ERR_INVALID_ARG
    mis = ctypes.c_void_p(0x1008)  # 8-byte aligned only
    assert J.jacap_score(lay, J.jacap_params(), mis, p, p, p, p, big, None) == J.JACAP_ERR_INVALID_ARG
    assert J.jacap_score(lay, J.jacap_params(), p, p, p, p, p, big - 1, None) == J.JACAP_ERR_WORKSPACE
    assert J.jacap_score(lay, J.jacap_params(), p, p, p, p, ctypes.c_void_p(0x1010), big, None) == J.JACAP_ERR_WORKSPACE
    assert J.jacap_select(lay, p, 0, p, p, p, big, None) == J.JACAP_ERR_INVALID_ARG
    assert J.jacap_compact(lay, p, p, p, 8, mis, p, None) == J.JACAP_ERR_INVALID_ARG
    # the fused calls check what the two calls they replace check
    assert J.jacap_select_compact(lay, p, 0, p, p, p, p, p, p, p, big, None) == J.JACAP_ERR_INVALID_ARG
    assert J.jacap_select_compact(lay, p, 8, p, p, p, p, mis, p, p, big, None) == J.JACAP_ERR_INVALID_ARG
    assert J.jacap_select_compact(lay, p, 8, p, p, p, p, p, p, p, big - 1, None) == J.JACAP_ERR_WORKSPACE
    assert J.jacap_select_compact_inplace(lay, p, 8, p, p, p, p, p, 2, p, big, None) == J.JACAP_ERR_INVALID_ARG
    assert J.jacap_select_compact_inplace(lay, p, 8, p, p, mis, p, p, 0, p, big, None) == J.JACAP_ERR_INVALID_ARG
    assert J.jacap_select_compact_inplace(lay, p, 8, p, p, p, p, None, 0, p, big - 1, None) == J.JACAP_ERR_WORKSPACE
    assert J.jacap_device_status(None, None) == J.JACAP_ERR_INVALID_ARG


def test_status_strings():
    for s in range(0, 8):
        assert isinstance(J.jacap_status_string(s), str) and J.jacap_status_string(s)
    assert J.jacap_status_string(0) == "ok"


def test_workspace_offsets_are_inside_the_workspace():
    lay = good_layout()
    st, off = J.jacap_workspace_offsets(lay, 8)
    assert st == J.JACAP_OK
    total = J.jacap_workspace_size(lay, 8)
    for name in ["mu_scaled", "lambda_", "weights", "gram", "chol_inv"]:
        assert 0 < getattr(off, name) < total
    assert J.jacap_workspace_offsets(good_layout(head_dim=64), 8)[0] == J.JACAP_ERR_UNSUPPORTED


def test_python_binding_names_match_the_c_abi():
    for name in _lib.EXPORTS:
        assert callable(getattr(J, name))


def test_host_cache_entry_checks_on_the_host():
    # jacap_evict_host: dense host layouts only; every refusal comes before any
    # CUDA call (the buffer size query needs no GPU either)
    lay = good_layout()
    p = ctypes.c_void_p(0x1000)
    null = ctypes.c_void_p(0)
    prm = J.jacap_params()
    with_rows = J.jacap_host_buffer_size(lay, 8, 1, 1)
    no_rows = J.jacap_host_buffer_size(lay, 8, 1, 0)
    one_layer = good_layout(num_layers=1, kv_stride_layer=2 * 500 * 128, q_stride_seq=8 * 16 * 128)
    assert with_rows > no_rows > J.jacap_workspace_size(one_layer, 8) > 0  # a group's workspace + buffers
    assert J.jacap_host_buffer_size(lay, 8, 2, 1) > with_rows  # two layers per group buffer
    assert J.jacap_host_buffer_size(lay, 8, 1, 2) == 0
    assert J.jacap_host_buffer_size(lay, 0, 1, 1) == 0
    padded = good_layout(kv_stride_token=136)  # a valid device layout, but not a dense host array
    assert J.jacap_workspace_size(padded, 8) > 0 and J.jacap_host_buffer_size(padded, 8, 1, 1) == 0
    args = lambda lay, b, gl, q, k_out, v_out, buf, nbytes: J.jacap_evict_host(  # noqa: E731
        lay, prm, b, gl, q, p, p, null, p, p, k_out, v_out, buf, nbytes, null, null)
    assert args(padded, 8, 1, p, p, p, p, 1 << 40) == J.JACAP_ERR_INVALID_ARG
    assert args(good_layout(num_q_heads=32), 8, 1, p, p, p, p, 1 << 40) == J.JACAP_ERR_UNSUPPORTED  # G = 16
    assert args(good_layout(head_dim=64), 8, 1, p, p, p, p, 1 << 40) == J.JACAP_ERR_UNSUPPORTED
    assert args(lay, 8, 1, null, p, p, p, 1 << 40) == J.JACAP_ERR_INVALID_ARG  # no window
    assert args(lay, 8, 1, p, p, null, p, 1 << 40) == J.JACAP_ERR_INVALID_ARG  # rows: both or neither
    assert args(lay, 8, 0, p, p, p, p, 1 << 40) == J.JACAP_ERR_INVALID_ARG
    assert args(lay, 8, 1, p, p, p, p, with_rows - 1) == J.JACAP_ERR_WORKSPACE
    assert args(lay, 8, 1, p, p, p, ctypes.c_void_p(0x1100), 1 << 40) == J.JACAP_ERR_WORKSPACE  # 256-B aligned


def test_tracing_and_checked_variants_compile(tmp_path):
    # JACAP_NVTX=1 / JACAP_CHECKED=1 / JACAP_TRACE=1 builds: the host side with
    # its NVTX ranges and trace section, and a persistent kernel with the checked
    # work-item stream and the trace resets, compile for sm_103a
    import subprocess

    for src in ("jacap_api.cu", "k_stream.cu"):
        cmd = [_lib.nvcc(), *_lib.ARCH, *_lib.CFLAGS, "-DJACAP_NVTX", "-DJACAP_CHECKED", "-DJACAP_TRACE", "-c",
               os.path.join(_lib.CSRC, src), "-o", str(tmp_path / (src + ".o"))]
        r = subprocess.run(cmd, capture_output=True, text=True)
        assert r.returncode == 0, r.stderr[-2000:]
