"""Jacap's prefill-time KV-cache eviction pass on one GB300 (sm_103a).

Thin Python binding of ``libjacap.so`` (C ABI in ``include/jacap.h``). The
functions ``jacap_*`` below carry the same names and arguments as the C entry
points and do argument marshalling only: every step of the pass runs in the
library's CUDA kernels. There is no CPU fallback; if the library is missing
the calls raise.

``api`` adds a torch-facing convenience layer (layouts from tensors,
workspace allocation, errors as exceptions, host-buffer end-to-end calls).
"""

from __future__ import annotations

import ctypes

from . import _lib

JACAP_OK = 0
JACAP_ERR_INVALID_ARG = 1
JACAP_ERR_UNSUPPORTED = 2
JACAP_ERR_WORKSPACE = 3
JACAP_ERR_CUDA = 4
JACAP_ERR_NONFINITE = 5
JACAP_ERR_TIMEOUT = 6

JACAP_F32 = 0
JACAP_BF16 = 1


class jacap_layout(ctypes.Structure):
    """Mirror of ``jacap_layout`` (include/jacap.h)."""

    _fields_ = [
        ("num_seqs", ctypes.c_int32),
        ("cu_seqlens", ctypes.c_void_p),
        ("max_seqlen", ctypes.c_int32),
        ("total_tokens", ctypes.c_int64),
        ("num_layers", ctypes.c_int32),
        ("num_q_heads", ctypes.c_int32),
        ("num_kv_heads", ctypes.c_int32),
        ("head_dim", ctypes.c_int32),
        ("window", ctypes.c_int32),
        ("dtype", ctypes.c_int32),
        ("kv_stride_layer", ctypes.c_int64),
        ("kv_stride_head", ctypes.c_int64),
        ("kv_stride_token", ctypes.c_int64),
        ("q_stride_seq", ctypes.c_int64),
        ("q_stride_layer", ctypes.c_int64),
        ("q_stride_head", ctypes.c_int64),
        ("q_stride_pos", ctypes.c_int64),
    ]


class jacap_params(ctypes.Structure):
    """Mirror of ``jacap_params``; defaults are the method's (tau = 10, Eq. 8 weights)."""

    _fields_ = [
        ("tau", ctypes.c_float),
        ("weight_div_dk", ctypes.c_int32),
        ("ridge", ctypes.c_int32),
        ("cov_unbiased", ctypes.c_int32),
        ("linear_weighting", ctypes.c_int32),
        ("full_covariance", ctypes.c_int32),
        ("schedule", ctypes.c_int32),
    ]

    # values of ``schedule``
    AUTO, SEPARATE, FUSED = 0, 1, 2

    def __init__(self, tau=10.0, weight_div_dk=1, ridge=1, cov_unbiased=0, linear_weighting=0, full_covariance=0,
                 schedule=0):
        super().__init__(tau, weight_div_dk, ridge, cov_unbiased, linear_weighting, full_covariance, schedule)


class jacap_ws_offsets(ctypes.Structure):
    _fields_ = [
        ("mu_scaled", ctypes.c_size_t),
        ("lambda_", ctypes.c_size_t),
        ("weights", ctypes.c_size_t),
        ("gram", ctypes.c_size_t),
        ("chol_inv", ctypes.c_size_t),
        ("trace_timeline", ctypes.c_size_t),
        ("trace_cta", ctypes.c_size_t),
    ]


_P = ctypes.c_void_p
_SIGS = {
    "jacap_workspace_size": (ctypes.c_size_t, [ctypes.POINTER(jacap_layout), ctypes.c_int32]),
    "jacap_score": (ctypes.c_int, [ctypes.POINTER(jacap_layout), ctypes.POINTER(jacap_params), _P, _P, _P, _P, _P,
                                   ctypes.c_size_t, _P]),
    "jacap_score_timed": (ctypes.c_int, [ctypes.POINTER(jacap_layout), ctypes.POINTER(jacap_params), _P, _P, _P, _P,
                                         _P, ctypes.c_size_t, _P, ctypes.POINTER(ctypes.c_void_p), ctypes.c_int32]),
    "jacap_score_out": (ctypes.c_int, [ctypes.POINTER(jacap_layout), ctypes.POINTER(jacap_params), _P, _P, _P, _P,
                                       _P, _P, ctypes.c_size_t, _P, ctypes.POINTER(ctypes.c_void_p), ctypes.c_int32]),
    "jacap_score_static": (ctypes.c_int, [ctypes.POINTER(jacap_layout), ctypes.POINTER(jacap_params), _P, _P, _P,
                                          _P, _P, ctypes.POINTER(ctypes.c_void_p)]),
    "jacap_select": (ctypes.c_int, [ctypes.POINTER(jacap_layout), _P, ctypes.c_int32, _P, _P, _P, ctypes.c_size_t,
                                    _P]),
    "jacap_compact": (ctypes.c_int, [ctypes.POINTER(jacap_layout), _P, _P, _P, ctypes.c_int32, _P, _P, _P]),
    "jacap_select_compact": (ctypes.c_int, [ctypes.POINTER(jacap_layout), _P, ctypes.c_int32, _P, _P, _P, _P, _P,
                                            _P, _P, ctypes.c_size_t, _P]),
    "jacap_score_stats": (ctypes.c_int, [ctypes.POINTER(jacap_layout), ctypes.POINTER(jacap_params), _P, _P, _P,
                                         _P, _P, _P, ctypes.c_size_t, _P, ctypes.POINTER(ctypes.c_void_p),
                                         ctypes.c_int32]),
    "jacap_stats_update": (ctypes.c_int, [ctypes.POINTER(jacap_layout), _P, ctypes.c_int32, _P, _P, _P]),
    "jacap_compact_inplace": (ctypes.c_int, [ctypes.POINTER(jacap_layout), _P, _P, _P, _P, ctypes.c_int32,
                                             ctypes.c_int32, _P, ctypes.c_size_t, _P]),
    "jacap_selftest_wait": (ctypes.c_int, [_P, ctypes.c_size_t, ctypes.c_int64, _P]),
    "jacap_select_compact_inplace": (ctypes.c_int, [ctypes.POINTER(jacap_layout), _P, ctypes.c_int32, _P, _P, _P, _P,
                                                    _P, ctypes.c_int32, _P, ctypes.c_size_t, _P]),
    "jacap_device_status": (ctypes.c_int, [_P, _P]),
    "jacap_host_buffer_size": (ctypes.c_size_t, [ctypes.POINTER(jacap_layout), ctypes.c_int32, ctypes.c_int32,
                                                 ctypes.c_int32]),
    "jacap_evict_host": (ctypes.c_int, [ctypes.POINTER(jacap_layout), ctypes.POINTER(jacap_params), ctypes.c_int32,
                                        ctypes.c_int32, _P, _P, _P, _P, _P, _P, _P, _P, _P, ctypes.c_size_t, _P, _P]),
    "jacap_status_string": (ctypes.c_char_p, [ctypes.c_int]),
    "jacap_schedule_info": (ctypes.c_int32, [ctypes.POINTER(jacap_layout), ctypes.POINTER(jacap_params),
                                             ctypes.POINTER(ctypes.c_int32)]),
    "jacap_workspace_offsets": (ctypes.c_int, [ctypes.POINTER(jacap_layout), ctypes.c_int32,
                                               ctypes.POINTER(jacap_ws_offsets)]),
}


def lib() -> ctypes.CDLL:
    """The loaded C library with argument types declared."""
    h = _lib.load(build_if_missing=True)
    if not getattr(h, "_jacap_typed", False):
        for name, (res, args) in _SIGS.items():
            fn = getattr(h, name)
            fn.restype = res
            fn.argtypes = args
        h._jacap_typed = True
    return h


def jacap_schedule_info(layout: jacap_layout, params: jacap_params):
    """(schedule, (factor CTAs, Gram CTAs, score CTAs, kept V tiles per item)) that the scoring
    entry points would run on the current device; schedule < 0 is -(jacap_status)."""
    roles = (ctypes.c_int32 * 4)()
    sched = lib().jacap_schedule_info(ctypes.byref(layout), ctypes.byref(params), roles)
    return sched, tuple(roles)


def jacap_workspace_size(layout: jacap_layout, budget: int) -> int:
    return lib().jacap_workspace_size(ctypes.byref(layout), budget)


def jacap_score(layout, params, q_win, k, v, scores, ws, ws_bytes, stream) -> int:
    return lib().jacap_score(ctypes.byref(layout), ctypes.byref(params), q_win, k, v, scores, ws, ws_bytes, stream)


JACAP_SCORE_KERNELS = 7
SCORE_KERNEL_NAMES = ("plan", "query_stats", "k_pass", "weights", "gram", "factor", "scores")


def jacap_score_timed(layout, params, q_win, k, v, scores, ws, ws_bytes, stream, events) -> int:
    """``events``: sequence of cudaEvent_t handles (ints), length 0 or JACAP_SCORE_KERNELS + 1."""
    arr = (ctypes.c_void_p * max(1, len(events)))(*[ctypes.c_void_p(e) for e in events])
    return lib().jacap_score_timed(ctypes.byref(layout), ctypes.byref(params), q_win, k, v, scores, ws, ws_bytes,
                                   stream, arr, len(events))


def jacap_score_out(layout, params, q_win, k, v, out_factor, scores, ws, ws_bytes, stream, events=()) -> int:
    """``out_factor``: device pointer to the per-plane 128 x 128 factors F, or None."""
    arr = (ctypes.c_void_p * max(1, len(events)))(*[ctypes.c_void_p(e) for e in events])
    return lib().jacap_score_out(ctypes.byref(layout), ctypes.byref(params), q_win, k, v, out_factor, scores, ws,
                                 ws_bytes, stream, arr, len(events))


def jacap_score_stats(layout, params, stats, counts, k, v, scores, ws, ws_bytes, stream, events=()) -> int:
    """Scoring pass with running query statistics (``stats``, ``counts``: device pointers)."""
    arr = (ctypes.c_void_p * max(1, len(events)))(*[ctypes.c_void_p(e) for e in events])
    return lib().jacap_score_stats(ctypes.byref(layout), ctypes.byref(params), stats, counts, k, v, scores, ws,
                                   ws_bytes, stream, arr, len(events))


def jacap_stats_update(layout, q_new, reset, stats, counts, stream) -> int:
    return lib().jacap_stats_update(ctypes.byref(layout), q_new, int(reset), stats, counts, stream)


def jacap_selftest_wait(ws, ws_bytes, limit_ns, stream) -> int:
    return lib().jacap_selftest_wait(ws, ws_bytes, limit_ns, stream)


def jacap_select_compact_inplace(layout, scores, budget, idx, kept, k, v, pos, preserve_order, ws, ws_bytes,
                                 stream) -> int:
    return lib().jacap_select_compact_inplace(ctypes.byref(layout), scores, budget, idx, kept, k, v, pos,
                                              preserve_order, ws, ws_bytes, stream)


def jacap_compact_inplace(layout, k, v, pos, idx, budget, preserve_order, ws, ws_bytes, stream) -> int:
    return lib().jacap_compact_inplace(ctypes.byref(layout), k, v, pos, idx, budget, int(preserve_order), ws,
                                       ws_bytes, stream)


JACAP_STATIC_SCRATCH_BYTES = 64 << 20


def jacap_score_static(layout, params, q_win, k, v, scores, stream):
    """Returns ``(status, scratch)``: ``scratch`` is the device address of the
    library-owned workspace the call used (0 when it was refused)."""
    out = ctypes.c_void_p(0)
    st = lib().jacap_score_static(ctypes.byref(layout), ctypes.byref(params), q_win, k, v, scores, stream,
                                  ctypes.byref(out))
    return st, out.value or 0


def jacap_select(layout, scores, budget, idx, kept, ws, ws_bytes, stream) -> int:
    return lib().jacap_select(ctypes.byref(layout), scores, budget, idx, kept, ws, ws_bytes, stream)


def jacap_select_compact(layout, scores, budget, idx, kept, k, v, k_out, v_out, ws, ws_bytes, stream) -> int:
    return lib().jacap_select_compact(ctypes.byref(layout), scores, budget, idx, kept, k, v, k_out, v_out, ws,
                                      ws_bytes, stream)


def jacap_compact(layout, k, v, idx, budget, k_out, v_out, stream) -> int:
    return lib().jacap_compact(ctypes.byref(layout), k, v, idx, budget, k_out, v_out, stream)


def jacap_host_buffer_size(layout: jacap_layout, budget: int, group_layers: int, copy_rows: int) -> int:
    return lib().jacap_host_buffer_size(ctypes.byref(layout), budget, group_layers, copy_rows)


def jacap_evict_host(layout, params, budget, group_layers, q_win_host, k_host, v_host, out_factor, idx_host,
                     kept_host, k_out_host, v_out_host, dev_buf, dev_bytes, stream, copy_stream) -> int:
    """Host-cache eviction (``layout.cu_seqlens`` is a host pointer here); blocks until done."""
    return lib().jacap_evict_host(ctypes.byref(layout), ctypes.byref(params), budget, group_layers, q_win_host,
                                  k_host, v_host, out_factor, idx_host, kept_host, k_out_host, v_out_host, dev_buf,
                                  dev_bytes, stream, copy_stream)


def jacap_device_status(ws, stream) -> int:
    return lib().jacap_device_status(ws, stream)


def jacap_status_string(status: int) -> str:
    return lib().jacap_status_string(status).decode()


def jacap_workspace_offsets(layout: jacap_layout, budget: int):
    out = jacap_ws_offsets()
    st = lib().jacap_workspace_offsets(ctypes.byref(layout), budget, ctypes.byref(out))
    return st, out
