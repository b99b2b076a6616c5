"""Torch-facing convenience layer over the C ABI.

PyTorch supplies device memory and streams only; every step runs in
libjacap's kernels. Errors from the library raise ``JacapError``.
"""

from __future__ import annotations

import ctypes
from dataclasses import dataclass

import torch

from . import (
    JACAP_BF16,
    JACAP_F32,
    JACAP_OK,
    jacap_compact,
    jacap_device_status,
    jacap_layout,
    jacap_params,
    jacap_score,
    jacap_score_timed,
    jacap_score_out,
    jacap_select,
    jacap_status_string,
    jacap_workspace_offsets,
    jacap_workspace_size,
)


class JacapError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {jacap_status_string(status)} (status {status})")


def _check(status: int, where: str):
    if status != JACAP_OK:
        raise JacapError(status, where)


def _ptr(t):
    return ctypes.c_void_p(t.data_ptr()) if t is not None else ctypes.c_void_p(0)


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


@dataclass
class Cache:
    """A KV cache in the library's layout plus the tensors that back it.

    k, v        [L, Hkv, N_tot, 128] (channel stride 1; K and V share strides)
    q_win       [S, L, Hq, w, 128]
    cu_seqlens  int32 [S + 1] on the device; seqlens: host list of n_s
    """

    q_win: torch.Tensor
    k: torch.Tensor
    v: torch.Tensor
    cu_seqlens: torch.Tensor
    seqlens: list
    num_q_heads: int

    def layout(self) -> jacap_layout:
        k, q = self.k, self.q_win
        if k.dtype not in (torch.float32, torch.bfloat16) or q.dtype != k.dtype or self.v.dtype != k.dtype:
            raise ValueError("q_win, k and v must share dtype float32 or bfloat16")
        if k.stride() != self.v.stride() or k.shape != self.v.shape:
            raise ValueError("k and v must have the same shape and strides")
        if k.stride(-1) != 1 or q.stride(-1) != 1:
            raise ValueError("the channel axis must be contiguous")
        L, Hkv, N, d = k.shape
        S = len(self.seqlens)
        lay = jacap_layout()
        lay.num_seqs = S
        lay.cu_seqlens = self.cu_seqlens.data_ptr()
        lay.max_seqlen = max(1, max(self.seqlens))
        lay.total_tokens = N
        lay.num_layers = L
        lay.num_q_heads = self.num_q_heads
        lay.num_kv_heads = Hkv
        lay.head_dim = d
        lay.window = q.shape[3]
        lay.dtype = JACAP_BF16 if k.dtype == torch.bfloat16 else JACAP_F32
        lay.kv_stride_layer, lay.kv_stride_head, lay.kv_stride_token = k.stride(0), k.stride(1), k.stride(2)
        lay.q_stride_seq, lay.q_stride_layer, lay.q_stride_head, lay.q_stride_pos = (
            q.stride(0), q.stride(1), q.stride(2), q.stride(3))
        return lay


class Evictor:
    """Owns the workspace and output buffers for repeated passes over caches
    of one shape; ``run()`` enqueues score, select and compact."""

    def __init__(self, cache: Cache, budget: int, params: jacap_params | None = None, out_factor=None):
        """``out_factor``: optional float32 [L][Hkv][128][128] device tensor of
        factors F with F^T F = W^T W for the output maps W (u_i = W v_i);
        None uses the proxy u_i = v_i."""
        self.cache = cache
        self.budget = int(budget)
        self.params = params if params is not None else jacap_params()
        if out_factor is not None:
            L, Hkv = cache.k.shape[0], cache.k.shape[1]
            if (out_factor.dtype != torch.float32 or tuple(out_factor.shape) != (L, Hkv, 128, 128)
                    or not out_factor.is_contiguous() or out_factor.device != cache.k.device):
                raise ValueError("out_factor must be a contiguous float32 [L][Hkv][128][128] tensor on the cache's device")
        self.out_factor = out_factor
        self.lay = cache.layout()
        dev = cache.k.device
        nbytes = jacap_workspace_size(self.lay, self.budget)
        if nbytes == 0:
            raise JacapError(1, "jacap_workspace_size")
        self.ws = torch.empty(nbytes, dtype=torch.uint8, device=dev)
        L, Hkv, N, d = cache.k.shape
        S = len(cache.seqlens)
        self.scores = torch.empty((L, Hkv, N), dtype=torch.float32, device=dev)
        self.idx = torch.empty((L, Hkv, S, self.budget), dtype=torch.int32, device=dev)
        self.kept = torch.empty((S,), dtype=torch.int32, device=dev)
        self.k_out = torch.empty((L, Hkv, S, self.budget, d), dtype=cache.k.dtype, device=dev)
        self.v_out = torch.empty_like(self.k_out)

    def score(self, stream=None, events=None):
        """jacap_score; with ``events`` (JACAP_SCORE_KERNELS + 1 torch.cuda.Event
        objects) the timed variant records them around the kernels of the pass."""
        c = self.cache
        if self.out_factor is not None:
            handles = [e.cuda_event for e in events] if events is not None else []
            _check(jacap_score_out(self.lay, self.params, _ptr(c.q_win), _ptr(c.k), _ptr(c.v), _ptr(self.out_factor),
                                   _ptr(self.scores), _ptr(self.ws), self.ws.numel(), _stream(stream), handles),
                   "jacap_score_out")
        elif events is None:
            _check(jacap_score(self.lay, self.params, _ptr(c.q_win), _ptr(c.k), _ptr(c.v), _ptr(self.scores),
                               _ptr(self.ws), self.ws.numel(), _stream(stream)), "jacap_score")
        else:
            handles = [e.cuda_event for e in events]
            _check(jacap_score_timed(self.lay, self.params, _ptr(c.q_win), _ptr(c.k), _ptr(c.v), _ptr(self.scores),
                                     _ptr(self.ws), self.ws.numel(), _stream(stream), handles), "jacap_score_timed")

    def select(self, stream=None):
        _check(jacap_select(self.lay, _ptr(self.scores), self.budget, _ptr(self.idx), _ptr(self.kept),
                            _ptr(self.ws), self.ws.numel(), _stream(stream)), "jacap_select")

    def compact(self, stream=None):
        c = self.cache
        _check(jacap_compact(self.lay, _ptr(c.k), _ptr(c.v), _ptr(self.idx), self.budget, _ptr(self.k_out),
                             _ptr(self.v_out), _stream(stream)), "jacap_compact")

    def run(self, stream=None):
        self.score(stream)
        self.select(stream)
        self.compact(stream)

    def device_status(self, stream=None) -> int:
        return jacap_device_status(_ptr(self.ws), _stream(stream))

    def check(self, stream=None):
        _check(self.device_status(stream), "device status")

    def intermediates(self):
        """Views of the workspace intermediates (see jacap_workspace_offsets)."""
        st, off = jacap_workspace_offsets(self.lay, self.budget)
        _check(st, "jacap_workspace_offsets")
        c = self.cache
        L, Hkv, N, d = c.k.shape
        S, Hq = len(c.seqlens), c.num_q_heads
        units = L * Hkv * S

        def view(o, shape):
            n = 1
            for s in shape:
                n *= s
            return self.ws[o:o + 4 * n].view(torch.float32).view(*shape)

        return {
            "mu_scaled": view(off.mu_scaled, (S, L, Hq, d)),
            "lambda": view(off.lambda_, (S, L, Hq, d)),
            "weights": view(off.weights, (L, Hkv, N)),
            "gram": view(off.gram, (L, Hkv, S, d, d)),
            "chol_inv": view(off.chol_inv, (L, Hkv, S, d, d)),
            "units": units,
        }


def evict(cache: Cache, budget: int, params: jacap_params | None = None, check: bool = True) -> Evictor:
    """One eviction pass over a device-resident cache; returns the Evictor
    whose scores / idx / kept / k_out / v_out hold the results."""
    ev = Evictor(cache, budget, params)
    ev.run()
    if check:
        ev.check()
    return ev
