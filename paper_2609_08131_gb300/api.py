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
    jacap_evict_host,
    jacap_host_buffer_size,
    jacap_layout,
    jacap_params,
    jacap_schedule_info,
    jacap_score,
    jacap_score_timed,
    jacap_score_out,
    jacap_score_stats,
    jacap_select,
    jacap_select_compact,
    jacap_select_compact_inplace,
    jacap_stats_update,
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

    def __init__(self, cache: Cache, budget: int, params: jacap_params | None = None, out_factor=None,
                 layer_group: int | None = None):
        """``out_factor``: optional float32 [L][Hkv][128][128] device tensor of
        factors F with F^T F = W^T W for the output maps W (u_i = W v_i);
        None uses the proxy u_i = v_i.

        ``layer_group``: run the pass over groups of this many layers, one
        after the other on the same stream, with a workspace sized for one
        group instead of the whole cache (units are independent, so the kept
        sets are those of one pass up to near ties; the workspace takes ~36
        bytes per token and KV head of every layer it covers)."""
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
        L = cache.k.shape[0]
        gl = L if layer_group is None else max(1, min(int(layer_group), L))
        self.groups = [(l0, min(gl, L - l0)) for l0 in range(0, L, gl)]
        self._glay = {}
        for _, n in self.groups:
            if n not in self._glay:
                lay = cache.layout()
                lay.num_layers = n
                self._glay[n] = lay
        nbytes = max(jacap_workspace_size(lay, self.budget) for lay in self._glay.values())
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

    def schedule_info(self):
        """(schedule, roles) of the scoring pass on the current device: 1 = separate kernels,
        2 = fused (roles = factor, Gram and score CTAs, V tiles per item kept in L2); see
        jacap_schedule_info. With output directions the pass always uses separate kernels."""
        if self.out_factor is not None:
            return 1, (0, 0, 0, 0)
        lay = self._glay[self.groups[0][1]]
        sched, roles = jacap_schedule_info(lay, self.params)
        if sched < 0:
            raise JacapError(-sched, "jacap_schedule_info")
        return sched, roles

    def bind_outputs(self, idx, kept, k_out, v_out):
        """Write the results into caller-owned device tensors (views into a
        larger buffer, for instance) of the shapes and dtypes of ``idx``,
        ``kept``, ``k_out`` and ``v_out``; each must be contiguous."""
        for name, t in (("idx", idx), ("kept", kept), ("k_out", k_out), ("v_out", v_out)):
            ref = getattr(self, name)
            if t.shape != ref.shape or t.dtype != ref.dtype or t.device != ref.device or not t.is_contiguous():
                raise ValueError(f"{name} must be a contiguous {ref.dtype} tensor of shape {tuple(ref.shape)} "
                                 f"on {ref.device}")
        self.idx, self.kept, self.k_out, self.v_out = idx, kept, k_out, v_out

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

    def select_compact(self, stream=None):
        """jacap_select and jacap_compact in one launch."""
        c = self.cache
        _check(jacap_select_compact(self.lay, _ptr(self.scores), self.budget, _ptr(self.idx), _ptr(self.kept),
                                    _ptr(c.k), _ptr(c.v), _ptr(self.k_out), _ptr(self.v_out), _ptr(self.ws),
                                    self.ws.numel(), _stream(stream)), "jacap_select_compact")

    def run(self, stream=None):
        if len(self.groups) == 1:
            self.score(stream)
            self.select_compact(stream)
            return
        # layer groups: the same calls on sub-layouts whose data pointers start
        # at the group's first layer, writing the group's slices of the outputs
        c, st = self.cache, _stream(stream)
        ek, eq = c.k.element_size(), c.q_win.element_size()
        ws, wn = _ptr(self.ws), self.ws.numel()
        for l0, n in self.groups:
            lay = self._glay[n]
            koff, qoff = l0 * self.lay.kv_stride_layer * ek, l0 * self.lay.q_stride_layer * eq
            k = ctypes.c_void_p(c.k.data_ptr() + koff)
            v = ctypes.c_void_p(c.v.data_ptr() + koff)
            q = ctypes.c_void_p(c.q_win.data_ptr() + qoff)
            scores = _ptr(self.scores[l0:l0 + n])
            if self.out_factor is not None:
                _check(jacap_score_out(lay, self.params, q, k, v, _ptr(self.out_factor[l0:l0 + n]), scores, ws, wn,
                                       st, []), "jacap_score_out")
            else:
                _check(jacap_score(lay, self.params, q, k, v, scores, ws, wn, st), "jacap_score")
            _check(jacap_select_compact(lay, scores, self.budget, _ptr(self.idx[l0:l0 + n]), _ptr(self.kept), k, v,
                                        _ptr(self.k_out[l0:l0 + n]), _ptr(self.v_out[l0:l0 + n]), ws, wn, st),
                   "jacap_select_compact")
            # a later group's first kernel clears the status word: surface a
            # problem of this group first
            if self.device_status(stream) != JACAP_OK:
                _check(self.device_status(stream), f"device status (layers {l0} .. {l0 + n - 1})")

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


# Slots of the per-CTA time accounting of a JACAP_TRACE build (jacap_ws_offsets.trace_cta):
# kernel index -> (name, {slot: meaning}); "tiles" counts tiles, every other slot sums ns.
TRACE_CTA_SLOTS = {
    2: ("k_pass", {0: "producer: wait for a free stage", 1: "producer: loop", 2: "logits MMA: wait for an image",
                   3: "logits MMA: wait for a K tile and a free buffer", 5: "logits MMA: loop", 6: "tiles",
                   7: "kappa warp: wait for a K tile", 8: "kappa warp: its quarter of kappa",
                   9: "kappa warp: wait for the group's slot", 10: "kappa warp: partials into the slot",
                   11: "kappa warp: loop", 12: "readout warp: wait for logits",
                   13: "readout warp: readout of a tile", 14: "readout warp: loop",
                   15: "readout warp: wait for the kappa partials"}),
    0: ("gram", {0: "producer: wait for a free stage", 1: "producer: loop", 2: "MMA: wait for a scaled operand",
                 3: "MMA: wait for a free accumulator", 4: "MMA: loop", 5: "tiles", 6: "scaling warp: wait for V",
                 7: "scaling warp: wait for the weights", 8: "scaling warp: wait for a free operand buffer",
                 9: "scaling warp: scaling", 10: "scaling warp: loop", 11: "weight warp: wait for V",
                 12: "weight warp: weights of a tile", 13: "weight warp: loop"}),
    1: ("scores", {0: "producer: wait for a free stage", 1: "producer: loop", 2: "MMA: wait for an image",
                   3: "MMA: wait for a free accumulator", 4: "MMA: wait for a V tile", 5: "MMA: loop", 6: "tiles",
                   7: "epilogue warp: wait for an accumulator", 8: "epilogue warp: read, reduce and meet its partner",
                   9: "epilogue warp: weight and store", 10: "epilogue warp: loop"}),
    3: ("factor", {0: "partial Grams summed into A", 1: "elimination of diagonal block 0",
                   2: "elimination of diagonal block 1", 3: "elimination of diagonal block 2",
                   4: "elimination of diagonal block 3", 5: "elimination warp: wait for the other warps",
                   6: "panels and look-ahead updates", 7: "last inverse phase", 8: "outputs", 9: "units",
                   10: "whole unit"}),
    4: ("selection", {0: "scores loaded", 1: "radix passes", 2: "emission", 3: "rows gathered", 4: "units",
                      5: "whole unit"}),
}


def cta_time_accounting(ev: Evictor) -> dict:
    """Per-CTA time accounting of the last pass of ``ev`` (a JACAP_TRACE build): for each
    streaming kernel and the factor, the mean over its CTAs (the first 1024) of every slot,
    in us per CTA and ns per 128-token tile (streaming kernels) or per unit (factor)."""
    st, off = jacap_workspace_offsets(ev.lay, ev.budget)
    _check(st, "jacap_workspace_offsets")
    if off.trace_cta == 0:
        raise RuntimeError("the library was not built with JACAP_TRACE=1")
    torch.cuda.synchronize(ev.ws.device)
    nk = len(TRACE_CTA_SLOTS)
    tc = ev.ws[off.trace_cta:off.trace_cta + nk * 1024 * 16 * 8].view(torch.int64).view(nk, 1024, 16).cpu().double()
    out = {}
    for k, (name, slots) in TRACE_CTA_SLOTS.items():
        # the streaming kernels count 128-token tiles, the factor units
        per = "tile" if "tiles" in slots.values() else "unit"
        count_slot = next(j for j, m in slots.items() if m == per + "s")
        a = tc[k]
        a = a[a[:, count_slot] > 0]
        if a.shape[0] == 0:
            continue
        cnt = a[:, count_slot].clamp(min=1)
        rep = {"ctas": int(a.shape[0]), per + "s_per_cta": float(cnt.mean())}
        for j, m in slots.items():
            if j != count_slot:
                rep[m] = {"us_per_cta": float(a[:, j].mean() / 1e3), "ns_per_" + per: float((a[:, j] / cnt).mean())}
        out[name] = rep
    return out


def evict(cache: Cache, budget: int, params: jacap_params | None = None, check: bool = True) -> Evictor:
    """One eviction pass over a device-resident cache; returns the Evictor
    whose scores / idx / kept / k_out / v_out hold the results."""
    ev = Evictor(cache, budget, params)
    ev.run()
    if check:
        ev.check()
    return ev


class DecodeEvictor:
    """Decoding-stage eviction (Sec. 3.4: statistics from the queries seen so
    far; the decoding experiments of Sec. 4): one cache slot of
    ``budget + interval`` tokens per request and running query statistics.
    Whenever a request's cache reaches budget + interval tokens it is scored
    with those statistics and compacted in place back to ``budget`` tokens
    (by default by moving the kept rows from past the budget into the evicted
    rows, so the slot order is not the token order; ``pos`` records it).
    Requests that fill on the same decode step and sit next to each other are
    evicted together in one pass (one launch of each kernel for all of them).

    Buffers (device), stored [L, Hkv, S, cap(, 128)] so that neighbouring
    requests form one cache layout, exposed request-major:
      k, v    [S, L, Hkv, cap, 128] views, cap = budget + interval; request s
              holds its ``lengths[s]`` tokens in rows 0 .. lengths[s] - 1
      pos     int32 [S, L, Hkv, cap] view: the id of every cached token (the
              prefill tokens are 0 .. n0 - 1, decode step t of a request adds
              n0 + t); it moves with the rows
      stats   float32 [S, L, Hq, 2, 128] (mean, M2), counts int32 [S, L, Hq]
    After an eviction of requests a .. b - 1, ``scores`` [L, Hkv, (b - a) cap]
    and ``idx`` [L, Hkv, b - a, budget] hold that pass's scores and positions.
    Writing a decode step's k, v into the slot is the model's cache write (a
    plain indexed copy here); the statistics, the scoring pass, the selection
    and the compaction run in libjacap's kernels.
    """

    def __init__(self, num_seqs: int, num_layers: int, num_q_heads: int, num_kv_heads: int, budget: int,
                 interval: int, dtype=torch.bfloat16, params: jacap_params | None = None, device="cuda",
                 preserve_order: bool = False):
        """``preserve_order``: keep the retained rows in ascending slot order
        (moves up to ``budget`` rows per eviction) instead of filling the
        evicted rows with the kept rows from past the budget (moves at most
        ``interval`` rows)."""
        if budget < 1 or interval < 1:
            raise ValueError("budget and interval must be >= 1")
        if dtype not in (torch.bfloat16, torch.float32):
            raise ValueError("dtype must be bfloat16 or float32")
        self.S, self.L, self.Hq, self.Hkv = num_seqs, num_layers, num_q_heads, num_kv_heads
        self.budget, self.interval = int(budget), int(interval)
        self.cap = self.budget + self.interval
        self.dtype = dtype
        self.params = params if params is not None else jacap_params()
        self.preserve_order = bool(preserve_order)
        dev = torch.device(device)
        S, L, Hq, Hkv, cap, d = self.S, self.L, self.Hq, self.Hkv, self.cap, 128
        self._k = torch.zeros((L, Hkv, S, cap, d), dtype=dtype, device=dev)
        self._v = torch.zeros_like(self._k)
        self._pos = torch.full((L, Hkv, S, cap), -1, dtype=torch.int32, device=dev)
        self.k = self._k.permute(2, 0, 1, 3, 4)
        self.v = self._v.permute(2, 0, 1, 3, 4)
        self.pos = self._pos.permute(2, 0, 1, 3)
        self.stats = torch.zeros((S, L, Hq, 2, d), dtype=torch.float32, device=dev)
        self.counts = torch.zeros((S, L, Hq), dtype=torch.int32, device=dev)
        self.lengths = [0] * S
        self.next_id = [0] * S
        self.events = 0   # request evictions
        self.passes = 0   # scoring passes (one per group of neighbouring requests)
        self.cu = torch.arange(0, (S + 1) * cap, cap, dtype=torch.int32, device=dev)
        self._layouts = {}
        # one request's slot as a cache of cap tokens
        self.slot = self._group_layout(1)
        # one query per (request, layer, head), [S, L, Hq, 128] contiguous
        self.step_layout = self._layout(S, window=1, q_strides=(L * Hq * d, Hq * d, d, d))
        # one workspace serves every group size (the work-item size depends on it)
        sizes = [jacap_workspace_size(self._group_layout(n), self.budget) for n in range(1, S + 1)]
        if min(sizes) == 0:
            raise JacapError(1, "jacap_workspace_size")
        nbytes = max(sizes)
        self.ws = torch.empty(nbytes, dtype=torch.uint8, device=dev)
        self._scores = torch.empty(L * Hkv * S * cap, dtype=torch.float32, device=dev)
        self._idx = torch.empty(L * Hkv * S * self.budget, dtype=torch.int32, device=dev)
        self._kept = torch.empty((S,), dtype=torch.int32, device=dev)
        self._views(1)

    def _views(self, n):
        L, Hkv = self.L, self.Hkv
        self.scores = self._scores[:L * Hkv * n * self.cap].view(L, Hkv, n * self.cap)
        self.idx = self._idx[:L * Hkv * n * self.budget].view(L, Hkv, n, self.budget)
        self.kept = self._kept[:n]

    def _layout(self, num_seqs, window, q_strides) -> jacap_layout:
        lay = jacap_layout()
        lay.num_seqs = num_seqs
        lay.cu_seqlens = self.cu.data_ptr()
        lay.max_seqlen = self.cap
        lay.total_tokens = num_seqs * self.cap
        lay.num_layers, lay.num_q_heads, lay.num_kv_heads, lay.head_dim = self.L, self.Hq, self.Hkv, 128
        lay.window = window
        lay.dtype = JACAP_BF16 if self.dtype == torch.bfloat16 else JACAP_F32
        st = self._k.stride()  # [L, Hkv, S, cap, 128]
        lay.kv_stride_layer, lay.kv_stride_head, lay.kv_stride_token = st[0], st[1], st[3]
        lay.q_stride_seq, lay.q_stride_layer, lay.q_stride_head, lay.q_stride_pos = q_strides
        return lay

    def _group_layout(self, n) -> jacap_layout:
        """n neighbouring requests' slots as one cache: request j of the group is
        tokens j cap .. (j + 1) cap - 1 (the storage puts them next to each
        other on the token axis of every (layer, KV head) plane)."""
        if n not in self._layouts:
            self._layouts[n] = self._layout(n, window=1, q_strides=(128, 128, 128, 128))
        return self._layouts[n]

    def _merge(self, q, reset: bool, stream=None):
        """q: [S, L, Hq, m, 128] queries (the slot dtype, channel contiguous)."""
        if q.dtype != self.dtype or q.stride(-1) != 1 or tuple(q.shape[:3]) != (self.S, self.L, self.Hq):
            raise ValueError("queries must be [S, L, Hq, m, 128] in the cache dtype")
        lay = self._layout(self.S, q.shape[3], (q.stride(0), q.stride(1), q.stride(2), q.stride(3)))
        _check(jacap_stats_update(lay, _ptr(q), 1 if reset else 0, _ptr(self.stats), _ptr(self.counts),
                                  _stream(stream)), "jacap_stats_update")

    def start(self, k0, v0, q_win, lengths, stream=None):
        """Load the prefill caches (k0, v0: [S, L, Hkv, n, 128], request s using
        its first lengths[s] < cap rows) and start the statistics from the
        prefill window queries q_win [S, L, Hq, w, 128]."""
        if any(n < 0 or n >= self.cap for n in lengths):
            raise ValueError("a prefill cache must hold fewer than budget + interval tokens; evict it first")
        n = k0.shape[3]
        self.k[:, :, :, :n].copy_(k0)
        self.v[:, :, :, :n].copy_(v0)
        ar = torch.arange(self.cap, dtype=torch.int32, device=self.pos.device)
        self.pos.copy_(torch.where(ar < torch.tensor(lengths, device=ar.device)[:, None], ar, -1)[:, None, None, :]
                       .expand_as(self.pos))
        self.lengths = list(lengths)
        self.next_id = list(lengths)
        self._merge(q_win, reset=True, stream=stream)

    def append(self, k_new, v_new, q_new, stream=None):
        """One decode step for every request: k_new, v_new [S, L, Hkv, 128],
        q_new [S, L, Hq, 128]. Returns the requests whose cache is now full
        (each must be evicted before its next append)."""
        full = [s for s in range(self.S) if self.lengths[s] >= self.cap]
        if full:
            raise RuntimeError(f"request {full[0]} is full; evict it first")
        dev = self._k.device
        rows = torch.tensor(self.lengths, dtype=torch.long, device=dev)
        reqs = torch.arange(self.S, device=dev)
        # one indexed copy per tensor for all requests (each writes its next free row)
        self._k[:, :, reqs, rows] = k_new.permute(1, 2, 0, 3).to(self.dtype)
        self._v[:, :, reqs, rows] = v_new.permute(1, 2, 0, 3).to(self.dtype)
        ids = torch.tensor(self.next_id, dtype=torch.int32, device=dev)
        self._pos[:, :, reqs, rows] = ids.view(1, 1, self.S).expand(self.L, self.Hkv, self.S)
        self.lengths = [n + 1 for n in self.lengths]
        self.next_id = [n + 1 for n in self.next_id]
        self.merge_queries(q_new, stream)
        return [s for s in range(self.S) if self.lengths[s] >= self.cap]

    def merge_queries(self, q_new, stream=None):
        """Merge one decode step's queries [S, L, Hq, 128] into the running statistics."""
        if q_new.is_contiguous() and q_new.dtype == self.dtype and tuple(q_new.shape) == (self.S, self.L, self.Hq, 128):
            _check(jacap_stats_update(self.step_layout, _ptr(q_new), 0, _ptr(self.stats), _ptr(self.counts),
                                      _stream(stream)), "jacap_stats_update")
        else:
            self._merge(q_new.unsqueeze(3), reset=False, stream=stream)

    def evict(self, s: int, stream=None, events=None, tail=None):
        """Score request s's full slot with the running statistics, select the
        budget best tokens and compact them in place to rows 0 .. budget - 1.
        ``events``: JACAP_SCORE_KERNELS + 1 torch.cuda.Event recorded around
        the scoring kernels; ``tail``: one more, recorded after the selection
        with its in-place compaction (one launch)."""
        self._evict_group(s, s + 1, stream, events, tail)

    def evict_many(self, requests, stream=None):
        """Evict every listed (full) request; neighbouring requests go through
        one pass together. Returns the groups (first, end) that were evicted."""
        groups = []
        for s in sorted(set(requests)):
            if groups and groups[-1][1] == s:
                groups[-1][1] = s + 1
            else:
                groups.append([s, s + 1])
        for a, b in groups:
            self._evict_group(a, b, stream)
        return [tuple(g) for g in groups]

    def schedule_info(self, requests: int | None = None):
        """(schedule, roles) of the scoring pass over ``requests`` slots evicted together
        (default: all), as jacap_schedule_info reports it."""
        lay = self._group_layout(self.S if requests is None else int(requests))
        sched, roles = jacap_schedule_info(lay, self.params)
        if sched < 0:
            raise JacapError(-sched, "jacap_schedule_info")
        return sched, roles

    def _evict_group(self, a, b, stream=None, events=None, tail=None):
        if any(self.lengths[s] != self.cap for s in range(a, b)):
            raise RuntimeError("only full slots are evicted")
        n = b - a
        lay, st = self._group_layout(n), _stream(stream)
        handles = [e.cuda_event for e in events] if events is not None else []
        stats = ctypes.c_void_p(self.stats[a].data_ptr())
        counts = ctypes.c_void_p(self.counts[a].data_ptr())
        k, v, pos = _ptr(self._k[0, 0, a]), _ptr(self._v[0, 0, a]), _ptr(self._pos[0, 0, a])
        self._views(n)
        _check(jacap_score_stats(lay, self.params, stats, counts, k, v, _ptr(self.scores), _ptr(self.ws),
                                 self.ws.numel(), st, handles), "jacap_score_stats")
        _check(jacap_select_compact_inplace(lay, _ptr(self.scores), self.budget, _ptr(self.idx), _ptr(self.kept), k,
                                            v, pos, self.preserve_order, _ptr(self.ws), self.ws.numel(), st),
               "jacap_select_compact_inplace")
        if tail is not None:
            tail[0].record(stream)
        for s in range(a, b):
            self.lengths[s] = self.budget
        self.events += n
        self.passes += 1

    def step(self, k_new, v_new, q_new, stream=None):
        """append() then evict every request that became full (neighbours together)."""
        full = self.append(k_new, v_new, q_new, stream)
        self.evict_many(full, stream)
        return full

    def check(self, stream=None):
        _check(jacap_device_status(_ptr(self.ws), _stream(stream)), "device status")


class HostEvictor:
    """Eviction of a cache held in pinned host memory (an offloaded cache),
    through ``jacap_evict_host``.

    The library moves the layers to the device in groups of ``group_layers``
    through two device buffers: while group g is scored, selected and
    compacted on the compute stream, group g + 1 is copied on a copy stream.
    Each ``run()`` returns when the kept positions (and, with ``copy_rows``,
    the retained K and V rows) are in host memory.

    q_win_h [S, L, Hq, w, 128], k_h and v_h [L, Hkv, N, 128]: contiguous
    tensors in pinned host memory; cu_seqlens: int32 [S + 1] (host or device),
    fixed with ``seqlens`` at construction like the layout; ``out_factor``:
    optional float32 [L][Hkv][128][128] device tensor, as for ``Evictor``.
    After ``run()``: ``idx_h`` [L, Hkv, S, B], ``kept_h`` [S] and, with
    ``copy_rows``, ``k_out_h``, ``v_out_h`` [L, Hkv, S, B, 128] (pinned host).
    The only device memory is one buffer of ``jacap_host_buffer_size`` bytes.
    """

    def __init__(self, q_win_h, k_h, v_h, cu_seqlens, seqlens, num_q_heads: int, budget: int,
                 params: jacap_params | None = None, group_layers: int = 8, device="cuda", out_factor=None,
                 copy_rows: bool = True):
        dev = torch.device(device)
        for name, t in (("q_win_h", q_win_h), ("k_h", k_h), ("v_h", v_h)):
            if t.device.type != "cpu" or not t.is_pinned() or not t.is_contiguous():
                raise ValueError(f"{name} must be a contiguous tensor in pinned host memory")
        L, Hkv, N, d = k_h.shape
        S = len(seqlens)
        if v_h.shape != k_h.shape or q_win_h.shape[:2] != (S, L):
            raise ValueError("k_h and v_h must be [L, Hkv, N, 128] and q_win_h [S, L, Hq, w, 128]")
        if out_factor is not None and (out_factor.dtype != torch.float32 or tuple(out_factor.shape) != (L, Hkv, d, d)
                                       or not out_factor.is_contiguous() or out_factor.device != dev):
            raise ValueError("out_factor must be a contiguous float32 [L][Hkv][128][128] tensor on the device")
        self.out_factor = out_factor
        self.L, self.S, self.gl = L, S, max(1, min(int(group_layers), L))
        self.q_h, self.k_h, self.v_h = q_win_h, k_h, v_h
        self.budget = int(budget)
        self.params = params if params is not None else jacap_params()
        self.num_q_heads = num_q_heads
        self.seqlens = list(seqlens)
        self.copy_rows = bool(copy_rows)
        self.cu_h = torch.as_tensor(cu_seqlens, dtype=torch.int32).cpu().contiguous()
        self.lay = Cache(q_win_h, k_h, v_h, self.cu_h, self.seqlens, num_q_heads).layout()  # cu_seqlens: host
        nbytes = jacap_host_buffer_size(self.lay, self.budget, self.gl, 1 if self.copy_rows else 0)
        if nbytes == 0:
            raise JacapError(1, "jacap_host_buffer_size")
        self.dev_buf = torch.empty(nbytes + 1024, dtype=torch.uint8, device=dev)
        off = (-self.dev_buf.data_ptr()) % 1024
        self.dev_buf = self.dev_buf[off:off + nbytes]
        self.idx_h = torch.empty((L, Hkv, S, self.budget), dtype=torch.int32).pin_memory()
        self.kept_h = torch.empty((S,), dtype=torch.int32).pin_memory()
        self.k_out_h = self.v_out_h = None
        if self.copy_rows:
            self.k_out_h = torch.empty((L, Hkv, S, self.budget, d), dtype=k_h.dtype).pin_memory()
            self.v_out_h = torch.empty_like(self.k_out_h).pin_memory()
        self.copy_stream = torch.cuda.Stream(device=dev)

    @property
    def h2d_bytes(self) -> int:
        """Bytes one ``run()`` copies host->device (the cache and its window; cu_seqlens aside)."""
        return sum(t.numel() * t.element_size() for t in (self.q_h, self.k_h, self.v_h))

    @property
    def d2h_bytes(self) -> int:
        """Bytes one ``run()`` copies device->host: positions, kept counts and, with copy_rows, the rows."""
        rows = 0 if not self.copy_rows else 2 * self.k_out_h.numel() * self.k_out_h.element_size()
        return (self.idx_h.numel() + self.kept_h.numel()) * 4 + rows

    def run(self, stream=None):
        of = _ptr(self.out_factor) if self.out_factor is not None else ctypes.c_void_p(0)
        st = jacap_evict_host(self.lay, self.params, self.budget, self.gl, _ptr(self.q_h), _ptr(self.k_h),
                              _ptr(self.v_h), of, _ptr(self.idx_h), _ptr(self.kept_h),
                              _ptr(self.k_out_h), _ptr(self.v_out_h), _ptr(self.dev_buf), self.dev_buf.numel(),
                              _stream(stream), _stream(self.copy_stream))
        _check(st, "jacap_evict_host")

    def check(self, stream=None):
        """Errors are returned by ``run()`` itself (it raises); nothing more to read."""
        return None
