"""Seeded synthetic KV caches shaped like the paper's long-context workloads.

The paper evaluates on LongBench, Needle-in-a-Haystack and AIME25 with
Llama-3.1-8B / Qwen3 / Mistral-class models (Sec. 4); no dataset or weight is
used here. These generators stand in for them with the same cache shapes
(32 layers, 32 query / 8 KV heads, head_dim 128) and context lengths, and
with structure that makes the method's weighting non-trivial (per-channel
scales, query-key correlation, outlier channels, attention sinks).

This module holds none of the method's arithmetic: it only draws numbers.
Both the CUDA path and the oracle consume the tensors it returns.

Layouts: k, v are [L, Hkv, N_tot, 128]; q_win is [S, L, Hq, w, 128];
cu_seqlens is int32 [S + 1]. Query head h is served by KV head h // G.
Every (request, layer, KV head) unit draws from its own generator seeded by
numpy.random.SeedSequence([seed, request, layer, kv_head]), so a unit's bytes
do not depend on which other units are generated.
"""

from __future__ import annotations

import math
from dataclasses import dataclass, field, replace

import numpy as np
import torch


@dataclass(frozen=True)
class Workload:
    name: str
    num_layers: int
    num_q_heads: int
    num_kv_heads: int
    seqlens: tuple
    window: int
    budget: int
    dtype: str = "bf16"          # "bf16" or "f32"
    dist: str = "latent"         # "latent" (configs 2-5) or "outlier" (config 1)
    seed: int = 0
    head_dim: int = 128
    corr: float = 0.3            # shared-latent weight of K and the window queries
    scale_sigma: float = 0.5     # LogNormal(0, sigma) per-channel scales of K and V
    outlier_channels: int = 0    # key channels scaled by outlier_scale ("outlier")
    outlier_scale: float = 1.0
    sink_tokens: int = 0         # first tokens whose keys are scaled by sink_scale
    sink_scale: float = 1.0
    budgets: tuple = field(default=())

    @property
    def total_tokens(self) -> int:
        return int(sum(self.seqlens))

    @property
    def torch_dtype(self):
        return torch.bfloat16 if self.dtype == "bf16" else torch.float32

    def algorithmic_bytes(self, budget=None) -> int:
        """Q window + K + V read, retained K and V written (elements x size)."""
        b = self.budget if budget is None else budget
        es = 2 if self.dtype == "bf16" else 4
        d = self.head_dim
        S = len(self.seqlens)
        q = S * self.num_layers * self.num_q_heads * self.window * d * es
        kv = 2 * self.num_layers * self.num_kv_heads * self.total_tokens * d * es
        kept = sum(min(n, b) for n in self.seqlens)
        out = 2 * self.num_layers * self.num_kv_heads * kept * d * es
        return q + kv + out


def _ragged_lengths(seed: int, count: int, lo: int, hi: int) -> tuple:
    g = np.random.Generator(np.random.PCG64(np.random.SeedSequence([seed, 999])))
    return tuple(int(x) for x in g.integers(lo, hi + 1, size=count))


def config(index: int, budget: int | None = None) -> Workload:
    """The five evaluation configurations (1-based, in the order they are listed)."""
    if index == 1:
        w = Workload("single-layer 8/8 heads, n=4096, fp32 with outlier key channels", 1, 8, 8, (4096,), 32, 256,
                     dtype="f32", dist="outlier", seed=0, outlier_channels=4, outlier_scale=8.0)
    elif index == 2:
        w = Workload("Llama-3-8B-shaped GQA cache, n=32768", 32, 32, 8, (32768,), 32, 512, seed=2,
                     budgets=(128, 512, 2048))
    elif index == 3:
        w = Workload("Mistral-7B-shaped cache, n=16384, 4 sink tokens", 32, 32, 8, (16384,), 64, 1638, seed=3,
                     sink_tokens=4, sink_scale=4.0)
    elif index == 4:
        w = Workload("long-context Llama-3-8B-shaped cache, n=131072", 32, 32, 8, (131072,), 32, 1024, seed=4)
    elif index == 5:
        w = Workload("ragged batch of 16 Llama-3-8B-shaped requests, n~U[2048,65536]", 32, 32, 8,
                     _ragged_lengths(5, 16, 2048, 65536), 32, 512, seed=5)
    else:
        raise ValueError(index)
    return replace(w, budget=budget) if budget is not None else w


def _gen(device, *key) -> torch.Generator:
    s = int(np.random.SeedSequence([int(k) for k in key]).generate_state(1, dtype=np.uint64)[0] & ((1 << 63) - 1))
    g = torch.Generator(device=device)
    g.manual_seed(s)
    return g


def _outlier_channels(wl: Workload) -> torch.Tensor:
    g = torch.Generator(device="cpu")
    g.manual_seed(0)
    return torch.randperm(wl.head_dim, generator=g)[: wl.outlier_channels]


def fill_unit(wl: Workload, s: int, layer: int, g: int, n: int, device):
    """(k, v, q) for one unit: k, v [n, d]; q [G, w, d], all float32 on device."""
    d, w = wl.head_dim, wl.window
    G = wl.num_q_heads // wl.num_kv_heads
    gen = _gen(device, wl.seed, s, layer, g)
    if wl.dist == "outlier":
        k = torch.randn(n, d, generator=gen, device=device)
        v = torch.randn(n, d, generator=gen, device=device)
        q = torch.randn(G, w, d, generator=gen, device=device)
        k[:, _outlier_channels(wl).to(device)] *= wl.outlier_scale
    elif wl.dist == "latent":
        sgen = _gen(device, wl.seed, 7777, layer, g)
        sk = torch.exp(wl.scale_sigma * torch.randn(d, generator=sgen, device=device))
        sv = torch.exp(wl.scale_sigma * torch.randn(d, generator=sgen, device=device))
        a, b = math.sqrt(wl.corr), math.sqrt(1.0 - wl.corr)
        z = torch.randn(max(n, w), d, generator=gen, device=device)
        k = sk * (a * z[:n] + b * torch.randn(n, d, generator=gen, device=device))
        v = sv * torch.randn(n, d, generator=gen, device=device)
        zq = z[max(n, w) - w:]  # latent of the last w positions
        q = a * zq.unsqueeze(0) + b * torch.randn(G, w, d, generator=gen, device=device)
    else:
        raise ValueError(wl.dist)
    if wl.sink_tokens:
        k[: wl.sink_tokens] *= wl.sink_scale
    return k, v, q


@dataclass
class Tensors:
    q_win: torch.Tensor
    k: torch.Tensor
    v: torch.Tensor
    cu_seqlens: torch.Tensor
    seqlens: list


def generate(wl: Workload, device="cpu") -> Tensors:
    """The whole cache of ``wl`` on ``device`` in the library's layout."""
    L, Hq, Hkv, d, w = wl.num_layers, wl.num_q_heads, wl.num_kv_heads, wl.head_dim, wl.window
    G = Hq // Hkv
    S = len(wl.seqlens)
    N = wl.total_tokens
    dt = wl.torch_dtype
    k = torch.empty((L, Hkv, N, d), dtype=dt, device=device)
    v = torch.empty((L, Hkv, N, d), dtype=dt, device=device)
    q = torch.empty((S, L, Hq, w, d), dtype=dt, device=device)
    cu = [0]
    for n in wl.seqlens:
        cu.append(cu[-1] + int(n))
    for s, n in enumerate(wl.seqlens):
        for layer in range(L):
            for g in range(Hkv):
                ku, vu, qu = fill_unit(wl, s, layer, g, int(n), device)
                k[layer, g, cu[s]:cu[s + 1]] = ku.to(dt)
                v[layer, g, cu[s]:cu[s + 1]] = vu.to(dt)
                q[s, layer, g * G:(g + 1) * G] = qu.to(dt)
    cu_t = torch.tensor(cu, dtype=torch.int32, device=device)
    return Tensors(q, k, v, cu_t, [int(n) for n in wl.seqlens])


def unit_arrays(t: Tensors, num_q_heads: int, s: int, layer: int, g: int):
    """Host float64 copies (exact) of one unit: (q_group [G,w,d], K [n,d], V [n,d])."""
    Hkv = t.k.shape[1]
    G = num_q_heads // Hkv
    cu = t.cu_seqlens.cpu().tolist()
    a, b = cu[s], cu[s + 1]
    q = t.q_win[s, layer, g * G:(g + 1) * G].float().cpu().double().numpy()
    k = t.k[layer, g, a:b].float().cpu().double().numpy()
    v = t.v[layer, g, a:b].float().cpu().double().numpy()
    return q, k, v
