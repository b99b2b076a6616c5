"""The seeded synthetic caches: shapes, determinism, unit independence and
the distribution structure each configuration asks for (CPU only)."""

from dataclasses import replace

import numpy as np
import torch

from paper_2609_08131_gb300.workloads import Workload, config, fill_unit, generate, unit_arrays


def test_config_shapes_match_the_evaluation_table():
    c = [config(i) for i in range(1, 6)]
    assert (c[0].num_layers, c[0].num_q_heads, c[0].num_kv_heads, c[0].seqlens, c[0].window, c[0].budget,
            c[0].dtype) == (1, 8, 8, (4096,), 32, 256, "f32")
    assert (c[1].num_layers, c[1].num_q_heads, c[1].num_kv_heads, c[1].seqlens, c[1].window) == (32, 32, 8, (32768,), 32)
    assert c[1].budgets == (128, 512, 2048)
    assert (c[2].seqlens, c[2].window, c[2].budget, c[2].sink_tokens) == ((16384,), 64, 1638, 4)
    assert (c[3].seqlens, c[3].budget) == ((131072,), 1024)
    assert len(c[4].seqlens) == 16 and all(2048 <= n <= 65536 for n in c[4].seqlens) and c[4].budget == 512
    assert c[4].seqlens == config(5).seqlens  # seeded


def test_algorithmic_bytes_config2():
    # 8 MiB of Q window + 2 x 2 GiB of K/V + 2 x 32x8x512x128x2 retained
    assert config(2).algorithmic_bytes() == 8388608 + 4294967296 + 67108864


def small():
    return Workload("t", 2, 8, 2, (300, 77), 16, 32, seed=5)


def test_generation_is_deterministic_and_per_unit():
    wl = small()
    a = generate(wl, "cpu")
    b = generate(wl, "cpu")
    assert torch.equal(a.k, b.k) and torch.equal(a.v, b.v) and torch.equal(a.q_win, b.q_win)
    # a unit's bytes do not depend on the other units that are generated
    other = replace(wl, seqlens=(77,))
    k, v, q = fill_unit(wl, 1, 1, 1, 77, "cpu")
    assert torch.equal(a.k[1, 1, 300:377], k.to(torch.bfloat16))
    assert a.cu_seqlens.tolist() == [0, 300, 377]
    assert other.total_tokens == 77


def test_unit_arrays_are_exact_copies():
    wl = small()
    t = generate(wl, "cpu")
    q, K, V = unit_arrays(t, wl.num_q_heads, 1, 0, 1)
    assert K.dtype == np.float64 and K.shape == (77, 128) and q.shape == (4, 16, 128)
    assert np.array_equal(K, t.k[0, 1, 300:377].double().numpy())


def test_latent_correlation_and_scales():
    wl = Workload("t", 1, 4, 1, (4096,), 64, 32, seed=9)
    k, v, q = fill_unit(wl, 0, 0, 0, 4096, "cpu")
    # queries at the window positions share the latent with the keys there
    kw = k[-64:] / k.std(dim=0)
    r = torch.corrcoef(torch.stack([kw.flatten(), q[0].flatten()]))[0, 1].item()
    assert 0.15 < r < 0.45
    ratio = k.std(dim=0).max() / k.std(dim=0).min()
    assert ratio > 2.0  # LogNormal(0, 0.5) channel scales


def test_outlier_channels_and_sinks():
    wl = config(1)
    k, v, q = fill_unit(wl, 0, 0, 0, 4096, "cpu")
    sd = k.std(dim=0)
    assert int((sd > 4).sum()) == 4
    ws = Workload("t", 1, 4, 1, (2000,), 16, 32, seed=3, sink_tokens=4, sink_scale=4.0)
    k, v, q = fill_unit(ws, 0, 0, 0, 2000, "cpu")
    assert k[:4].norm(dim=1).mean() > 3 * k[4:].norm(dim=1).mean()
