#!/usr/bin/env python
"""Throughput of Jacap's prefill eviction pass on GB300; prints ONE JSON line.

A step is one whole pass (jacap_score + jacap_select_compact, i.e. the
selection and the compaction in one launch: every row of the hot path) over one synthetic Llama-3-8B-shaped cache (32 layers,
32 query / 8 KV heads, head_dim 128, n = 32768, w = 32, B = 512, bf16), with
the inputs resident in HBM. The metric is evicted-cache tokens per second per
layer-pass, sum_s n_s * L / t_step, summed over ranks.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--budget B] [--config C]
  python bench.py --impl reference ...   # the float64 CPU oracle, bounded sample

Under torchrun every rank evicts its own cache of the same shape (weak
scaling, no collective on the data path); the time is the max over ranks.
"""

from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "evicted-cache tokens/s per layer-pass (1 GB300) and % of HBM roofline"
UNIT = "tokens/s"
NOMINAL_HBM_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1,
                   help="ranks (one GPU each); without a launcher's environment (WORLD_SIZE) the script "
                        "re-runs itself under torch.distributed.run with this many ranks")
    p.add_argument("--backend", default="nccl", choices=["nccl", "gloo"],
                   help="process-group backend of the multi-rank run (gloo: CPU-only checks of the launcher)")
    p.add_argument("--steps", type=int, default=500)
    p.add_argument("--warmup", type=int, default=10)
    p.add_argument("--impl", default="ours", choices=["ours", "reference"])
    p.add_argument("--config", type=int, default=2)
    p.add_argument("--trace-report", action="store_true",
                   help="diagnostic (a JACAP_TRACE=1 build): print the per-CTA time accounting of one pass, no bench line")
    p.add_argument("--schedule", default="auto", choices=["auto", "separate", "fused"],
                   help="Gram / factor / scores as separate kernels or one fused launch (auto: the library's choice)")
    p.add_argument("--budget", type=int, default=None)
    p.add_argument("--weighting", default="jacobian", choices=["jacobian", "linear"],
                   help="Eq. 8 softmax-aware weights (the method) or the linear S = I surrogate")
    p.add_argument("--covariance", default="diagonal", choices=["diagonal", "full"],
                   help="query-response variance from the diagonal Lambda_Q (the method) or the full "
                        "window covariance (App. B.2)")
    p.add_argument("--out-proj", type=int, default=0, metavar="D_O",
                   help="use true output directions u = W v with synthetic W (D_O x 128) per plane")
    p.add_argument("--decode", type=int, default=0, metavar="B",
                   help="measure decoding-stage eviction instead: one request whose cache slot of B + interval "
                        "tokens is scored with running query statistics and compacted to B")
    p.add_argument("--decode-model", default="nemotron-7b", choices=["nemotron-7b", "llama-3-8b"],
                   help="head layout of the decoding benchmark: Nemotron-7B (28 layers, 28 query / 4 KV heads, "
                        "the paper's decoding-stage model) or Llama-3-8B (32 layers, 32 / 8)")
    p.add_argument("--interval", type=int, default=128, help="decoding-stage eviction interval (tokens)")
    p.add_argument("--decode-requests", type=int, default=1,
                   help="decoding-stage eviction: requests whose slots fill on the same step (one pass for all)")
    p.add_argument("--preserve-order", action="store_true",
                   help="decoding-stage eviction: compact to ascending slot order instead of filling the holes")
    p.add_argument("--e2e-steps", type=int, default=10)
    p.add_argument("--e2e-group", type=int, default=8, help="layers per host->device copy group of the e2e pass")
    p.add_argument("--cpu-seconds", type=float, default=15.0)
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-graph", action="store_true", help="skip timing the pass replayed from a CUDA graph")
    p.add_argument("--layers", type=int, default=None,
                   help="override the layer count (small profiling captures; the line reports it)")
    p.add_argument("--extra-configs", default="4",
                   help="comma-separated evaluation configurations measured after the headline one in the same "
                        "run and reported under extra_configs ('' for none)")
    p.add_argument("--extra-steps", type=int, default=100)
    p.add_argument("--ref-seconds", type=float, default=150.0,
                   help="reference arm: CPU seconds the whole --steps + --warmup run is sized to")
    return p.parse_args()


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def aggregate_ranks(t_ms: float, tokens_layers: int, dist=None, device=None):
    """Whole-job throughput over ranks: every rank processed `tokens_layers`
    in `t_ms`; the job time is the max over ranks (weak scaling, replicas)."""
    world = 1
    if dist is not None and dist.is_initialized():
        import torch

        world = dist.get_world_size()
        if dist.get_backend() == "gloo":
            device = "cpu"
        x = torch.tensor([float(t_ms)], dtype=torch.float64, device=device)
        dist.all_reduce(x, op=dist.ReduceOp.MAX)
        t_ms = float(x.item())
        n = torch.tensor([int(tokens_layers)], dtype=torch.int64, device=device)
        dist.all_reduce(n, op=dist.ReduceOp.SUM)
        tokens_layers = int(n.item())
    return tokens_layers / (t_ms * 1e-3), t_ms, world


def recorded_traffic(kernel: str):
    """DRAM bytes per launch of `kernel` from the committed ncu record, or None
    when there is no record or the kernel's sources changed since the capture."""
    import hashlib

    try:
        with open(os.path.join(ROOT, "profiles", "dram_traffic.json")) as f:
            rec = json.load(f)["kernels"][kernel]
        h = hashlib.sha256()
        for src in rec["sources"]:
            with open(os.path.join(ROOT, src), "rb") as f:
                h.update(f.read())
        return int(rec["traffic_bytes_per_launch"]) if h.hexdigest() == rec["source_sha256"] else None
    except Exception:
        return None


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons while running."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "20"], stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.1)
        self.proc.terminate()
        self.proc.wait()
        rows = []
        for line in open(self.path):
            parts = [x.strip() for x in line.split(",")]
            if len(parts) == 8:
                rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}

        def num(x):
            try:
                return float(x)
            except ValueError:
                return None

        sm = [num(r[0]) for r in rows if num(r[0]) is not None]
        mx = [num(r[1]) for r in rows if num(r[1]) is not None]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[4 + i].lower() == "active"})
        pw = [num(r[2]) for r in rows if num(r[2]) is not None]
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows), "power_w_max": max(pw) if pw else None}


def workload_config(wl, budget, gpus, weighting="jacobian", out_proj=0, covariance="diagonal"):
    return {
        "workload": wl.name,
        "layers": wl.num_layers,
        "q_heads": wl.num_q_heads,
        "kv_heads": wl.num_kv_heads,
        "head_dim": wl.head_dim,
        "seqlens": list(wl.seqlens) if len(wl.seqlens) <= 4 else f"{len(wl.seqlens)} requests, sum {wl.total_tokens}",
        "window": wl.window,
        "budget": budget,
        "tau": 10.0,
        "weighting": weighting,
        "query_covariance": covariance,
        "output_directions": f"u = W v, synthetic W ({out_proj} x 128) per plane" if out_proj else "u = v (proxy)",
        "cache_dtype": wl.dtype,
        "l2": "inputs larger than L2: each step streams the whole cache (K and V alone are "
              f"{2 * wl.num_layers * wl.num_kv_heads * wl.total_tokens * wl.head_dim * (2 if wl.dtype == 'bf16' else 4) / 1e9:.2f} GB)",
        "parallelism": f"{gpus} independent replica(s), one cache per GPU",
    }


# ------------------------------------------------------------------ oracle --
def oracle_sample(wl, budget, seconds, device, tensors=None, weighting="jacobian", out_factor=None,
                  covariance="diagonal"):
    """Time the float64 oracle on whole units of the workload for ~`seconds`.

    Returns (tokens_layers_per_s, sample_description, wall_s)."""
    from oracle import JacapParams, oracle_unit
    from paper_2609_08131_gb300.workloads import fill_unit, unit_arrays

    units = [(s, l, g) for l in range(wl.num_layers) for g in range(wl.num_kv_heads) for s in range(len(wl.seqlens))]
    done, tok, t_total = 0, 0, 0.0
    for (s, l, g) in units:
        n = wl.seqlens[s]
        if tensors is not None:
            q, K, V = unit_arrays(tensors, wl.num_q_heads, s, l, g)
        else:
            k, v, qq = fill_unit(wl, s, l, g, n, "cpu")
            dt = wl.torch_dtype
            q = qq.to(dt).double().numpy()
            K = k.to(dt).double().numpy()
            V = v.to(dt).double().numpy()
        t0 = time.perf_counter()
        proj = None if out_factor is None else out_factor[l, g].double().cpu().numpy()
        oracle_unit(q, K, V, budget, JacapParams(linear_weighting=weighting == "linear",
                                                 full_covariance=covariance == "full"), out_proj=proj)
        t_total += time.perf_counter() - t0
        done += 1
        tok += n
        if t_total >= seconds:
            break
    # tokens x layers: a unit is one (layer, KV head) of a request, i.e. 1/Hkv of a layer-pass
    value = tok / wl.num_kv_heads / t_total
    desc = f"{done} whole unit(s) (request, layer, KV head) of {tok} tokens in total, float64 numpy"
    return value, desc, t_total


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if int(os.environ.get("WORLD_SIZE", "1")) > 1:
        # the ranks meet once over gloo (host only: the oracle uses no GPU);
        # then rank 0 alone runs the oracle and the others exit without work
        import torch.distributed as dist

        dist.init_process_group("gloo")
        dist.barrier()
        dist.destroy_process_group()
    if rank != 0:
        return 0
    from oracle import JacapParams, oracle_unit
    from paper_2609_08131_gb300.workloads import config, fill_unit

    wl = config(args.config)
    budget = args.budget or wl.budget
    # per-step sample: a prefix of one unit, sized so K + W steps take ~150 s
    n_full = wl.seqlens[0]
    k, v, q = fill_unit(wl, 0, 0, 0, n_full, "cpu")
    dt = wl.torch_dtype
    K64, V64, Q64 = k.to(dt).double().numpy(), v.to(dt).double().numpy(), q.to(dt).double().numpy()
    t0 = time.perf_counter()
    P = JacapParams(linear_weighting=args.weighting == "linear", full_covariance=args.covariance == "full")
    oracle_unit(Q64, K64[:2048], V64[:2048], budget, P)
    per_tok = (time.perf_counter() - t0) / 2048
    target = args.ref_seconds / max(1, args.steps + args.warmup)
    m = int(max(min(256, n_full), min(n_full, target / per_tok)))
    for _ in range(args.warmup):
        oracle_unit(Q64, K64[:m], V64[:m], budget, P)
    times = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        oracle_unit(Q64, K64[:m], V64[:m], budget, P)
        times.append(time.perf_counter() - t0)
    avg = sum(times) / len(times)
    value = m / wl.num_kv_heads / avg
    sample = (f"each step: the float64 oracle on the first {m} tokens of one (layer, KV head) unit of the workload "
              f"(a sub-cache of {m} tokens); tokens x layers = {m}/{wl.num_kv_heads} per step")
    line = {
        "impl": "reference",
        "metric": METRIC,
        "value": value,
        "unit": UNIT,
        "n_gpus": int(os.environ.get("WORLD_SIZE", "1")),
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": avg * 1e3,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "f64",
        "data": "synthetic",
        "config": workload_config(wl, budget, args.gpus, args.weighting, covariance=args.covariance),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))
    return 0


# The fused schedule runs the Gram, the factor and the scores as one launch,
# timed in the Gram's slot of jacap_score_timed.
FUSED_NAME = "gram_factor_scores"
SCHEDULES = {"auto": 0, "separate": 1, "fused": 2}


def fused_kernel_names(kern, schedule):
    if schedule != 2:
        return kern
    out = {}
    for k, v in kern.items():
        if k == "gram":
            out[FUSED_NAME] = v
        elif k not in ("factor", "scores"):
            out[k] = v
    return out


def schedule_desc(schedule, roles):
    if schedule != 2:
        return {"kind": "separate kernels"}
    return {"kind": "fused Gram-factor-scores launch", "factor_ctas": roles[0], "gram_ctas": roles[1],
            "score_ctas": roles[2], "v_tiles_kept_in_l2_per_item": roles[3]}


# -------------------------------------------------------------------- ours --
def run_ours(args):
    import torch

    from paper_2609_08131_gb300 import SCORE_KERNEL_NAMES
    from paper_2609_08131_gb300.api import Cache, Evictor
    from paper_2609_08131_gb300.workloads import config, generate
    from dataclasses import replace

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    dist = None
    if world > 1:
        import torch.distributed as dist

        torch.cuda.set_device(local)
        dist.init_process_group(args.backend)
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)

    wl = config(args.config)
    budget = args.budget or wl.budget
    wl = replace(wl, seed=wl.seed + 1000 * rank, budget=budget)
    if args.layers:
        wl = replace(wl, num_layers=args.layers, name=wl.name + f", {args.layers} layers")
    t = generate(wl, dev)
    cache = Cache(t.q_win, t.k, t.v, t.cu_seqlens, t.seqlens, wl.num_q_heads)
    from paper_2609_08131_gb300 import jacap_params

    out_factor = None
    if args.out_proj:
        # synthetic output maps W (d_o x 128) per plane and their QR factors R
        # (F^T F = W^T W); set-up only, outside every timed region
        gen = torch.Generator(device=dev).manual_seed(7)
        W = torch.randn(wl.num_layers * wl.num_kv_heads, args.out_proj, 128, generator=gen, device=dev) / 128 ** 0.5
        out_factor = torch.linalg.qr(W, mode="r").R.reshape(wl.num_layers, wl.num_kv_heads, 128, 128).contiguous()
    ev = Evictor(cache, budget, jacap_params(linear_weighting=1 if args.weighting == "linear" else 0,
                                             full_covariance=1 if args.covariance == "full" else 0,
                                             schedule=SCHEDULES[args.schedule]),
                 out_factor=out_factor)
    stream = torch.cuda.current_stream(dev)

    def barrier():
        if dist is not None:
            dist.barrier()

    for _ in range(max(3, args.warmup)):
        ev.run()
    ev.check()
    if args.trace_report:
        from paper_2609_08131_gb300.api import cta_time_accounting

        ev.run()
        ev.check()
        print(json.dumps({"mode": "trace report", "config": workload_config(wl, budget, world, args.weighting,
                                                                              args.out_proj, args.covariance),
                          "schedule": schedule_desc(*ev.schedule_info()), "cta_time_accounting":
                          cta_time_accounting(ev)}))
        return 0

    # The end-to-end number first: right after seconds of HBM-saturating passes
    # the host link of these boxes delivers 70-120 GB/s instead of 211 for a
    # while (measured with plain host->device copies), which a steady
    # offloaded-cache loop, mostly waiting on its copies, does not see.
    e2e = None
    if not args.no_e2e:
        e2e = run_e2e(args, ev, t, stream, world, dist)

    K = args.steps
    nk = len(SCORE_KERNEL_NAMES)
    ev_score = [[torch.cuda.Event(enable_timing=True) for _ in range(nk + 1)] for _ in range(K)]
    ev_tail = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(K)]
    start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    # torch creates the CUDA event lazily: record each once so its handle exists
    for e in [x for row in ev_score + ev_tail for x in row] + [start, stop]:
        e.record(stream)
    torch.cuda.synchronize()
    sampler = ClockSampler(local)
    barrier()
    torch.cuda.synchronize()
    sampler.start()
    # the timed steps: the pass as a user runs it (consecutive kernels may
    # overlap their launch with the previous kernel's tail)
    start.record(stream)
    for i in range(K):
        ev.run()
    stop.record(stream)
    torch.cuda.synchronize()
    # the same pass captured once into a CUDA graph and replayed K times
    graph_ms = None
    if not args.no_graph:
        graph_ms = time_cuda_graph(ev, stream, dev, K)
    # per-kernel durations: the same steps again with an event between kernels
    # (which serialises the launches)
    KB = min(K, 100)
    kb0, kb1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    kb0.record(stream)
    for i in range(KB):
        ev.score(events=ev_score[i])
        ev.select_compact()
        ev_tail[i][0].record(stream)
    kb1.record(stream)
    torch.cuda.synchronize()
    clocks = sampler.stop()
    barrier()
    ev.check()
    t_ms = start.elapsed_time(stop) / K
    t_ms_events = kb0.elapsed_time(kb1) / KB
    value, t_ms, _ = aggregate_ranks(t_ms, sum(t.seqlens) * t.k.shape[0], dist, dev)

    # per-kernel average durations inside the timed region
    kern = {name: 0.0 for name in SCORE_KERNEL_NAMES}
    kern["select_compact"] = 0.0
    for i in range(KB):
        for j, name in enumerate(SCORE_KERNEL_NAMES):
            kern[name] += ev_score[i][j].elapsed_time(ev_score[i][j + 1])
        kern["select_compact"] += ev_score[i][nk].elapsed_time(ev_tail[i][0])
    kern = {k: v / KB for k, v in kern.items()}
    schedule, roles = ev.schedule_info()
    kern = fused_kernel_names(kern, schedule)

    L, Hkv, N, d = t.k.shape
    es = t.k.element_size()
    kv_bytes = L * Hkv * N * d * es
    kept_rows = L * Hkv * sum(min(n, budget) for n in t.seqlens)
    G = wl.num_q_heads // wl.num_kv_heads
    # Algorithmic bytes count the K, V, window and retained-row traffic only; the
    # logits/kappa round trip, the second read of V and the partials are extra
    # traffic (visible in `traffic`). With bf16 caches the Gram computes the
    # Eq. 8 weights itself (it also reads the logits/kappa rows).
    fused_weights = wl.dtype == "bf16"
    # full covariance on the tensor cores runs inside the K pass (one kernel)
    full_cov_fused = (wl.dtype == "bf16" and wl.window in (8, 16, 32, 64)
                      and (wl.num_q_heads // wl.num_kv_heads) * wl.window <= 128)
    alg_kernel = {
        "k_pass": kv_bytes,                       # K read once
        "gram": kv_bytes,                         # V read once
        "scores": kv_bytes + L * Hkv * N * 4,     # V read, scores written
        # scores read; retained K, V rows read and written
        "select_compact": L * Hkv * N * 4 + 4 * kept_rows * d * es,
    }
    if schedule == 2:  # one launch: V read once (its second read is extra traffic), scores written
        for k in ("gram", "scores"):
            del alg_kernel[k]
        alg_kernel[FUSED_NAME] = kv_bytes + L * Hkv * N * 4
    if not fused_weights:
        alg_kernel["weights"] = L * Hkv * N * (8 * G + 4)  # logits + kappa read, w written
    dom = max(alg_kernel, key=lambda k: kern[k])
    hbm, src = peaks()
    achieved = alg_kernel[dom] / (kern[dom] * 1e-3) / 1e9
    tokens_layers = sum(t.seqlens) * L
    alg_pass = wl.algorithmic_bytes(budget)

    extra = []
    for x in [c for c in args.extra_configs.split(",") if c.strip()]:
        if int(x) == args.config and not args.layers:
            continue
        extra.append(measure_config(int(x), args, dev, dist, rank, peaks()[0]))

    cpu = None
    if rank == 0 and not args.no_cpu_baseline:
        v_cpu, desc, wall = oracle_sample(wl, budget, args.cpu_seconds, dev, tensors=t, weighting=args.weighting,
                                          out_factor=out_factor, covariance=args.covariance)
        cpu = {"value": v_cpu, "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle",
               "sample": desc + f"; {wall:.1f} s of CPU work; numpy BLAS threads left at their default"}


    if rank == 0:
        line = {
            "metric": METRIC,
            "value": value,
            "unit": UNIT,
            "n_gpus": world,
            "steps": K,
            "warmup": args.warmup,
            "ms_per_step": t_ms,
            "higher_is_better": True,
            "scaling": "weak",
            "vs_baseline": None,
            "dtype": "bf16" if wl.dtype == "bf16" else "f32",
            "data": "synthetic",
            "config": workload_config(wl, budget, world, args.weighting, args.out_proj, args.covariance),
            "roofline": {
                "bound": "hbm",
                "kernel": dom,
                "achieved": achieved,
                "peak": hbm,
                "unit": "GB/s",
                "frac": achieved / hbm,
                "traffic": recorded_traffic(dom) if wl.num_layers == 32 and wl.seqlens == (32768,) else None,
                "peak_source": f"{src} copy bandwidth (MEASURED_PEAKS.json hbm_gbs)" if src == "measured" else "fallback",
            },
            "pass_roofline": {
                "algorithmic_bytes": alg_pass,
                "achieved_gbs": alg_pass / (t_ms * 1e-3) / 1e9,
                "frac_of_8tbs": alg_pass / (t_ms * 1e-3) / 1e9 / NOMINAL_HBM_GBS,
                "frac_of_measured": alg_pass / (t_ms * 1e-3) / 1e9 / hbm,
            },
            "kernel_ms": kern,
            "ms_per_step_with_kernel_events": t_ms_events,
            "ms_per_step_cuda_graph": graph_ms,
            # plan, query statistics, K pass (with the full-covariance kappa when that
            # runs on the tensor cores), [full covariance on the CUDA cores], unit
            # softmax statistics, [weights: float32 only], Gram, factor, scores (or the
            # three as one fused launch), selection + compaction
            "gpu_launches": K * (8 + (1 if args.covariance == "full" and not full_cov_fused else 0)
                                 + (0 if fused_weights else 1) - (2 if schedule == 2 else 0)),
            "schedule": schedule_desc(schedule, roles),
            "clocks": clocks,
            "extra_configs": extra,
            "cpu_baseline": cpu,
            "e2e": e2e,
        }
        print(json.dumps(line))
    if dist is not None:
        dist.destroy_process_group()
    return 0


def measure_config(index, args, dev, dist, rank, hbm):
    """One more evaluation configuration in the same run: the plain pass timed
    over --extra-steps steps (CUDA events around them), per-kernel durations
    from as many steps with an event between kernels, clocks sampled during
    both, and the pass roofline. The cache is freed afterwards."""
    import torch

    from paper_2609_08131_gb300 import SCORE_KERNEL_NAMES, jacap_params
    from paper_2609_08131_gb300.api import Cache, Evictor
    from paper_2609_08131_gb300.workloads import config, generate
    from dataclasses import replace

    wl = config(index)
    wl = replace(wl, seed=wl.seed + 1000 * rank)
    budget = wl.budget
    t = generate(wl, dev)
    ev = Evictor(Cache(t.q_win, t.k, t.v, t.cu_seqlens, t.seqlens, wl.num_q_heads), budget,
                 jacap_params(schedule=SCHEDULES[args.schedule]))
    stream = torch.cuda.current_stream(dev)
    for _ in range(max(3, args.warmup)):
        ev.run()
    ev.check()
    K = max(1, args.extra_steps)
    nk = len(SCORE_KERNEL_NAMES)
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(nk + 2)] for _ in range(K)]
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    for e in [x for row in evs for x in row] + [a, b]:
        e.record(stream)
    torch.cuda.synchronize()
    sampler = ClockSampler(dev.index)
    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize()
    sampler.start()
    a.record(stream)
    for _ in range(K):
        ev.run()
    b.record(stream)
    torch.cuda.synchronize()
    t_ms = a.elapsed_time(b) / K
    for i in range(K):
        ev.score(events=evs[i][:nk + 1])
        ev.select_compact()
        evs[i][nk + 1].record(stream)
    torch.cuda.synchronize()
    clocks = sampler.stop()
    ev.check()
    kern = {name: sum(evs[i][j].elapsed_time(evs[i][j + 1]) for i in range(K)) / K
            for j, name in enumerate(SCORE_KERNEL_NAMES)}
    kern["select_compact"] = sum(evs[i][nk].elapsed_time(evs[i][nk + 1]) for i in range(K)) / K
    schedule, roles = ev.schedule_info()
    kern = fused_kernel_names(kern, schedule)
    L = t.k.shape[0]
    value, t_ms, world = aggregate_ranks(t_ms, sum(t.seqlens) * L, dist, dev)
    alg = wl.algorithmic_bytes(budget)
    out = {
        "config": index,
        "workload": wl.name,
        "layers": wl.num_layers, "q_heads": wl.num_q_heads, "kv_heads": wl.num_kv_heads,
        "seqlens": list(wl.seqlens) if len(wl.seqlens) <= 4 else f"{len(wl.seqlens)} requests, sum {wl.total_tokens}",
        "window": wl.window, "budget": budget, "cache_dtype": wl.dtype,
        "steps": K,
        "value": value,
        "unit": UNIT,
        "ms_per_step": t_ms,
        "pass_roofline": {
            "algorithmic_bytes": alg,
            "achieved_gbs": alg / (t_ms * 1e-3) / 1e9,
            "frac_of_8tbs": alg / (t_ms * 1e-3) / 1e9 / NOMINAL_HBM_GBS,
            "frac_of_measured": alg / (t_ms * 1e-3) / 1e9 / hbm,
        },
        "kernel_ms": kern,
        "clocks": clocks,
        "gpu_launches": K * (8 + (0 if wl.dtype == "bf16" else 1) - (2 if schedule == 2 else 0)),
        "schedule": schedule_desc(schedule, roles),
    }
    del ev, t
    torch.cuda.empty_cache()
    return out


def time_cuda_graph(ev, stream, dev, K):
    """ms per pass replayed from a CUDA graph captured once (None if the
    capture is refused)."""
    import torch

    try:
        side = torch.cuda.Stream(device=dev)
        side.wait_stream(stream)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.stream(side):
            with torch.cuda.graph(g, stream=side, capture_error_mode="thread_local"):
                ev.run(side)
        stream.wait_stream(side)
        for _ in range(3):
            g.replay()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(K):
            g.replay()
        b.record(stream)
        torch.cuda.synchronize()
        ev.check()
        return a.elapsed_time(b) / K
    except RuntimeError as e:
        print(f"cuda graph timing skipped: {e}", file=sys.stderr)
        return None


def run_e2e(args, ev, t, stream, world, dist):
    """Same metric through the public API with the cache in pinned host memory
    (``jacap_evict_host`` via ``api.HostEvictor``): every step copies the whole
    cache host->device in layer groups, overlapped with the pass over the
    previous group, and brings the kept positions and the retained K and V rows
    back to host memory."""
    import torch

    from paper_2609_08131_gb300.api import HostEvictor

    c = ev.cache
    # every rank pins a host copy of its cache; if any rank cannot, all skip
    # the end-to-end number together (no rank may wait alone at a barrier)
    he, why = None, ""

    def pinned(x):  # straight into pinned memory: no pageable intermediate copy
        h = torch.empty(x.shape, dtype=x.dtype, pin_memory=True)
        h.copy_(x)
        return h

    try:
        he = HostEvictor(pinned(c.q_win), pinned(c.k), pinned(c.v), c.cu_seqlens, c.seqlens, c.num_q_heads,
                         ev.budget, ev.params, group_layers=args.e2e_group, device=c.k.device,
                         out_factor=ev.out_factor)
    except RuntimeError as e:
        why = str(e).splitlines()[0][:200]
    ok = torch.tensor([1 if he is not None else 0], device=c.k.device)
    if dist is not None:
        dist.all_reduce(ok, op=dist.ReduceOp.MIN)
    if int(ok.item()) == 0:
        return {"unavailable": "pinned host copy of the cache could not be made" + (f": {why}" if why else
                                                                                      " on every rank")}
    for _ in range(2):
        he.run(stream)
    torch.cuda.synchronize()
    # the host link on its own: one layer group's K copied host -> device
    # (before the timed loop and again after it: the host's memory and link
    # are shared with whatever else runs on the machine)
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    grp = he.k_h[:he.gl]
    probe = torch.empty(grp.shape, dtype=grp.dtype, device=c.k.device)

    def link():
        a.record(stream)
        for _ in range(3):
            probe.copy_(grp, non_blocking=True)
        b.record(stream)
        torch.cuda.synchronize()
        return 3 * grp.numel() * grp.element_size() / (a.elapsed_time(b) * 1e-3) / 1e9

    link_gbs = link()
    if dist is not None:
        dist.barrier()
    a.record(stream)
    n = max(1, args.e2e_steps)
    for _ in range(n):
        he.run(stream)
    b.record(stream)
    torch.cuda.synchronize()
    ms = a.elapsed_time(b) / n
    link_after_gbs = link()
    del probe
    if dist is not None:
        x = torch.tensor([ms], device=c.k.device)
        dist.all_reduce(x, op=dist.ReduceOp.MAX)
        ms = float(x.item())
    he.check()
    # the per-group layouts may cut a sequence into other chunks than the
    # whole-cache layout (another fp32 summation order), so a near tie at the
    # budget boundary may fall the other way; anything more is an error
    import numpy as np

    B = ev.budget
    mine, resident = he.idx_h.reshape(-1, B).numpy(), ev.idx.cpu().reshape(-1, B).numpy()
    differ = sum(len(np.setdiff1d(x, y)) for x, y in zip(mine, resident)) / max(1, mine.size)
    if differ > 1e-3:
        raise RuntimeError(f"the host-cache pass kept other tokens than the device-resident pass ({differ:.2e})")
    L = c.k.shape[0]
    return {"value": sum(t.seqlens) * L * world / (ms * 1e-3), "unit": UNIT, "h2d_bytes_per_step": he.h2d_bytes,
            "d2h_bytes_per_step": he.d2h_bytes, "ms_per_step": ms, "steps": n, "group_layers": he.gl,
            "idx_differ_vs_resident": differ, "h2d_link_gbs": link_gbs, "h2d_link_after_gbs": link_after_gbs,
            "h2d_achieved_gbs": he.h2d_bytes / (ms * 1e-3) / 1e9,
            "h2d_bound_ms": he.h2d_bytes / (link_gbs * 1e9) * 1e3, "api": "jacap_evict_host (C ABI)",
            "returns": "kept positions and the retained K and V rows, in pinned host memory"}


def run_decode(args):
    """Decoding-stage eviction events (reading R16) on one GPU.

    One request of the Nemotron-7B head layout (28 layers, 28 query / 4 KV
    heads; the paper's decoding-stage model) or, with --decode-model
    llama-3-8b, of the Llama-3-8B one (32 layers, 32 / 8), with a full slot of
    B + interval tokens; each timed step is one eviction
    event: the scoring pass with running statistics, TOP-B and the in-place
    compaction. After an event the slot is marked full again (its free rows
    still hold earlier tokens), so every event scores B + interval tokens."""
    import torch

    from paper_2609_08131_gb300 import SCORE_KERNEL_NAMES, jacap_params
    from paper_2609_08131_gb300.api import DecodeEvictor
    from paper_2609_08131_gb300.workloads import Workload, generate

    dev = torch.device("cuda", int(os.environ.get("LOCAL_RANK", "0")))
    torch.cuda.set_device(dev)
    B, D, S = args.decode, args.interval, max(1, args.decode_requests)
    cap = B + D
    # Nemotron-7B: 28 layers, 28 query / 4 KV heads (G = 7), head_dim 128
    L, Hq, Hkv, w = (28, 28, 4, 32) if args.decode_model == "nemotron-7b" else (32, 32, 8, 32)
    shape = "Nemotron-7B-shaped" if args.decode_model == "nemotron-7b" else "Llama-3-8B-shaped"
    wl = Workload(f"decoding-stage eviction, {shape}, reserved tokens B={B}, interval {D}, {S} request(s) "
                  "filling together", L, Hq, Hkv, (cap,) * S, w + 1, B, seed=40)
    t = generate(wl, dev)
    ev = DecodeEvictor(S, L, Hq, Hkv, B, D, dtype=t.k.dtype, params=jacap_params(), device=dev,
                       preserve_order=args.preserve_order)
    kk = t.k.view(L, Hkv, S, cap, 128).permute(2, 0, 1, 3, 4)
    vv = t.v.view(L, Hkv, S, cap, 128).permute(2, 0, 1, 3, 4)
    ev.start(kk[:, :, :, :cap - 1], vv[:, :, :, :cap - 1], t.q_win[:, :, :, :w].contiguous(), [cap - 1] * S)
    q_new = t.q_win[:, :, :, w].contiguous()
    ev.append(kk[:, :, :, cap - 1], vv[:, :, :, cap - 1], q_new)
    stream = torch.cuda.current_stream(dev)
    everyone = list(range(S))

    def refill():
        ev.lengths = [cap] * S

    def event(events=None, tail=None):  # all S slots in one pass
        refill()
        if S == 1:
            ev.evict(0, events=events, tail=tail)
        else:
            ev._evict_group(0, S, None, events, tail)

    for _ in range(max(3, args.warmup)):
        event()
    ev.check()
    K = args.steps
    nk = len(SCORE_KERNEL_NAMES)
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(nk + 2)] for _ in range(K)]
    start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    for e in [x for row in evs for x in row] + [start, stop]:
        e.record(stream)
    torch.cuda.synchronize()
    sampler = ClockSampler(dev.index)
    sampler.start()
    # the timed events: eviction as a user runs it (consecutive kernels prepare
    # their launch while the previous one runs) ...
    start.record(stream)
    for i in range(K):
        event()
    stop.record(stream)
    torch.cuda.synchronize()
    t_ms = start.elapsed_time(stop) / K
    # ... and again with an event between kernels for the breakdown
    start.record(stream)
    for i in range(K):
        event(events=evs[i][:nk + 1], tail=evs[i][nk + 1:])
    stop.record(stream)
    torch.cuda.synchronize()
    t_ms_events = start.elapsed_time(stop) / K
    clocks = sampler.stop()
    ev.check()
    kern = {name: sum(evs[i][j].elapsed_time(evs[i][j + 1]) for i in range(K)) / K
            for j, name in enumerate(SCORE_KERNEL_NAMES)}
    kern["select_compact_inplace"] = sum(evs[i][nk].elapsed_time(evs[i][nk + 1]) for i in range(K)) / K
    schedule, roles = ev.schedule_info()
    kern = fused_kernel_names(kern, schedule)
    # one decode step's statistics update (one query per layer and head)
    M = 200
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(stream)
    for _ in range(M):
        ev.merge_queries(q_new)
    b.record(stream)
    torch.cuda.synchronize()
    upd_us = a.elapsed_time(b) / M * 1e3
    kv_bytes = 2 * L * Hkv * S * cap * 128 * t.k.element_size()
    line = {
        "mode": "decode",
        "metric": "decoding-stage eviction: cached tokens x layers scored per second (1 GB300)",
        "value": S * cap * L / (t_ms * 1e-3),
        "unit": "tokens/s",
        "ms_per_event": t_ms,
        "ms_per_event_with_kernel_events": t_ms_events,
        "n_gpus": 1,
        "steps": K,
        "warmup": args.warmup,
        "higher_is_better": True,
        "dtype": "bf16",
        "data": "synthetic",
        "config": {"workload": wl.name, "layers": L, "q_heads": Hq, "kv_heads": Hkv, "head_dim": 128,
                   "requests": S, "slot_tokens": cap, "budget": B, "interval": D,
                   "statistics": "running, all queries seen",
                   "compaction": "ascending order" if args.preserve_order else "hole filling",
                   "l2": f"inputs larger than L2: each event reads K and V of the slot ({kv_bytes / 1e6:.0f} MB)"},
        "kernel_ms": kern,
        "stats_update_us_per_decode_step": upd_us,
        "event_hbm_fraction": {"kv_bytes": kv_bytes, "of_8tbs": kv_bytes / (t_ms * 1e-3) / 8e12},
        "clocks": clocks,
        # plan, query statistics, K pass, unit softmax statistics, Gram (with the
        # weights), factor, scores (or the three fused), selection with the hole
        # filling (ascending order: a second launch)
        "gpu_launches_per_event": 8 + (1 if args.preserve_order else 0) - (2 if schedule == 2 else 0),
        "schedule": schedule_desc(schedule, roles),
    }
    print(json.dumps(line))
    return 0


def free_port() -> int:
    import socket

    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def launch_ranks(args) -> int:
    """`--gpus N` (N > 1) outside a launcher: run this script again under
    torch.distributed.run with N ranks on this node (one GPU each, rendezvous
    on 127.0.0.1); rank 0 prints the JSON line. Returns the launcher's status."""
    if args.impl == "ours" and args.backend == "nccl":
        import torch

        have = torch.cuda.device_count()
        if have < args.gpus:
            print(f"bench.py: --gpus {args.gpus} needs {args.gpus} GPUs, this node has {have}", file=sys.stderr)
            return 2
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", f"--nproc-per-node={args.gpus}",
           "--master-addr", "127.0.0.1", "--master-port", str(free_port()), os.path.abspath(__file__),
           *sys.argv[1:]]
    return subprocess.call(cmd)


def main():
    args = parse()
    if args.gpus > 1 and "WORLD_SIZE" not in os.environ:
        return launch_ranks(args)
    if args.impl == "reference":
        return run_reference(args)
    if args.decode:
        return run_decode(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
