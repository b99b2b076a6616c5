"""bench.py starts its own ranks for --gpus N (CPU, gloo).

Without a launcher's environment, `bench.py --gpus 2` re-runs itself under
torch.distributed.run with two ranks that rendezvous on 127.0.0.1. The
reference arm (the CPU oracle) runs here so no GPU is needed: its ranks meet
over gloo, rank 0 measures and prints the one JSON line, which must report
both ranks.
"""

import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_bench_gpus_two_launches_two_ranks_itself():
    env = {k: v for k, v in os.environ.items()
           if k not in ("WORLD_SIZE", "RANK", "LOCAL_RANK", "MASTER_ADDR", "MASTER_PORT")}
    env["OMP_NUM_THREADS"] = "2"
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--gpus", "2",
                        "--backend", "gloo", "--config", "1", "--steps", "1", "--warmup", "0", "--ref-seconds", "1"],
                       capture_output=True, text=True, timeout=600, cwd=ROOT, env=env)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [x for x in r.stdout.splitlines() if x.startswith("{")]
    assert len(lines) == 1, r.stdout
    line = json.loads(lines[0])
    assert line["impl"] == "reference" and line["n_gpus"] == 2
    assert line["value"] > 0 and line["cpu_baseline"]["kind"] == "oracle"
