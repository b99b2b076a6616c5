"""Build and load libjacap.so (the sm_103a CUDA library behind the C ABI).

The library is compiled in-tree with nvcc (one -gencode: sm_103a), one
translation unit per process in parallel, then linked into
``paper_2609_08131_gb300/libjacap.so``. There is no fallback: if the library
cannot be built or loaded, ``load()`` raises.
"""

from __future__ import annotations

import ctypes
import os
import shutil
import subprocess
import threading
from concurrent.futures import ThreadPoolExecutor

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD = os.path.join(ROOT, "_build")
LIB = os.path.join(PKG, "libjacap.so")

SOURCES = ["jacap_api.cu", "k_stream.cu", "k_kpass.cu", "k_gram.cu", "k_factor.cu", "k_score.cu", "k_select.cu",
           "jacap_static.cu", "k_kfull.cu", "k_decode.cu", "jacap_host.cu", "k_fused.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
CFLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "--expt-relaxed-constexpr",
          "-I" + INCLUDE, "-I" + CSRC]

_lock = threading.Lock()
_handle = None


def nvcc() -> str:
    for cand in (shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libjacap")


def _sources_mtime() -> float:
    files = [os.path.join(CSRC, f) for f in os.listdir(CSRC)] + [os.path.join(INCLUDE, "jacap.h")]
    return max(os.path.getmtime(f) for f in files)


def build_flags() -> list:
    """Optional build variants, from the environment of the build:
    JACAP_NVTX=1 marks every kernel launch with an NVTX range (tracing);
    JACAP_CHECKED=1 makes the persistent kernels validate every work-item
    record against the cache bounds and report violations in the status word;
    JACAP_TRACE=1 records the fused schedule's per-unit timeline (%globaltimer
    stamps of each role's first and last work on the unit) in a section
    appended to the workspace."""
    extra = []
    if os.environ.get("JACAP_NVTX") == "1":
        extra.append("-DJACAP_NVTX")
    if os.environ.get("JACAP_CHECKED") == "1":
        extra.append("-DJACAP_CHECKED")
    if os.environ.get("JACAP_TRACE") == "1":
        extra.append("-DJACAP_TRACE")
    return extra


def _stamp() -> str:
    return " ".join(ARCH + CFLAGS + build_flags())


def build(verbose: bool = False, force: bool = False) -> str:
    """Compile and link libjacap.so; returns its path."""
    stamp_path = os.path.join(BUILD, "flags.txt")
    same_flags = os.path.exists(stamp_path) and open(stamp_path).read() == _stamp()
    if not force and same_flags and os.path.exists(LIB) and os.path.getmtime(LIB) >= _sources_mtime():
        return LIB
    os.makedirs(BUILD, exist_ok=True)
    cc = nvcc()
    extra = build_flags()

    def compile_one(src):
        obj = os.path.join(BUILD, src.replace(".cu", ".o"))
        cmd = [cc, *ARCH, *CFLAGS, *extra, "-c", os.path.join(CSRC, src), "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed for {src}:\n{r.stdout}\n{r.stderr}")
        if verbose and r.stderr.strip():
            print(r.stderr)
        return obj

    with ThreadPoolExecutor(max_workers=min(len(SOURCES), os.cpu_count() or 4)) as ex:
        objs = list(ex.map(compile_one, SOURCES))
    tmp = LIB + ".tmp"
    cmd = [cc, *ARCH, "-shared", "-o", tmp, *objs]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, LIB)
    with open(stamp_path, "w") as f:
        f.write(_stamp())
    return LIB


def load(build_if_missing: bool = True) -> ctypes.CDLL:
    """The loaded library (built first if missing or stale and allowed)."""
    global _handle
    with _lock:
        if _handle is not None:
            return _handle
        if build_if_missing:
            build()
        if not os.path.exists(LIB):
            raise RuntimeError("libjacap.so is not built (call paper_2609_08131_gb300._lib.build())")
        _handle = ctypes.CDLL(LIB)
        return _handle


EXPORTS = [
    "jacap_workspace_size",
    "jacap_schedule_info",
    "jacap_score",
    "jacap_score_timed",
    "jacap_score_static",
    "jacap_score_out",
    "jacap_score_stats",
    "jacap_stats_update",
    "jacap_compact_inplace",
    "jacap_select_compact_inplace",
    "jacap_select",
    "jacap_select_compact",
    "jacap_compact",
    "jacap_device_status",
    "jacap_selftest_wait",
    "jacap_status_string",
    "jacap_workspace_offsets",
    "jacap_host_buffer_size",
    "jacap_evict_host",
]
