"""In-tree build of the CUDA library ``libwam_gb300.so`` for sm_103a.

Each translation unit is compiled by nvcc in parallel into ``_build/`` and linked into a shared
library next to this file.  Rebuilds only what changed (source or header newer than its object).
Run ``python -m paper_2609_34608_gb300._build`` or call ``build()``.
"""
from __future__ import annotations

import concurrent.futures as cf
import glob
import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD_DIR = os.path.join(HERE, "_build")
LIB_PATH = os.path.join(HERE, "libwam_gb300.so")

SOURCES = ["wam_api.cu", "ops.cu", "gemm_tc.cu", "gemm_simt.cu", "attention.cu", "elementwise.cu",
           "tr_static.cu", "attention_tc.cu", "dit_chain.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ARCH + ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-I", INCLUDE,
                "--expt-relaxed-constexpr"]


def _nvcc() -> str:
    for cand in (shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libwam_gb300.so")


def _headers() -> list[str]:
    return glob.glob(os.path.join(CSRC, "*.cuh")) + glob.glob(os.path.join(INCLUDE, "*.h"))


def _stale(src: str, obj: str, newest_header: float) -> bool:
    if not os.path.exists(obj):
        return True
    t = os.path.getmtime(obj)
    return os.path.getmtime(src) > t or newest_header > t


def _run(cmd: list[str]) -> None:
    res = subprocess.run(cmd, capture_output=True, text=True)
    if res.returncode != 0:
        raise RuntimeError("build step failed:\n" + " ".join(cmd) + "\n" + res.stdout + res.stderr)


def build(force: bool = False, verbose: bool = False, jobs: int | None = None) -> str:
    nvcc = _nvcc()
    os.makedirs(BUILD_DIR, exist_ok=True)
    newest = max([os.path.getmtime(h) for h in _headers()] + [0.0])
    objs, todo = [], []
    for name in SOURCES:
        src = os.path.join(CSRC, name)
        obj = os.path.join(BUILD_DIR, name.replace(".cu", ".o"))
        objs.append(obj)
        if force or _stale(src, obj, newest):
            todo.append([nvcc, *FLAGS, "-c", src, "-o", obj])
    with cf.ThreadPoolExecutor(max_workers=jobs or min(len(SOURCES), os.cpu_count() or 4)) as ex:
        for cmd, fut in [(c, ex.submit(_run, c)) for c in todo]:
            fut.result()
            if verbose:
                print("compiled", os.path.basename(cmd[-3]), file=sys.stderr)
    lib_time = os.path.getmtime(LIB_PATH) if os.path.exists(LIB_PATH) else -1.0
    if force or todo or any(os.path.getmtime(o) > lib_time for o in objs):
        tmp = LIB_PATH + ".tmp"
        _run([nvcc, *ARCH, "-shared", "-o", tmp, *objs, "-lpthread", "-ldl", "-lrt"])
        os.replace(tmp, LIB_PATH)
    return LIB_PATH


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose=True))
