"""Builds ``libstatekv.so`` (the C-ABI library) in-tree with nvcc for sm_103a.

Each translation unit compiles in parallel into ``_build/``; the objects link
into ``paper_2605_31598_gb300/libstatekv.so`` with the CUDA runtime linked
statically and no other library, so it loads on a machine without a GPU
driver (it needs one only when a call reaches the device).
"""
from __future__ import annotations

import concurrent.futures as cf
import os
import shutil
import subprocess
import sys

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
OUT = os.path.join(PKG, "_build")
LIB = os.path.join(PKG, "libstatekv.so")
# the debug build: bounds checks that record a fault in the status word, and
# guard bands around the arena's regions (STATEKV_DEBUG_CHECKS=1)
OUT_DEBUG = os.path.join(PKG, "_build_debug")
LIB_DEBUG = os.path.join(PKG, "libstatekv_debug.so")
SOURCES = ["attn_kernel.cu", "select_kernel.cu", "diag_kernel.cu", "block_kernel.cu", "decode_kernel.cu",
           "gemm_kernel.cu", "statekv_api.cu", "noalloc.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-Xcompiler", "-O2",
         "--expt-relaxed-constexpr", "-I", os.path.join(ROOT, "include")]


def _nvcc() -> str:
    for cand in (shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is needed to build libstatekv.so")


def _newer(target: str, deps) -> bool:
    if not os.path.exists(target):
        return False
    t = os.path.getmtime(target)
    return all(os.path.getmtime(d) <= t for d in deps)


def _headers():
    hs = [os.path.join(ROOT, "include", "statekv.h")]
    hs += [os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith((".cuh", ".h"))]
    return hs


def build(force: bool = False, verbose: bool = False, extra_flags=(), debug: bool = False) -> str:
    """Compile and link; returns the library path.  Rebuilds only what changed.
    ``debug`` builds ``libstatekv_debug.so`` with STATEKV_DEBUG_CHECKS=1."""
    nvcc = _nvcc()
    out_dir, lib_path = (OUT_DEBUG, LIB_DEBUG) if debug else (OUT, LIB)
    if debug:
        extra_flags = tuple(extra_flags) + ("-DSTATEKV_DEBUG_CHECKS=1",)
    os.makedirs(out_dir, exist_ok=True)
    headers = _headers()
    objs, jobs = [], []
    for src in SOURCES:
        spath = os.path.join(CSRC, src)
        obj = os.path.join(out_dir, src.replace(".cu", ".o"))
        objs.append(obj)
        if force or not _newer(obj, [spath] + headers):
            jobs.append([nvcc, *ARCH, *FLAGS, *extra_flags, "-c", spath, "-o", obj])

    def run(cmd):
        r = subprocess.run(cmd, capture_output=True, text=True)
        if verbose or r.returncode != 0:
            sys.stderr.write(r.stdout + r.stderr)
        if r.returncode != 0:
            raise RuntimeError("nvcc failed: " + " ".join(cmd))

    with cf.ThreadPoolExecutor(max_workers=len(SOURCES)) as ex:
        list(ex.map(run, jobs))
    if force or jobs or not _newer(lib_path, objs):
        tmp = lib_path + ".tmp.%d" % os.getpid()
        run([nvcc, *ARCH, "-shared", "-o", tmp, *objs])
        os.replace(tmp, lib_path)
    return lib_path


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose="-v" in sys.argv))
