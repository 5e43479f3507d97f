"""Compiles the CUDA library ``libtsd.so`` in-tree with nvcc for sm_103a.

Translation units are compiled in parallel and linked into one shared
library with the CUDA runtime linked statically.  Nothing here needs a GPU.
"""
from __future__ import annotations

import concurrent.futures
import os
import shutil
import subprocess
import sys
from typing import List

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD_DIR = os.path.join(PKG, "_build")
LIB_PATH = os.path.join(PKG, "libtsd.so")
# the range-checked variant (TSD_CHECKS): every index the fused row pass
# follows is checked, a violation recorded in the decoder's status word
CHECKS_BUILD_DIR = os.path.join(PKG, "_build_checks")
CHECKS_LIB_PATH = os.path.join(PKG, "libtsd_checks.so")

SOURCES = ["tables.cpp", "arpa.cpp", "decoder.cu", "row_pass.cu", "row_fused.cu", "row_stream.cu", "joint_simt.cu", "joint_tc.cu", "joint_greedy.cu", "noalloc.cu", "row_beam.cu", "row_pruned.cu", "gemm_tc.cu", "encoder.cu", "encoder_gemm.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def nvcc() -> str:
    for c in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if c and os.path.exists(c):
            return c
    raise RuntimeError("nvcc not found")


def _flags() -> List[str]:
    return ARCH + ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC,-fvisibility=hidden", "-I", INCLUDE,
                   "-I", CSRC, "--expt-relaxed-constexpr"]


def _stale(target: str, deps: List[str]) -> bool:
    if not os.path.exists(target):
        return True
    t = os.path.getmtime(target)
    return any(os.path.getmtime(p) > t for p in deps)


def build(force: bool = False, verbose: bool = False, extra: List[str] = (), checks: bool = False) -> str:
    """Compiles libtsd.so (or, with checks, libtsd_checks.so built with
    -DTSD_CHECKS) and returns its path."""
    build_dir = CHECKS_BUILD_DIR if checks else BUILD_DIR
    lib_path = CHECKS_LIB_PATH if checks else LIB_PATH
    if checks:
        extra = list(extra) + ["-DTSD_CHECKS"]
    os.makedirs(build_dir, exist_ok=True)
    headers = [os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith((".h", ".cuh"))] + [os.path.join(INCLUDE, "tsd.h")]
    objs, jobs = [], []
    for src in SOURCES:
        path = os.path.join(CSRC, src)
        obj = os.path.join(build_dir, src + ".o")
        objs.append(obj)
        if force or _stale(obj, [path] + headers):
            x = ["-x", "cu"] if src.endswith(".cu") else []
            jobs.append([nvcc()] + _flags() + list(extra) + x + ["-c", path, "-o", obj])

    def run(cmd):
        r = subprocess.run(cmd, capture_output=True, text=True)
        if verbose or r.returncode:
            sys.stderr.write(" ".join(cmd) + "\n" + r.stdout + r.stderr)
        if r.returncode:
            raise RuntimeError(f"nvcc failed for {cmd[-3]}")
        return r

    with concurrent.futures.ThreadPoolExecutor(max_workers=max(1, min(len(jobs), os.cpu_count() or 4))) as ex:
        list(ex.map(run, jobs))
    if force or jobs or _stale(lib_path, objs):
        tmp = lib_path + f".tmp{os.getpid()}"
        run([nvcc()] + ARCH + ["-shared", "-cudart", "static", "-o", tmp] + objs)
        os.replace(tmp, lib_path)
    return lib_path


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose=True, checks="--checks" in sys.argv))
