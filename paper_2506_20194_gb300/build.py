"""Builds libduo.so in-tree with nvcc for sm_103a (no cmake, no torch).

Usage: ``python -m paper_2506_20194_gb300.build`` or ``build_library()``.
The translation units compile in parallel; the result is
``paper_2506_20194_gb300/libduo.so`` (git-ignored).
"""
from __future__ import annotations

import os
import shutil
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
OUT = os.path.join(PKG, "libduo.so")
BUILD_DIR = os.path.join(PKG, "_build")
SOURCES = ("kernels.cu", "api.cu", "noalloc.cu", "calib.cu", "copy.cu", "tcgemm.cu")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def nvcc_path() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found")


def _compile(src: str, extra: list[str]) -> str:
    obj = os.path.join(BUILD_DIR, os.path.splitext(src)[0] + ".o")
    # Warnings are errors: a host-only call from __host__ __device__ code, for
    # one, is only a warning but leaves the device code undefined.
    cmd = [nvcc_path(), *ARCH, "-O3", "-lineinfo", "-std=c++17", "-Werror", "all-warnings",
           "-Xcompiler", "-fPIC", "-I", os.path.join(ROOT, "include"), "-c", os.path.join(CSRC, src),
           "-o", obj, *extra]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"nvcc failed for {src}:\n{r.stdout}\n{r.stderr}")
    if extra:
        sys.stderr.write(r.stdout + r.stderr)
    return obj


def build_library(verbose_ptxas: bool = False, force: bool = False) -> str:
    srcs = [os.path.join(CSRC, s) for s in SOURCES]
    hdrs = [os.path.join(CSRC, h) for h in os.listdir(CSRC) if h.endswith((".cuh", ".h"))]
    hdrs.append(os.path.join(ROOT, "include", "duo.h"))
    if (not force and os.path.exists(OUT)
            and os.path.getmtime(OUT) > max(os.path.getmtime(p) for p in srcs + hdrs + [__file__])):
        return OUT
    os.makedirs(BUILD_DIR, exist_ok=True)
    extra = ["-Xptxas", "-v"] if verbose_ptxas else []
    with ThreadPoolExecutor(max_workers=len(SOURCES)) as ex:
        objs = list(ex.map(lambda s: _compile(s, extra), SOURCES))
    tmp = OUT + ".tmp"
    cmd = [nvcc_path(), *ARCH, "-shared", "-o", tmp, *objs, "-lcudart_static", "-lrt", "-ldl", "-lpthread"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, OUT)
    return OUT


if __name__ == "__main__":
    print(build_library(verbose_ptxas="-v" in sys.argv, force="-f" in sys.argv))
