"""Build libtlf.so (the CUDA library) in-tree for sm_103a with nvcc.

Each translation unit under csrc/ compiles in parallel to an object file in
_build/, then nvcc links them into _build/libtlf.so (CUDA runtime linked
statically; the driver entry points it needs are resolved at run time, so the
library loads on a machine without a GPU). A unit is recompiled only when it
or a header changed.
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
BUILD = os.path.join(PKG, "_build")
LIB = os.path.join(BUILD, "libtlf.so")
INCLUDE = os.path.join(ROOT, "include")
SOURCES = ["k_router.cu", "k_gemm.cu", "k_attn.cu", "k_misc.cu", "k_prefill.cu", "k_cond.cu", "tlf_api.cu", "tlf_ops.cu",
           "tlf_static.cu"]
HEADERS = [os.path.join(CSRC, "tlf_internal.cuh"), os.path.join(INCLUDE, "tlf.h")]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "--expt-relaxed-constexpr",
         "-I", INCLUDE, "-I", CSRC]


def nvcc() -> str:
    exe = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(exe):
        raise RuntimeError("nvcc not found")
    return exe


def _stale(obj: str, src: str) -> bool:
    if not os.path.exists(obj):
        return True
    t = os.path.getmtime(obj)
    return any(os.path.getmtime(p) > t for p in [src] + HEADERS)


def _compile(src: str, extra) -> str:
    path = os.path.join(CSRC, src)
    obj = os.path.join(BUILD, src.replace(".cu", ".o"))
    if _stale(obj, path):
        cmd = [nvcc(), *ARCH, *FLAGS, *extra, "-c", path, "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed for {src}:\n{r.stderr}")
        if r.stderr.strip() and os.environ.get("TLF_BUILD_VERBOSE"):
            sys.stderr.write(r.stderr)
    return obj


def build(extra_flags=None, force: bool = False) -> str:
    """Compile and link; returns the path of libtlf.so."""
    os.makedirs(BUILD, exist_ok=True)
    extra = list(extra_flags or [])
    if force:
        for s in SOURCES:
            o = os.path.join(BUILD, s.replace(".cu", ".o"))
            if os.path.exists(o):
                os.remove(o)
    with cf.ThreadPoolExecutor(max_workers=len(SOURCES)) as ex:
        objs = list(ex.map(lambda s: _compile(s, extra), SOURCES))
    if not os.path.exists(LIB) or any(os.path.getmtime(o) > os.path.getmtime(LIB) for o in objs):
        cmd = [nvcc(), *ARCH, "-shared", "-o", LIB, *objs]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"link failed:\n{r.stderr}")
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv))
