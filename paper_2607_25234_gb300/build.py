"""Builds the C-ABI shared library ``_lib/libwhtmix.so`` with nvcc for sm_103a (no torch involved).

Usage: ``python -m paper_2607_25234_gb300.build`` (or ``__graft_entry__.build()``).
"""
from __future__ import annotations

import os
import shutil
import subprocess
import sys

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
LIBDIR = os.path.join(PKG, "_lib")
LIB = os.path.join(LIBDIR, "libwhtmix.so")
SOURCES = ["whtmix_capi.cu", "whtmix_fast_f32.cu", "whtmix_fast_bf16.cu", "whtmix_fast_sep_f32.cu", "whtmix_block.cu", "whtmix_plane.cu",
           "whtmix_fast_sep_bf16.cu", "whtmix_fast_x16.cu", "whtmix_noalloc.cu", "whtmix_proj.cu", "whtmix_block_bwd.cu"]
OBJDIR = os.path.join(LIBDIR, "obj")
# the bench's memory-only floor model of the three-phase forward (bench.py --floor); not the mixer
FLOOR_SOURCE = "bench_floor.cu"
FLOOR_LIB = os.path.join(LIBDIR, "libwhtmix_floor.so")
ARCH = "-gencode=arch=compute_103a,code=sm_103a"


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the WHTMix CUDA library cannot be built")


def _deps() -> list[str]:
    files = [os.path.join(INCLUDE, "whtmix.h")]
    for f in os.listdir(CSRC):
        if f.endswith((".cu", ".cuh", ".h")):
            files.append(os.path.join(CSRC, f))
    return files


def up_to_date() -> bool:
    for lib in (LIB, FLOOR_LIB):
        if not os.path.exists(lib):
            return False
        t = os.path.getmtime(lib)
        if not all(os.path.getmtime(f) <= t for f in _deps()):
            return False
    return True


def build(force: bool = False, verbose: bool = False) -> str:
    """Compiles every translation unit in parallel (one nvcc per file), then links the library."""
    if not force and up_to_date():
        return LIB
    os.makedirs(OBJDIR, exist_ok=True)
    common = [nvcc(), ARCH, "-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC",
              "-Xcompiler", "-fvisibility=hidden", "-I", INCLUDE, "-I", CSRC]
    if verbose:
        common += ["-Xptxas", "-v"]
    procs, objs = [], []
    for src in SOURCES + [FLOOR_SOURCE]:
        obj = os.path.join(OBJDIR, src.replace(".cu", f".{os.getpid()}.o"))
        objs.append(obj)
        procs.append((src, subprocess.Popen(common + ["-c", os.path.join(CSRC, src), "-o", obj])))
    failed = [src for src, p in procs if p.wait() != 0]
    if failed:
        raise RuntimeError(f"nvcc failed for {failed}")
    floor_obj = objs.pop()
    for lib, lib_objs in ((LIB, objs), (FLOOR_LIB, [floor_obj])):
        tmp = lib + f".tmp{os.getpid()}"
        subprocess.run([nvcc(), ARCH, "-shared", "-o", tmp] + lib_objs + ["-lcudart"], check=True)
        os.replace(tmp, lib)
    for obj in objs + [floor_obj]:
        os.remove(obj)
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose="-v" in sys.argv))
