"""Compile libkvlink.so (sm_103a) in-tree with nvcc.

Every translation unit is compiled in parallel into _build/, then linked into
paper_2502_16002_gb300/libkvlink.so.  The library links the CUDA runtime
statically and resolves driver entry points at run time, so it loads (and its
host-only calls work) on a machine without a GPU driver.

build(debug=True) makes libkvlink_debug.so from the same sources with
KVLINK_DEBUG_CHECKS: its kernels check every index table entry they use against
the plan's bounds and record a code in the device status word instead of
touching memory through a bad entry (select it with KVLINK_LIBRARY).
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
INCLUDE = os.path.join(ROOT, "include")
BUILD = os.path.join(ROOT, "_build")
LIB = os.path.join(PKG, "libkvlink.so")
LIB_DEBUG = os.path.join(PKG, "libkvlink_debug.so")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
COMMON = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", f"-I{INCLUDE}", f"-I{CSRC}"]

SOURCES = [
    "kvlink_plan.cpp",
    "kvlink_api.cu",
    "kvlink_reencode.cu",
    "kvlink_attention_simt.cu",
    "kvlink_attention_tc.cu",
    "kvlink_attention_fused.cu",
    "kvlink_noalloc.cu",
]


def nvcc() -> str:
    for c in (os.environ.get("NVCC"), "/usr/local/cuda/bin/nvcc", shutil.which("nvcc")):
        if c and os.path.exists(c):
            return c
    raise RuntimeError("nvcc not found")


def _deps_mtime() -> float:
    files = [os.path.join(CSRC, f) for f in os.listdir(CSRC)] + [os.path.join(INCLUDE, "kvlink.h")]
    return max(os.path.getmtime(f) for f in files) if files else 0.0


def _compile(src: str, extra, objdir: str = BUILD) -> str:
    obj = os.path.join(objdir, os.path.basename(src) + ".o")
    cmd = [nvcc(), *ARCH, *COMMON, *extra, "-c", os.path.join(CSRC, src), "-o", obj]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"nvcc failed for {src}:\n{' '.join(cmd)}\n{r.stdout}\n{r.stderr}")
    return obj


def build(force: bool = False, verbose: bool = False, extra=(), debug: bool = False) -> str:
    """Build libkvlink.so (libkvlink_debug.so with debug=True) unless it is newer than
    every source.  Returns its path."""
    lib = LIB_DEBUG if debug else LIB
    if not force and os.path.exists(lib) and os.path.getmtime(lib) >= _deps_mtime():
        return lib
    objdir = os.path.join(BUILD, "debug") if debug else BUILD
    flags = list(extra) + (["-DKVLINK_DEBUG_CHECKS"] if debug else [])
    os.makedirs(objdir, exist_ok=True)
    with ThreadPoolExecutor(max_workers=max(1, min(len(SOURCES), os.cpu_count() or 1))) as ex:
        objs = list(ex.map(lambda s: _compile(s, flags, objdir), SOURCES))
    tmp = lib + ".tmp"
    cmd = [nvcc(), *ARCH, "-shared", "-cudart", "static", "-o", tmp, *objs]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{' '.join(cmd)}\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, lib)
    if verbose:
        print(f"built {lib}", file=sys.stderr)
    return lib


if __name__ == "__main__":
    build(force="--force" in sys.argv, verbose=True, debug="--debug" in sys.argv)
