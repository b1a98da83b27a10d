"""Builds libdomino.so in-tree with nvcc for sm_103a (GB300).

Three translation units (host.cpp: C ABI and loaders; kernels.cu and trie.cu:
kernels) are compiled in parallel and linked into paper_2403_06988_gb300/libdomino.so.
Objects go to paper_2403_06988_gb300/_build/.

build(debug=True) makes libdomino_debug.so instead (objects in _build_debug/),
compiled with -DDOMINO_DEBUG: every transition-table lookup checks its state,
class and entry against the table's bounds and reports a violation in the
device error word (DOMINO_DEVERR_INTERNAL) instead of reading outside it.  The
binding loads it when DOMINO_DEBUG_LIB=1 is set in the environment.
"""
from __future__ import annotations

import concurrent.futures
import os
import shutil
import subprocess

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD = os.path.join(PKG, "_build")
LIB = os.path.join(PKG, "libdomino.so")
LIB_DEBUG = os.path.join(PKG, "libdomino_debug.so")
SOURCES = ["host.cpp", "kernels.cu", "trie.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def nvcc() -> str:
    exe = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(exe):
        raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libdomino.so")
    return exe


def _inputs():
    files = [os.path.join(CSRC, f) for f in SOURCES]
    files += [os.path.join(CSRC, "domino_internal.h"), os.path.join(CSRC, "walk_common.cuh"),
              os.path.join(INCLUDE, "domino.h")]
    return files


def up_to_date(lib: str = LIB) -> bool:
    if not os.path.exists(lib):
        return False
    t = os.path.getmtime(lib)
    return all(os.path.getmtime(f) <= t for f in _inputs())


def build(force: bool = False, verbose: bool = False, extra_flags=(), debug: bool = False) -> str:
    lib = LIB_DEBUG if debug else LIB
    bdir = BUILD + "_debug" if debug else BUILD
    if not force and up_to_date(lib):
        return lib
    os.makedirs(bdir, exist_ok=True)
    exe = nvcc()
    common = ["-O3", "-std=c++17", *ARCH, "-lineinfo", "-Xcompiler", "-fPIC", "-I", INCLUDE, "-I", CSRC,
              *(["-DDOMINO_DEBUG"] if debug else []), *extra_flags]
    if verbose:
        common += ["-Xptxas", "-v"]

    def compile_one(src):
        obj = os.path.join(bdir, os.path.splitext(src)[0] + ".o")
        cmd = [exe, *common, "-c", os.path.join(CSRC, src), "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed for {src}:\n{r.stdout}\n{r.stderr}")
        return obj, r.stderr

    with concurrent.futures.ThreadPoolExecutor(len(SOURCES)) as ex:
        results = list(ex.map(compile_one, SOURCES))
    if verbose:
        for _, log in results:
            print(log)
    tmp = lib + f".tmp{os.getpid()}"
    cmd = [exe, "-shared", *ARCH, "-o", tmp, *[o for o, _ in results]]   # cudart linked statically
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, lib)
    return lib


if __name__ == "__main__":
    import sys
    print(build(force="--force" in sys.argv, verbose="-v" in sys.argv))
