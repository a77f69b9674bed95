"""Builds the CUDA library in-tree with nvcc for sm_103a.

    python -m paper_2609_04523_gb300.build [--force] [-v] [--debug]

Output: paper_2609_04523_gb300/libmk_attn.so (git-ignored), and with
debug=True the check build libmk_attn_debug.so (compiled with MK_DEBUG: every
kernel checks its store indices and records MK_ERR_BOUNDS instead of writing
out of range).  Each translation unit is compiled to an object in parallel,
then the objects are linked.  The library is compiled for sm_103a only; the
host code is portable C++ (x86_64 and aarch64).
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
OBJ_DIR = os.path.join(PKG, "_build")
LIB_NAME = "libmk_attn.so"
LIB_PATH = os.path.join(PKG, LIB_NAME)
DEBUG_LIB_PATH = os.path.join(PKG, "libmk_attn_debug.so")
SOURCES = [os.path.join(CSRC, f) for f in ("fmha_fwd.cu", "fmha_bwd.cu", "decode.cu", "mla_decode.cu", "status.cu")]
DEPENDS = SOURCES + [os.path.join(CSRC, "ptx.cuh"), os.path.join(CSRC, "tma_host.h"),
                     os.path.join(INCLUDE, "mk_attn.h")]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-Xcompiler",
         "-fvisibility=hidden"]


def nvcc() -> str:
    path = shutil.which("nvcc")
    if path:
        return path
    cand = "/usr/local/cuda/bin/nvcc"
    if os.path.exists(cand):
        return cand
    raise RuntimeError("nvcc not found: the CUDA 13 toolkit is required to build the library")


def _stale(out: str, deps) -> bool:
    if not os.path.exists(out):
        return True
    t = os.path.getmtime(out)
    return any(os.path.getmtime(d) > t for d in deps)


def compile_command(src: str, obj: str, extra=()) -> list[str]:
    """nvcc command compiling one translation unit to a relocatable object."""
    return [nvcc(), *ARCH, *FLAGS, "-I", INCLUDE, "-I", CSRC, *extra, "-c", src, "-o", obj]


def link_command(objs, out: str) -> list[str]:
    return [nvcc(), *ARCH, "-shared", *objs, "-o", out]


def _run(cmd):
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"nvcc failed: {' '.join(cmd)}\n{r.stdout}\n{r.stderr}")
    return r.stderr


def _build_variants(variants, verbose: bool) -> None:
    """variants: list of (output path, extra nvcc flags, object suffix)."""
    os.makedirs(OBJ_DIR, exist_ok=True)
    jobs = []
    for out, extra, tag in variants:
        for src in SOURCES:
            obj = os.path.join(OBJ_DIR, os.path.basename(src)[:-3] + tag + ".o")
            flags = list(extra) + (["-Xptxas", "-v"] if verbose else [])
            jobs.append((out, compile_command(src, obj, flags), obj))
    workers = max(1, min(len(jobs), os.cpu_count() or 1))
    with ThreadPoolExecutor(max_workers=workers) as pool:
        logs = list(pool.map(lambda j: _run(j[1]), jobs))
    if verbose:
        for log in logs:
            sys.stderr.write(log)
    for out, _extra, _tag in variants:
        objs = [obj for o, _cmd, obj in jobs if o == out]
        tmp = out + f".tmp{os.getpid()}"
        _run(link_command(objs, tmp))
        os.replace(tmp, out)


def build_library(force: bool = False, verbose: bool = False, debug: bool = False) -> str:
    """Compiles the release library (and, with debug=True, also the check
    build) if it is missing or older than its sources.  Returns the path of
    the release library, or of the check build when debug=True."""
    variants = []
    if force or _stale(LIB_PATH, DEPENDS):
        variants.append((LIB_PATH, [], ""))
    if debug and (force or _stale(DEBUG_LIB_PATH, DEPENDS)):
        variants.append((DEBUG_LIB_PATH, ["-DMK_DEBUG=1"], ".dbg"))
    if variants:
        _build_variants(variants, verbose)
    return DEBUG_LIB_PATH if debug else LIB_PATH


if __name__ == "__main__":
    print(build_library(force="--force" in sys.argv, verbose="-v" in sys.argv,
                        debug="--debug" in sys.argv))
