"""Builds the CUDA library in-tree with nvcc for sm_103a.

    python -m paper_2609_04523_gb300.build      # or build_library()

Output: paper_2609_04523_gb300/libmk_attn.so (git-ignored).  The library is
compiled for sm_103a only; the host code is portable C++ (x86_64 and aarch64).
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
LIB_NAME = "libmk_attn.so"
LIB_PATH = os.path.join(PKG, LIB_NAME)
SOURCES = [os.path.join(CSRC, f) for f in ("fmha_fwd.cu", "fmha_bwd.cu", "decode.cu", "mla_decode.cu", "status.cu")]
DEPENDS = SOURCES + [os.path.join(CSRC, "ptx.cuh"), os.path.join(CSRC, "tma_host.h"),
                     os.path.join(INCLUDE, "mk_attn.h")]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


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


def compile_command(out: str, extra=()) -> list[str]:
    return [nvcc(), *ARCH, "-O3", "-lineinfo", "-std=c++17", "-shared",
            "-Xcompiler", "-fPIC", "-Xcompiler", "-fvisibility=hidden",
            "-I", INCLUDE, "-I", CSRC, *extra, *SOURCES, "-o", out]


def build_library(force: bool = False, verbose: bool = False) -> str:
    """Compiles the library if it is missing or older than its sources."""
    if not force and not _stale(LIB_PATH, DEPENDS):
        return LIB_PATH
    tmp = LIB_PATH + f".tmp{os.getpid()}"
    extra = ["-Xptxas", "-v"] if verbose else []
    r = subprocess.run(compile_command(tmp, extra), capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"nvcc failed:\n{r.stdout}\n{r.stderr}")
    if verbose:
        sys.stderr.write(r.stderr)
    os.replace(tmp, LIB_PATH)
    return LIB_PATH


if __name__ == "__main__":
    print(build_library(force="--force" in sys.argv, verbose="-v" in sys.argv))
