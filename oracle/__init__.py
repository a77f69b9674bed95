"""fp64 CPU oracle for the attention forward and backward passes and the paged
decode step (TEST INFRASTRUCTURE).

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s cpu_baseline /
reference legs may import this package.  The product path never does, and the
two share no code: this package compiles ``mk_oracle.c`` with gcc and calls
it through ctypes, with numpy arrays in and out.

What is computed is the plain definition of scaled dot-product attention with
an optional causal mask, grouped-query head sharing and packed variable-length
sequences (the reference operation that the paper's Flash Attention and GQA
Attention kernels must reproduce; Section 2.1 and Section 3.1, Table 2).  See
the header of ``mk_oracle.c`` for the formula and the layouts.

Parity status: pinned.  ``tests/test_oracle_pins.py`` checks it against closed
forms, a brute-force explicit-softmax-matrix formulation, a library routine
(PyTorch's fp64 scaled_dot_product_attention on CPU), and invariants;
``tests/test_oracle_mutants.py`` shows that planted mistakes fail those pins.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "mk_oracle.c")
_BUILD_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD_DIR, "libmk_oracle.so")

_lock = threading.Lock()
_lib = None


def compile_oracle(src: str = _SRC, out: str = _LIB_PATH) -> str:
    """Compiles an oracle C source into a shared library; returns its path."""
    os.makedirs(os.path.dirname(out), exist_ok=True)
    tmp = out + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-pthread",
           "-fno-fast-math", "-ffp-contract=off", src, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True, capture_output=True, text=True)
    os.replace(tmp, out)
    return out


def build(force: bool = False) -> str:
    """Builds the oracle library if it is missing or older than its source."""
    with _lock:
        if force or not os.path.exists(_LIB_PATH) or \
                os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
            compile_oracle()
    return _LIB_PATH


def _bind(lib: ctypes.CDLL) -> ctypes.CDLL:
    p = ctypes.c_void_p
    i = ctypes.c_int
    lib.mk_oracle_attn_fwd_f64.argtypes = [p, p, p, p, p, i, i, i, i, i, i,
                                           ctypes.c_double, p, i]
    lib.mk_oracle_attn_fwd_f64.restype = i
    lib.mk_oracle_attn_rows_f64.argtypes = [p, p, p, i, i, i, i, i, i, ctypes.c_double,
                                            p, p, ctypes.c_int64, p, p, i]
    lib.mk_oracle_attn_rows_f64.restype = i
    lib.mk_oracle_decode_paged_f64.argtypes = [p, p, p, p, p, p, p, i, i, i, i, i, i, i,
                                               ctypes.c_double, i]
    lib.mk_oracle_decode_paged_f64.restype = i
    lib.mk_oracle_attn_bwd_f64.argtypes = [p, p, p, p, p, p, p, i, i, i, i, i, i,
                                           ctypes.c_double, p, i]
    lib.mk_oracle_attn_bwd_f64.restype = i
    lib.mk_oracle_attn_bwd_dq_rows_f64.argtypes = [p, p, p, p, i, i, i, i, i, i, ctypes.c_double,
                                                   p, p, ctypes.c_int64, p, i]
    lib.mk_oracle_attn_bwd_dq_rows_f64.restype = i
    lib.mk_oracle_attn_bwd_dkv_ranges_f64.argtypes = [p, p, p, p, i, i, i, i, i, i,
                                                      ctypes.c_double, p, p, ctypes.c_int64, p,
                                                      p, i]
    lib.mk_oracle_attn_bwd_dkv_ranges_f64.restype = i
    lib.mk_oracle_mla_decode_f64.argtypes = [p, p, p, p, p, p, i, i, i, i, i, i, i,
                                             ctypes.c_double, i]
    lib.mk_oracle_mla_decode_f64.restype = i
    return lib


def load(path: str | None = None) -> ctypes.CDLL:
    """Loads the default oracle library (building it on first use), or `path`."""
    global _lib
    if path is not None:
        return _bind(ctypes.CDLL(path))
    if _lib is None:
        build()
        _lib = _bind(ctypes.CDLL(_LIB_PATH))
    return _lib


def default_threads() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:  # pragma: no cover
        return os.cpu_count() or 1


def _bits(x) -> np.ndarray:
    """bf16 data as a contiguous uint16 bit-pattern array.

    Accepts a numpy uint16 array or a torch bfloat16 CPU tensor."""
    if isinstance(x, np.ndarray):
        if x.dtype != np.uint16:
            raise TypeError("oracle inputs are bf16 bit patterns (uint16)")
        return np.ascontiguousarray(x)
    import torch  # only for the tensor -> bits view
    if x.dtype != torch.bfloat16:
        raise TypeError("oracle inputs are bf16")
    return np.ascontiguousarray(x.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16))


def _shape(q, k, cu_seqlens):
    if cu_seqlens is None:
        B, S, Hq, D = q.shape
        Hkv = k.shape[2]
        return B, Hq, Hkv, S, D
    T, Hq, D = q.shape
    Hkv = k.shape[1]
    B = len(cu_seqlens) - 1
    return B, Hq, Hkv, T, D


def _cu(cu_seqlens):
    if cu_seqlens is None:
        return None
    return np.ascontiguousarray(np.asarray(cu_seqlens, dtype=np.int32))


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def attn_fwd(q, k, v, causal: bool, scale: float, cu_seqlens=None,
             n_threads: int | None = None, lib: ctypes.CDLL | None = None):
    """Full forward pass in fp64.

    q: [B,S,Hq,D] (or [T,Hq,D] with cu_seqlens), k/v: [B,S,Hkv,D] (or
    [T,Hkv,D]); bf16 tensors or uint16 bit arrays.  Returns (o, lse) as fp64
    numpy arrays, o shaped like q, lse [B,Hq,S] (or [Hq,T])."""
    qb, kb, vb = _bits(q), _bits(k), _bits(v)
    cu = _cu(cu_seqlens)
    B, Hq, Hkv, S, D = _shape(qb, kb, cu)
    o = np.zeros(qb.shape, dtype=np.float64)
    lse = np.zeros((Hq, S) if cu is not None else (B, Hq, S), dtype=np.float64)
    lib = lib or load()
    st = lib.mk_oracle_attn_fwd_f64(_ptr(qb), _ptr(kb), _ptr(vb), _ptr(o), _ptr(lse),
                                    B, Hq, Hkv, S, D, int(bool(causal)), float(scale),
                                    _ptr(cu), int(n_threads or default_threads()))
    if st != 0:
        raise ValueError(f"oracle rejected the problem (status {st})")
    return o, lse


def attn_rows(q, k, v, causal: bool, scale: float, rows, cu_seqlens=None,
              n_threads: int | None = None, lib: ctypes.CDLL | None = None):
    """The definition on selected rows only.

    rows: int array [n, 3] of (sequence b, query head h, position i within the
    sequence).  Returns (o_rows [n, D], lse_rows [n]) in fp64."""
    qb, kb, vb = _bits(q), _bits(k), _bits(v)
    cu = _cu(cu_seqlens)
    B, Hq, Hkv, S, D = _shape(qb, kb, cu)
    r = np.ascontiguousarray(np.asarray(rows, dtype=np.int64).reshape(-1, 3))
    n = r.shape[0]
    o = np.zeros((n, D), dtype=np.float64)
    lse = np.zeros((n,), dtype=np.float64)
    lib = lib or load()
    st = lib.mk_oracle_attn_rows_f64(_ptr(qb), _ptr(kb), _ptr(vb), B, Hq, Hkv, S, D,
                                     int(bool(causal)), float(scale), _ptr(cu), _ptr(r),
                                     n, _ptr(o), _ptr(lse), int(n_threads or default_threads()))
    if st != 0:
        raise ValueError(f"oracle rejected the rows (status {st})")
    return o, lse


def decode_paged(q, k_cache, v_cache, page_table, seq_lens, scale: float,
                 n_threads: int | None = None, lib: ctypes.CDLL | None = None):
    """One decode step against a paged K/V cache, in fp64.

    q: [B,Hq,D]; k_cache/v_cache: [num_pages, page_size, Hkv, D] (bf16 tensors
    or uint16 bit arrays); page_table: int32 [B, max_pages]; seq_lens: int32
    [B].  Returns (o [B,Hq,D], lse [B,Hq]) as fp64 numpy arrays."""
    qb, kb, vb = _bits(q), _bits(k_cache), _bits(v_cache)
    pt = np.ascontiguousarray(np.asarray(page_table, dtype=np.int32))
    sl = np.ascontiguousarray(np.asarray(seq_lens, dtype=np.int32))
    B, Hq, D = qb.shape
    num_pages, page_size, Hkv, _ = kb.shape
    o = np.zeros((B, Hq, D), dtype=np.float64)
    lse = np.zeros((B, Hq), dtype=np.float64)
    lib = lib or load()
    st = lib.mk_oracle_decode_paged_f64(_ptr(qb), _ptr(kb), _ptr(vb), _ptr(pt), _ptr(sl),
                                        _ptr(o), _ptr(lse), B, Hq, Hkv, D, page_size,
                                        pt.shape[1], num_pages, float(scale),
                                        int(n_threads or default_threads()))
    if st != 0:
        raise ValueError(f"oracle rejected the decode problem (status {st})")
    return o, lse


def attn_bwd(q, k, v, do, causal: bool, scale: float, cu_seqlens=None,
             n_threads: int | None = None, lib: ctypes.CDLL | None = None):
    """Full backward pass in fp64: the gradients of the forward definition
    with respect to q, k and v for the output gradient `do` (layout of q).

    Returns (dq, dk, dv) as fp64 numpy arrays shaped like q, k, v."""
    qb, kb, vb, dob = _bits(q), _bits(k), _bits(v), _bits(do)
    if dob.shape != qb.shape:
        raise ValueError("do must have the shape of q")
    cu = _cu(cu_seqlens)
    B, Hq, Hkv, S, D = _shape(qb, kb, cu)
    dq = np.zeros(qb.shape, dtype=np.float64)
    dk = np.zeros(kb.shape, dtype=np.float64)
    dv = np.zeros(vb.shape, dtype=np.float64)
    lib = lib or load()
    st = lib.mk_oracle_attn_bwd_f64(_ptr(qb), _ptr(kb), _ptr(vb), _ptr(dob), _ptr(dq), _ptr(dk),
                                    _ptr(dv), B, Hq, Hkv, S, D, int(bool(causal)), float(scale),
                                    _ptr(cu), int(n_threads or default_threads()))
    if st != 0:
        raise ValueError(f"oracle rejected the problem (status {st})")
    return dq, dk, dv


def attn_bwd_dq_rows(q, k, v, do, causal: bool, scale: float, rows, cu_seqlens=None,
                     n_threads: int | None = None, lib: ctypes.CDLL | None = None):
    """dq of the backward pass on selected rows (b, h, i) only: [n, D] fp64."""
    qb, kb, vb, dob = _bits(q), _bits(k), _bits(v), _bits(do)
    cu = _cu(cu_seqlens)
    B, Hq, Hkv, S, D = _shape(qb, kb, cu)
    r = np.ascontiguousarray(np.asarray(rows, dtype=np.int64).reshape(-1, 3))
    out = np.zeros((r.shape[0], D), dtype=np.float64)
    lib = lib or load()
    st = lib.mk_oracle_attn_bwd_dq_rows_f64(_ptr(qb), _ptr(kb), _ptr(vb), _ptr(dob), B, Hq, Hkv,
                                            S, D, int(bool(causal)), float(scale), _ptr(cu),
                                            _ptr(r), r.shape[0], _ptr(out),
                                            int(n_threads or default_threads()))
    if st != 0:
        raise ValueError(f"oracle rejected the rows (status {st})")
    return out


def attn_bwd_dkv_ranges(q, k, v, do, causal: bool, scale: float, ranges, cu_seqlens=None,
                        n_threads: int | None = None, lib: ctypes.CDLL | None = None):
    """dk and dv of the backward pass for key ranges (b, g, j0, j1) of a
    sequence and key/value head (positions within the sequence).  Returns
    (dk_rows, dv_rows), each [sum of (j1 - j0), D] fp64, ranges in order."""
    qb, kb, vb, dob = _bits(q), _bits(k), _bits(v), _bits(do)
    cu = _cu(cu_seqlens)
    B, Hq, Hkv, S, D = _shape(qb, kb, cu)
    r = np.ascontiguousarray(np.asarray(ranges, dtype=np.int64).reshape(-1, 4))
    n = int(np.sum(r[:, 3] - r[:, 2])) if r.size else 0
    dk = np.zeros((max(n, 0), D), dtype=np.float64)
    dv = np.zeros((max(n, 0), D), dtype=np.float64)
    lib = lib or load()
    st = lib.mk_oracle_attn_bwd_dkv_ranges_f64(_ptr(qb), _ptr(kb), _ptr(vb), _ptr(dob), B, Hq,
                                               Hkv, S, D, int(bool(causal)), float(scale),
                                               _ptr(cu), _ptr(r), r.shape[0], _ptr(dk), _ptr(dv),
                                               int(n_threads or default_threads()))
    if st != 0:
        raise ValueError(f"oracle rejected the ranges (status {st})")
    return dk, dv


def mla_decode(q, cache, page_table, seq_lens, scale: float, dv: int,
               n_threads: int | None = None, lib: ctypes.CDLL | None = None):
    """One latent (MLA) decode step in fp64: q [B,Hq,Dqk], cache
    [num_pages, page_size, Dqk] (keys in full, values = the first dv
    components), page_table int32 [B, max_pages], seq_lens int32 [B].
    Returns (o [B,Hq,dv], lse [B,Hq]) as fp64 numpy arrays."""
    qb, cb = _bits(q), _bits(cache)
    pt = np.ascontiguousarray(np.asarray(page_table, dtype=np.int32))
    sl = np.ascontiguousarray(np.asarray(seq_lens, dtype=np.int32))
    B, Hq, Dqk = qb.shape
    num_pages, page_size, Dc = cb.shape
    if Dc != Dqk:
        raise ValueError("cache rows must have the query's dimension")
    o = np.zeros((B, Hq, dv), dtype=np.float64)
    lse = np.zeros((B, Hq), dtype=np.float64)
    lib = lib or load()
    st = lib.mk_oracle_mla_decode_f64(_ptr(qb), _ptr(cb), _ptr(pt), _ptr(sl), _ptr(o), _ptr(lse),
                                      B, Hq, Dqk, dv, page_size, pt.shape[1], num_pages,
                                      float(scale), int(n_threads or default_threads()))
    if st != 0:
        raise ValueError(f"oracle rejected the MLA decode problem (status {st})")
    return o, lse
