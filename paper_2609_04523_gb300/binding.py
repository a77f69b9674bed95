"""Thin ctypes binding of the C ABI in include/mk_attn.h.

Argument marshalling only: every step of the attention forward pass runs in
the CUDA library.  There is no CPU or PyTorch fallback; if the library is
missing or cannot be loaded, every call raises.
"""
from __future__ import annotations

import ctypes
import os
import threading

PKG = os.path.dirname(os.path.abspath(__file__))
RELEASE_LIB_PATH = os.path.join(PKG, "libmk_attn.so")
CHECK_LIB_PATH = os.path.join(PKG, "libmk_attn_debug.so")
# MK_ATTN_CHECK_BUILD=1 in the environment loads the check build (compiled
# with MK_DEBUG: store indices checked in every kernel) instead of the release
# build.  Build it with paper_2609_04523_gb300.build.build_library(debug=True).
LIB_PATH = (CHECK_LIB_PATH if os.environ.get("MK_ATTN_CHECK_BUILD", "0") not in ("", "0")
            else RELEASE_LIB_PATH)

MK_OK = 0
MK_ERR_INVALID_ARG = -1
MK_ERR_UNSUPPORTED = -2
MK_ERR_ALIGNMENT = -3
MK_ERR_CUDA = -4
MK_ERR_TIMEOUT = -5
MK_ERR_SCRATCH_LIMIT = -6
MK_ERR_BOUNDS = -7

# Backward-pass stages (MK_BWD_* in include/mk_attn.h).
BWD_DELTA, BWD_DKDV, BWD_DQ, BWD_ALL = 1, 2, 4, 7

# Latent (MLA) decode row widths (MK_MLA_DQK, MK_MLA_DV).
MLA_DQK, MLA_DV = 576, 512

# Unit schedules (MK_SCHED_*).
SCHED_SNAKE, SCHED_ROUND_ROBIN, SCHED_BLOCKED, SCHED_DYNAMIC = 0, 1, 2, 3


class MkAttnTuning(ctypes.Structure):
    """mk_attn_tuning: launch parameters that change speed, not results."""
    _fields_ = [("ctas", ctypes.c_int), ("schedule", ctypes.c_int),
                ("rescale_log2", ctypes.c_float), ("split_ctas_per_sm", ctypes.c_int),
                ("split_min_pages", ctypes.c_int), ("mla_split_ctas_per_sm", ctypes.c_int)]

    def as_dict(self) -> dict:
        return {name: getattr(self, name) for name, _ in self._fields_}


DEFAULT_TUNING = dict(ctas=0, schedule=SCHED_SNAKE, rescale_log2=8.0, split_ctas_per_sm=24,
                      split_min_pages=2, mla_split_ctas_per_sm=3)

# Bytes of the library's own decode scratch array (MK_ATTN_DECODE_STATIC_SCRATCH_BYTES).
DECODE_STATIC_SCRATCH_BYTES = 16 * 1024 * 1024

# Symbols declared in include/mk_attn.h.
EXPORTED = ("mk_attn_fwd", "mk_attn_fwd_stall_test", "mk_attn_bwd_workspace_bytes", "mk_attn_bwd",
            "mk_attn_bwd_stages",
            "mk_attn_decode_workspace_bytes",
            "mk_attn_decode_paged", "mk_attn_decode_paged_noalloc", "mk_attn_error_string",
            "mk_attn_check_status", "mk_attn_version", "mk_attn_set_tuning",
            "mk_attn_get_tuning", "mk_attn_mla_decode_workspace_bytes", "mk_attn_mla_decode_paged")

_lock = threading.Lock()
_lib = None


class MkAttnError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"{msg} (status {status})")
        self.status = status


def library_path() -> str:
    return LIB_PATH


def load_library() -> ctypes.CDLL:
    """Loads the in-tree CUDA library; raises if it has not been built."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIB_PATH):
                raise MkAttnError(MK_ERR_CUDA,
                                  f"CUDA library not built: {LIB_PATH} is missing "
                                  "(run paper_2609_04523_gb300.build.build_library())")
            lib = ctypes.CDLL(LIB_PATH)
            vp, i = ctypes.c_void_p, ctypes.c_int
            lib.mk_attn_fwd.argtypes = [vp, vp, vp, vp, vp, i, i, i, i, i, i, ctypes.c_float,
                                        vp, vp]
            lib.mk_attn_fwd.restype = i
            lib.mk_attn_fwd_stall_test.argtypes = lib.mk_attn_fwd.argtypes
            lib.mk_attn_fwd_stall_test.restype = i
            i64 = ctypes.c_int64
            lib.mk_attn_bwd_workspace_bytes.argtypes = [i, i, i, i]
            lib.mk_attn_bwd_workspace_bytes.restype = i64
            lib.mk_attn_bwd.argtypes = [vp, vp, vp, vp, vp, vp, vp, vp, vp, i, i, i, i, i, i,
                                        ctypes.c_float, vp, vp, i64, vp]
            lib.mk_attn_bwd.restype = i
            lib.mk_attn_bwd_stages.argtypes = lib.mk_attn_bwd.argtypes[:-1] + [i, vp]
            lib.mk_attn_bwd_stages.restype = i
            lib.mk_attn_decode_workspace_bytes.argtypes = [i, i, i, i, i, i]
            lib.mk_attn_decode_workspace_bytes.restype = i64
            lib.mk_attn_decode_paged.argtypes = [vp, vp, vp, vp, vp, vp, vp, i, i, i, i, i, i, i,
                                                 ctypes.c_float, vp, i64, vp]
            lib.mk_attn_decode_paged.restype = i
            lib.mk_attn_decode_paged_noalloc.argtypes = [vp, vp, vp, vp, vp, vp, vp, i, i, i, i, i,
                                                         i, i, ctypes.c_float, vp]
            lib.mk_attn_decode_paged_noalloc.restype = i
            lib.mk_attn_error_string.argtypes = [i]
            lib.mk_attn_error_string.restype = ctypes.c_char_p
            lib.mk_attn_check_status.argtypes = [vp]
            lib.mk_attn_check_status.restype = i
            lib.mk_attn_version.argtypes = []
            lib.mk_attn_version.restype = i
            lib.mk_attn_mla_decode_workspace_bytes.argtypes = [i, i, i, i]
            lib.mk_attn_mla_decode_workspace_bytes.restype = i64
            lib.mk_attn_mla_decode_paged.argtypes = [vp, vp, vp, vp, vp, vp, i, i, i, i, i,
                                                     ctypes.c_float, vp, i64, vp]
            lib.mk_attn_mla_decode_paged.restype = i
            lib.mk_attn_set_tuning.argtypes = [ctypes.POINTER(MkAttnTuning)]
            lib.mk_attn_set_tuning.restype = i
            lib.mk_attn_get_tuning.argtypes = [ctypes.POINTER(MkAttnTuning)]
            lib.mk_attn_get_tuning.restype = i
            _lib = lib
    return _lib


def mk_attn_fwd(q: int, k: int, v: int, o: int, lse: int, B: int, Hq: int, Hkv: int, S: int,
                D: int, causal: int, scale: float, cu_seqlens: int | None, stream: int | None) -> int:
    """Raw C-ABI call: integer device pointers in, status code out."""
    return load_library().mk_attn_fwd(q, k, v, o, lse, B, Hq, Hkv, S, D, int(causal),
                                      float(scale), cu_seqlens, stream)


def mk_attn_fwd_stall_test(q: int, k: int, v: int, o: int, lse: int, B: int, Hq: int, Hkv: int,
                           S: int, D: int, causal: int, scale: float, cu_seqlens: int | None,
                           stream: int | None) -> int:
    """Raw C-ABI call of the failure-path test entry (a kernel wait runs out)."""
    return load_library().mk_attn_fwd_stall_test(q, k, v, o, lse, B, Hq, Hkv, S, D, int(causal),
                                                 float(scale), cu_seqlens, stream)


def mk_attn_error_string(status: int) -> str:
    return load_library().mk_attn_error_string(int(status)).decode()


def mk_attn_check_status(stream: int | None) -> int:
    return load_library().mk_attn_check_status(stream)


def mk_attn_version() -> int:
    return load_library().mk_attn_version()


def mk_attn_set_tuning(tuning: MkAttnTuning | None) -> int:
    """Raw C-ABI call; None restores the defaults."""
    return load_library().mk_attn_set_tuning(None if tuning is None else ctypes.byref(tuning))


def mk_attn_get_tuning() -> MkAttnTuning:
    t = MkAttnTuning()
    _check(load_library().mk_attn_get_tuning(ctypes.byref(t)))
    return t


def set_tuning(**fields) -> None:
    """Sets the process-wide tuning: the defaults, overridden by `fields`
    (ctas, schedule, rescale_log2, split_ctas_per_sm, split_min_pages)."""
    unknown = set(fields) - set(DEFAULT_TUNING)
    if unknown:
        raise ValueError(f"unknown tuning fields {sorted(unknown)}")
    _check(mk_attn_set_tuning(MkAttnTuning(**{**DEFAULT_TUNING, **fields})))


class tuning:
    """Context manager: `with tuning(ctas=120): ...` applies a tuning and
    restores the previous one on exit."""

    def __init__(self, **fields):
        self.fields = fields
        self.saved = None

    def __enter__(self):
        self.saved = mk_attn_get_tuning()
        set_tuning(**self.fields)
        return self

    def __exit__(self, *exc):
        _check(mk_attn_set_tuning(self.saved))
        return False


def _check(status: int):
    if status != MK_OK:
        raise MkAttnError(status, mk_attn_error_string(status))


def attn_fwd(q, k, v, causal: bool = True, scale: float | None = None, cu_seqlens=None,
             out=None, lse=None, stream=None):
    """Attention forward on CUDA tensors through mk_attn_fwd.

    q: [B,S,Hq,D] bf16 (or [T,Hq,D] with cu_seqlens, an int32 CUDA tensor
    [B+1]); k, v: [B,S,Hkv,D] (or [T,Hkv,D]).  Returns (o, lse): o like q (bf16),
    lse fp32 [B,Hq,S] (or [Hq,T]).  PyTorch only allocates the outputs and
    provides the stream."""
    import torch
    if not (q.is_cuda and k.is_cuda and v.is_cuda):
        raise ValueError("q, k, v must be CUDA tensors")
    if q.dtype != torch.bfloat16 or k.dtype != torch.bfloat16 or v.dtype != torch.bfloat16:
        raise ValueError("q, k, v must be bfloat16")
    if not (q.is_contiguous() and k.is_contiguous() and v.is_contiguous()):
        raise ValueError("q, k, v must be contiguous")
    if cu_seqlens is None:
        if q.dim() != 4 or k.dim() != 4 or k.shape != v.shape:
            raise ValueError("fixed-length layout is q [B,S,Hq,D], k/v [B,S,Hkv,D]")
        B, S, Hq, D = q.shape
        Hkv = k.shape[2]
        if k.shape[0] != B or k.shape[1] != S or k.shape[3] != D:
            raise ValueError("k/v shape does not match q")
        lse_shape = (B, Hq, S)
        cu_ptr = None
    else:
        if q.dim() != 3 or k.dim() != 3 or k.shape != v.shape:
            raise ValueError("varlen layout is q [T,Hq,D], k/v [T,Hkv,D]")
        if not cu_seqlens.is_cuda or cu_seqlens.dtype != torch.int32 or cu_seqlens.dim() != 1:
            raise ValueError("cu_seqlens must be a 1-D int32 CUDA tensor")
        S, Hq, D = q.shape
        Hkv = k.shape[1]
        B = cu_seqlens.numel() - 1
        if k.shape[0] != S or k.shape[2] != D:
            raise ValueError("k/v shape does not match q")
        lse_shape = (Hq, S)
        cu_ptr = cu_seqlens.data_ptr()
    if scale is None:
        scale = 1.0 / float(D) ** 0.5
    if out is None:
        out = torch.empty_like(q)
    if lse is None:
        lse = torch.empty(lse_shape, dtype=torch.float32, device=q.device)
    if stream is None:
        stream = torch.cuda.current_stream(q.device)
    _check(mk_attn_fwd(q.data_ptr(), k.data_ptr(), v.data_ptr(), out.data_ptr(), lse.data_ptr(),
                       B, Hq, Hkv, S, D, int(bool(causal)), float(scale), cu_ptr,
                       stream.cuda_stream))
    return out, lse


def mk_attn_bwd_workspace_bytes(B: int, Hq: int, S: int, varlen: int) -> int:
    return load_library().mk_attn_bwd_workspace_bytes(B, Hq, S, int(bool(varlen)))


def mk_attn_bwd(q: int, k: int, v: int, o: int, lse: int, do: int, dq: int, dk: int, dv: int,
                B: int, Hq: int, Hkv: int, S: int, D: int, causal: int, scale: float,
                cu_seqlens: int | None, workspace: int | None, workspace_bytes: int,
                stream: int | None) -> int:
    """Raw C-ABI call: integer device pointers in, status code out."""
    return load_library().mk_attn_bwd(q, k, v, o, lse, do, dq, dk, dv, B, Hq, Hkv, S, D,
                                      int(causal), float(scale), cu_seqlens, workspace,
                                      int(workspace_bytes), stream)


def mk_attn_bwd_stages(q: int, k: int, v: int, o: int, lse: int, do: int, dq: int, dk: int,
                       dv: int, B: int, Hq: int, Hkv: int, S: int, D: int, causal: int,
                       scale: float, cu_seqlens: int | None, workspace: int | None,
                       workspace_bytes: int, stages: int, stream: int | None) -> int:
    """Raw C-ABI call of selected backward stages (BWD_* flags)."""
    return load_library().mk_attn_bwd_stages(q, k, v, o, lse, do, dq, dk, dv, B, Hq, Hkv, S, D,
                                             int(causal), float(scale), cu_seqlens, workspace,
                                             int(workspace_bytes), int(stages), stream)


def attn_bwd(q, k, v, o, lse, do, causal: bool = True, scale: float | None = None,
             cu_seqlens=None, dq=None, dk=None, dv=None, workspace=None, stream=None,
             stages: int = BWD_ALL):
    """Attention backward on CUDA tensors through mk_attn_bwd.

    q, k, v, causal, scale, cu_seqlens as for attn_fwd; o, lse its outputs;
    do: bf16 gradient of o (layout of q).  Returns (dq, dk, dv), bf16, the
    layouts of q, k, v.  `stages` (BWD_* flags) enqueues only some stages:
    BWD_DQ computes Delta itself and writes it to `workspace`; BWD_DKDV reads
    the Delta an earlier BWD_DQ or BWD_DELTA stage wrote there.  PyTorch only
    allocates the outputs and the fp32 workspace and provides the stream."""
    import torch
    for name, t in (("q", q), ("k", k), ("v", v), ("o", o), ("do", do)):
        if not t.is_cuda or t.dtype != torch.bfloat16 or not t.is_contiguous():
            raise ValueError(f"{name} must be a contiguous bf16 CUDA tensor")
    if not lse.is_cuda or lse.dtype != torch.float32 or not lse.is_contiguous():
        raise ValueError("lse must be a contiguous fp32 CUDA tensor")
    if o.shape != q.shape or do.shape != q.shape or k.shape != v.shape:
        raise ValueError("o and do must have the shape of q, v that of k")
    if cu_seqlens is None:
        if q.dim() != 4:
            raise ValueError("fixed-length layout is q [B,S,Hq,D], k/v [B,S,Hkv,D]")
        B, S, Hq, D = q.shape
        Hkv = k.shape[2]
        lse_shape = (B, Hq, S)
        cu_ptr = None
    else:
        if q.dim() != 3:
            raise ValueError("varlen layout is q [T,Hq,D], k/v [T,Hkv,D]")
        if not cu_seqlens.is_cuda or cu_seqlens.dtype != torch.int32 or cu_seqlens.dim() != 1:
            raise ValueError("cu_seqlens must be a 1-D int32 CUDA tensor")
        S, Hq, D = q.shape
        Hkv = k.shape[1]
        B = cu_seqlens.numel() - 1
        lse_shape = (Hq, S)
        cu_ptr = cu_seqlens.data_ptr()
    if tuple(lse.shape) != lse_shape:
        raise ValueError(f"lse must have shape {lse_shape}")
    if scale is None:
        scale = 1.0 / float(D) ** 0.5
    dq = torch.empty_like(q) if dq is None else dq
    dk = torch.empty_like(k) if dk is None else dk
    dv = torch.empty_like(v) if dv is None else dv
    need = mk_attn_bwd_workspace_bytes(B, Hq, S, cu_seqlens is not None)
    if need < 0:
        raise MkAttnError(MK_ERR_INVALID_ARG, "invalid backward sizes")
    if workspace is None:
        workspace = torch.empty((need + 15) // 16 * 4, dtype=torch.float32, device=q.device)
    if stream is None:
        stream = torch.cuda.current_stream(q.device)
    _check(mk_attn_bwd_stages(q.data_ptr(), k.data_ptr(), v.data_ptr(), o.data_ptr(),
                              lse.data_ptr(), do.data_ptr(), dq.data_ptr(), dk.data_ptr(),
                              dv.data_ptr(), B, Hq, Hkv, S, D, int(bool(causal)), float(scale),
                              cu_ptr, workspace.data_ptr(),
                              workspace.numel() * workspace.element_size(), int(stages),
                              stream.cuda_stream))
    return dq, dk, dv


def mk_attn_decode_workspace_bytes(B: int, Hq: int, Hkv: int, D: int, page_size: int,
                                   max_pages: int) -> int:
    return load_library().mk_attn_decode_workspace_bytes(B, Hq, Hkv, D, page_size, max_pages)


def mk_attn_decode_paged(q: int, k_cache: int, v_cache: int, page_table: int, seq_lens: int,
                         o: int, lse: int, B: int, Hq: int, Hkv: int, D: int, page_size: int,
                         max_pages: int, num_pages: int, scale: float, workspace: int | None,
                         workspace_bytes: int, stream: int | None) -> int:
    """Raw C-ABI call: integer device pointers in, status code out."""
    return load_library().mk_attn_decode_paged(q, k_cache, v_cache, page_table, seq_lens, o, lse,
                                               B, Hq, Hkv, D, page_size, max_pages, num_pages,
                                               float(scale), workspace, int(workspace_bytes),
                                               stream)


def mk_attn_decode_paged_noalloc(q: int, k_cache: int, v_cache: int, page_table: int,
                                 seq_lens: int, o: int, lse: int, B: int, Hq: int, Hkv: int,
                                 D: int, page_size: int, max_pages: int, num_pages: int,
                                 scale: float, stream: int | None) -> int:
    """Raw C-ABI call of the decode step that uses the library's static
    scratch instead of a caller workspace: integer device pointers in, status
    code out."""
    return load_library().mk_attn_decode_paged_noalloc(q, k_cache, v_cache, page_table, seq_lens,
                                                       o, lse, B, Hq, Hkv, D, page_size,
                                                       max_pages, num_pages, float(scale), stream)


def decode_paged(q, k_cache, v_cache, page_table, seq_lens, scale: float | None = None,
                 out=None, lse=None, workspace=None, stream=None):
    """One decode step against a paged K/V cache through mk_attn_decode_paged.

    q: [B,Hq,D] bf16; k_cache/v_cache: [num_pages, page_size, Hkv, D] bf16;
    page_table: int32 [B, max_pages]; seq_lens: int32 [B]; all CUDA tensors.
    Returns (o [B,Hq,D] bf16, lse [B,Hq] fp32).  The fp32 workspace for the
    split partials is allocated here unless one is passed."""
    import torch
    for name, t in (("q", q), ("k_cache", k_cache), ("v_cache", v_cache)):
        if not t.is_cuda or t.dtype != torch.bfloat16 or not t.is_contiguous():
            raise ValueError(f"{name} must be a contiguous bf16 CUDA tensor")
    for name, t in (("page_table", page_table), ("seq_lens", seq_lens)):
        if not t.is_cuda or t.dtype != torch.int32 or not t.is_contiguous():
            raise ValueError(f"{name} must be a contiguous int32 CUDA tensor")
    if q.dim() != 3 or k_cache.dim() != 4 or k_cache.shape != v_cache.shape:
        raise ValueError("q [B,Hq,D], k_cache/v_cache [num_pages, page_size, Hkv, D]")
    B, Hq, D = q.shape
    num_pages, page_size, Hkv, Dk = k_cache.shape
    if Dk != D or page_table.dim() != 2 or page_table.shape[0] != B or seq_lens.shape != (B,):
        raise ValueError("shapes do not match")
    max_pages = page_table.shape[1]
    if scale is None:
        scale = 1.0 / float(D) ** 0.5
    if out is None:
        out = torch.empty_like(q)
    if lse is None:
        lse = torch.empty((B, Hq), dtype=torch.float32, device=q.device)
    need = mk_attn_decode_workspace_bytes(B, Hq, Hkv, D, page_size, max_pages)
    if need < 0:
        raise MkAttnError(MK_ERR_INVALID_ARG, "invalid decode sizes")
    if workspace is None and need > 0:
        workspace = torch.empty((need + 15) // 16 * 4, dtype=torch.float32, device=q.device)
    ws_ptr = None if workspace is None else workspace.data_ptr()
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    if stream is None:
        stream = torch.cuda.current_stream(q.device)
    _check(mk_attn_decode_paged(q.data_ptr(), k_cache.data_ptr(), v_cache.data_ptr(),
                                page_table.data_ptr(), seq_lens.data_ptr(), out.data_ptr(),
                                lse.data_ptr(), B, Hq, Hkv, D, page_size, max_pages, num_pages,
                                float(scale), ws_ptr, ws_bytes, stream.cuda_stream))
    return out, lse


def mk_attn_mla_decode_workspace_bytes(B: int, Hq: int, page_size: int, max_pages: int) -> int:
    return load_library().mk_attn_mla_decode_workspace_bytes(B, Hq, page_size, max_pages)


def mk_attn_mla_decode_paged(q: int, cache: int, page_table: int, seq_lens: int, o: int, lse: int,
                             B: int, Hq: int, page_size: int, max_pages: int, num_pages: int,
                             scale: float, workspace: int | None, workspace_bytes: int,
                             stream: int | None) -> int:
    """Raw C-ABI call: integer device pointers in, status code out."""
    return load_library().mk_attn_mla_decode_paged(q, cache, page_table, seq_lens, o, lse, B, Hq,
                                                   page_size, max_pages, num_pages, float(scale),
                                                   workspace, int(workspace_bytes), stream)


def mla_decode_paged(q, cache, page_table, seq_lens, scale: float | None = None, out=None,
                     lse=None, workspace=None, stream=None):
    """One latent (MLA) decode step through mk_attn_mla_decode_paged.

    q: [B, Hq, 576] bf16; cache: [num_pages, page_size, 576] bf16 (keys in
    full, values = the first 512 components); page_table: int32 [B,
    max_pages]; seq_lens: int32 [B]; all CUDA tensors.  Returns (o [B, Hq,
    512] bf16, lse [B, Hq] fp32).  The fp32 split workspace is allocated here
    unless one is passed."""
    import torch
    for name, t in (("q", q), ("cache", cache)):
        if not t.is_cuda or t.dtype != torch.bfloat16 or not t.is_contiguous():
            raise ValueError(f"{name} must be a contiguous bf16 CUDA tensor")
    for name, t in (("page_table", page_table), ("seq_lens", seq_lens)):
        if not t.is_cuda or t.dtype != torch.int32 or not t.is_contiguous():
            raise ValueError(f"{name} must be a contiguous int32 CUDA tensor")
    if q.dim() != 3 or q.shape[2] != MLA_DQK or cache.dim() != 3 or cache.shape[2] != MLA_DQK:
        raise ValueError(f"q [B, Hq, {MLA_DQK}], cache [num_pages, page_size, {MLA_DQK}]")
    B, Hq, _ = q.shape
    num_pages, page_size, _ = cache.shape
    if page_table.dim() != 2 or page_table.shape[0] != B or seq_lens.shape != (B,):
        raise ValueError("page_table [B, max_pages], seq_lens [B]")
    max_pages = page_table.shape[1]
    if scale is None:
        scale = 1.0 / float(MLA_DQK) ** 0.5
    if out is None:
        out = torch.empty((B, Hq, MLA_DV), dtype=torch.bfloat16, device=q.device)
    if lse is None:
        lse = torch.empty((B, Hq), dtype=torch.float32, device=q.device)
    need = mk_attn_mla_decode_workspace_bytes(B, Hq, page_size, max_pages)
    if need < 0:
        raise MkAttnError(MK_ERR_INVALID_ARG, "invalid MLA decode sizes")
    if workspace is None and need > 0:
        workspace = torch.empty((need + 15) // 16 * 4, dtype=torch.float32, device=q.device)
    ws_ptr = None if workspace is None else workspace.data_ptr()
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    if stream is None:
        stream = torch.cuda.current_stream(q.device)
    _check(mk_attn_mla_decode_paged(q.data_ptr(), cache.data_ptr(), page_table.data_ptr(),
                                    seq_lens.data_ptr(), out.data_ptr(), lse.data_ptr(), B, Hq,
                                    page_size, max_pages, num_pages, float(scale), ws_ptr,
                                    ws_bytes, stream.cuda_stream))
    return out, lse
