"""The C-ABI library loads, exports what include/*.h declares, and rejects
invalid arguments on the host before any CUDA call (no GPU needed)."""
import glob
import os
import re

import pytest

from paper_2609_04523_gb300 import binding
from paper_2609_04523_gb300.build import build_library

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    build_library()
    return binding.load_library()


def declared_symbols():
    names = set()
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        text = open(h).read()
        names |= set(re.findall(r"MK_API\s+[\w\s\*]*?\b(mk_\w+)\s*\(", text))
    return names


def test_header_declares_the_entry_points():
    assert {"mk_attn_fwd", "mk_attn_error_string", "mk_attn_check_status",
            "mk_attn_version"} <= declared_symbols()


def test_every_declared_symbol_is_exported(lib):
    for name in declared_symbols():
        assert hasattr(lib, name), f"{name} declared in include/ but not exported"


def test_version_and_error_strings(lib):
    assert binding.mk_attn_version() >= 100
    for st in (0, -1, -2, -3, -4, -5, -99):
        assert isinstance(binding.mk_attn_error_string(st), str)
    assert "align" in binding.mk_attn_error_string(binding.MK_ERR_ALIGNMENT)


A = 0x10000  # fake 16-byte-aligned addresses: never dereferenced by a rejected call
GOOD = dict(q=A, k=2 * A, v=3 * A, o=4 * A, lse=5 * A, B=2, Hq=8, Hkv=2, S=256, D=128,
            causal=1, scale=0.088, cu_seqlens=None, stream=None)


def call(**kw):
    args = dict(GOOD)
    args.update(kw)
    return binding.mk_attn_fwd(**args)


@pytest.mark.parametrize("kw, want", [
    (dict(q=None), binding.MK_ERR_INVALID_ARG),
    (dict(k=None), binding.MK_ERR_INVALID_ARG),
    (dict(v=None), binding.MK_ERR_INVALID_ARG),
    (dict(o=None), binding.MK_ERR_INVALID_ARG),
    (dict(lse=None), binding.MK_ERR_INVALID_ARG),
    (dict(B=0), binding.MK_ERR_INVALID_ARG),
    (dict(S=0), binding.MK_ERR_INVALID_ARG),
    (dict(Hq=0), binding.MK_ERR_INVALID_ARG),
    (dict(Hkv=0), binding.MK_ERR_INVALID_ARG),
    (dict(Hkv=3), binding.MK_ERR_INVALID_ARG),
    (dict(B=-1), binding.MK_ERR_INVALID_ARG),
    (dict(scale=float("nan")), binding.MK_ERR_INVALID_ARG),
    (dict(scale=float("inf")), binding.MK_ERR_INVALID_ARG),
    (dict(D=96), binding.MK_ERR_UNSUPPORTED),
    (dict(D=256), binding.MK_ERR_UNSUPPORTED),
    (dict(D=0), binding.MK_ERR_UNSUPPORTED),
    (dict(q=A + 8), binding.MK_ERR_ALIGNMENT),
    (dict(o=A + 2), binding.MK_ERR_ALIGNMENT),
    (dict(lse=A + 4), binding.MK_ERR_ALIGNMENT),
    (dict(cu_seqlens=A + 2), binding.MK_ERR_ALIGNMENT),
    (dict(B=1 << 20, S=1 << 12), binding.MK_ERR_INVALID_ARG),  # token count overflows int32
])
def test_invalid_arguments_rejected_on_host(lib, kw, want):
    assert call(**kw) == want


def test_missing_library_fails_loudly(monkeypatch, tmp_path):
    monkeypatch.setattr(binding, "_lib", None)
    monkeypatch.setattr(binding, "LIB_PATH", str(tmp_path / "absent.so"))
    with pytest.raises(binding.MkAttnError):
        binding.load_library()


# The other entry points check their arguments on the host before their first
# CUDA call too, so these rejections need no GPU.  (Checks that depend on the
# device -- the decode split plan's workspace size -- are covered by the GPU
# tests.)
BWD_GOOD = dict(q=A, k=2 * A, v=3 * A, o=4 * A, lse=5 * A, do=6 * A, dq=7 * A, dk=8 * A,
                dv=9 * A, B=2, Hq=8, Hkv=2, S=256, D=128, causal=1, scale=0.088,
                cu_seqlens=None, workspace=10 * A, workspace_bytes=2 * 8 * 256 * 4,
                stages=binding.BWD_ALL, stream=None)


@pytest.mark.parametrize("kw, want", [
    (dict(stages=0), binding.MK_ERR_INVALID_ARG),
    (dict(stages=8), binding.MK_ERR_INVALID_ARG),
    (dict(do=None), binding.MK_ERR_INVALID_ARG),
    (dict(dv=None), binding.MK_ERR_INVALID_ARG),
    (dict(workspace=None), binding.MK_ERR_INVALID_ARG),
    (dict(Hkv=3), binding.MK_ERR_INVALID_ARG),
    (dict(scale=float("nan")), binding.MK_ERR_INVALID_ARG),
    (dict(D=96), binding.MK_ERR_UNSUPPORTED),
    (dict(Hq=65536 * 2, Hkv=2), binding.MK_ERR_UNSUPPORTED),
    (dict(workspace_bytes=2 * 8 * 256 * 4 - 4), binding.MK_ERR_INVALID_ARG),
    (dict(dq=7 * A + 8), binding.MK_ERR_ALIGNMENT),
    (dict(workspace=10 * A + 4), binding.MK_ERR_ALIGNMENT),
    (dict(lse=5 * A + 2), binding.MK_ERR_ALIGNMENT),
])
def test_backward_rejects_on_host(lib, kw, want):
    args = dict(BWD_GOOD)
    args.update(kw)
    assert binding.mk_attn_bwd_stages(**args) == want


DEC_GOOD = dict(q=A, k_cache=2 * A, v_cache=3 * A, page_table=4 * A, seq_lens=5 * A, o=6 * A,
                lse=7 * A, B=4, Hq=8, Hkv=2, D=128, page_size=64, max_pages=16, num_pages=64,
                scale=0.088, workspace=None, workspace_bytes=0, stream=None)


@pytest.mark.parametrize("kw, want", [
    (dict(q=None), binding.MK_ERR_INVALID_ARG),
    (dict(page_table=None), binding.MK_ERR_INVALID_ARG),
    (dict(Hkv=3), binding.MK_ERR_INVALID_ARG),
    (dict(max_pages=0), binding.MK_ERR_INVALID_ARG),
    (dict(scale=float("inf")), binding.MK_ERR_INVALID_ARG),
    (dict(D=256), binding.MK_ERR_UNSUPPORTED),
    (dict(page_size=48), binding.MK_ERR_UNSUPPORTED),
    (dict(B=70000), binding.MK_ERR_UNSUPPORTED),
    (dict(num_pages=1 << 26), binding.MK_ERR_INVALID_ARG),
    (dict(o=6 * A + 8), binding.MK_ERR_ALIGNMENT),
    (dict(seq_lens=5 * A + 2), binding.MK_ERR_ALIGNMENT),
])
def test_paged_decode_rejects_on_host(lib, kw, want):
    args = dict(DEC_GOOD)
    args.update(kw)
    assert binding.mk_attn_decode_paged(**args) == want


MLA_GOOD = dict(q=A, cache=2 * A, page_table=3 * A, seq_lens=4 * A, o=5 * A, lse=6 * A, B=4,
                Hq=128, page_size=64, max_pages=16, num_pages=64, scale=0.04, workspace=None,
                workspace_bytes=0, stream=None)


@pytest.mark.parametrize("kw, want", [
    (dict(cache=None), binding.MK_ERR_INVALID_ARG),
    (dict(B=0), binding.MK_ERR_INVALID_ARG),
    (dict(num_pages=0), binding.MK_ERR_INVALID_ARG),
    (dict(scale=float("nan")), binding.MK_ERR_INVALID_ARG),
    (dict(page_size=8), binding.MK_ERR_UNSUPPORTED),
    (dict(max_pages=1 << 26), binding.MK_ERR_INVALID_ARG),
    (dict(q=A + 8), binding.MK_ERR_ALIGNMENT),
    (dict(lse=6 * A + 2), binding.MK_ERR_ALIGNMENT),
])
def test_latent_decode_rejects_on_host(lib, kw, want):
    args = dict(MLA_GOOD)
    args.update(kw)
    assert binding.mk_attn_mla_decode_paged(**args) == want


def test_binding_constants_match_the_header():
    """Constants the binding restates from include/mk_attn.h."""
    text = open(os.path.join(ROOT, "include", "mk_attn.h")).read()
    m = re.search(r"#define\s+MK_ATTN_DECODE_STATIC_SCRATCH_BYTES\s+\(([^)]*)\)", text)
    assert m, "MK_ATTN_DECODE_STATIC_SCRATCH_BYTES not found"
    assert eval(m.group(1), {"__builtins__": {}}) == binding.DECODE_STATIC_SCRATCH_BYTES
    codes = dict(re.findall(r"\b(MK_(?:OK|ERR_\w+))\s*=\s*(-?\d+)", text))
    assert codes, "status codes not found"
    for name, val in codes.items():
        assert getattr(binding, name) == int(val), name
    for name in ("MK_MLA_DQK", "MK_MLA_DV"):
        m = re.search(r"#define\s+%s\s+(\d+)" % name, text)
        assert int(m.group(1)) == getattr(binding, name.replace("MK_", ""))


# The allocation-free decode entry point runs the host checks of
# mk_attn_decode_paged before anything else (no CUDA call), so it rejects the
# same arguments with the same status.
@pytest.mark.parametrize("kw, want", [
    (dict(q=None), binding.MK_ERR_INVALID_ARG),
    (dict(seq_lens=None), binding.MK_ERR_INVALID_ARG),
    (dict(Hkv=3), binding.MK_ERR_INVALID_ARG),
    (dict(num_pages=0), binding.MK_ERR_INVALID_ARG),
    (dict(scale=float("nan")), binding.MK_ERR_INVALID_ARG),
    (dict(D=256), binding.MK_ERR_UNSUPPORTED),
    (dict(page_size=48), binding.MK_ERR_UNSUPPORTED),
    (dict(page_size=48, B=60000), binding.MK_ERR_UNSUPPORTED),  # not MK_ERR_SCRATCH_LIMIT
    (dict(B=70000), binding.MK_ERR_UNSUPPORTED),
    (dict(num_pages=1 << 26), binding.MK_ERR_INVALID_ARG),
    (dict(o=6 * A + 8), binding.MK_ERR_ALIGNMENT),
    (dict(lse=7 * A + 2), binding.MK_ERR_ALIGNMENT),
])
def test_noalloc_decode_rejects_on_host(lib, kw, want):
    args = dict(DEC_GOOD)
    args.update(kw)
    del args["workspace"], args["workspace_bytes"]
    assert binding.mk_attn_decode_paged_noalloc(**args) == want
    full = dict(DEC_GOOD)
    full.update(kw)
    assert binding.mk_attn_decode_paged(**full) == want
