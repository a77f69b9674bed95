"""The check build (MK_DEBUG) compiles for sm_103a without a GPU, exports every
symbol that include/*.h declares, and rejects invalid arguments on the host
exactly as the release build does."""
import ctypes
import os

import pytest

from paper_2609_04523_gb300 import binding
from paper_2609_04523_gb300.build import build_library

from test_abi import declared_symbols

A = 0x10000


@pytest.fixture(scope="module")
def check_lib():
    path = build_library(debug=True)
    assert os.path.basename(path) == "libmk_attn_debug.so"
    lib = ctypes.CDLL(path)
    vp, i = ctypes.c_void_p, ctypes.c_int
    lib.mk_attn_fwd.argtypes = [vp, vp, vp, vp, vp, i, i, i, i, i, i, ctypes.c_float, vp, vp]
    lib.mk_attn_fwd.restype = i
    lib.mk_attn_error_string.argtypes = [i]
    lib.mk_attn_error_string.restype = ctypes.c_char_p
    return lib


def test_check_build_exports_every_declared_symbol(check_lib):
    for name in declared_symbols():
        assert hasattr(check_lib, name), f"{name} missing from the check build"


def test_check_build_has_the_bounds_status(check_lib):
    assert b"check" in check_lib.mk_attn_error_string(binding.MK_ERR_BOUNDS)


@pytest.mark.parametrize("args, want", [
    ((0, 2 * A, 3 * A, 4 * A, 5 * A, 2, 8, 2, 256, 128, 1, 0.1, None, None),
     binding.MK_ERR_INVALID_ARG),
    ((A, 2 * A, 3 * A, 4 * A, 5 * A, 2, 8, 3, 256, 128, 1, 0.1, None, None),
     binding.MK_ERR_INVALID_ARG),
    ((A, 2 * A, 3 * A, 4 * A, 5 * A, 2, 8, 2, 256, 96, 1, 0.1, None, None),
     binding.MK_ERR_UNSUPPORTED),
    ((A + 8, 2 * A, 3 * A, 4 * A, 5 * A, 2, 8, 2, 256, 128, 1, 0.1, None, None),
     binding.MK_ERR_ALIGNMENT),
])
def test_check_build_rejects_on_host_like_the_release_build(check_lib, args, want):
    build_library()
    assert check_lib.mk_attn_fwd(*args) == want
    assert binding.load_library().mk_attn_fwd(*args) == want
