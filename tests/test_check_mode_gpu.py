"""Check mode (MK_ATTN_DEBUG) and check build (MK_DEBUG) on the GPU, on valid
inputs: each runs tests/check_mode_run.py in a child process (both switches
are read once per process), which calls every kernel family through the C ABI
and compares with the fp64 oracle.  Under the check mode every call returns
the device status after synchronising, so a device-side error would fail the
call itself; the check build's store-index checks must all pass."""
import os
import subprocess
import sys

import pytest
import torch

from paper_2609_04523_gb300.build import build_library

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.mark.parametrize("debug_env, check_build", [("1", False), ("0", True), ("1", True)])
def test_every_family_green_under_check_mode_and_check_build(debug_env, check_build):
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need a CUDA device")
    build_library(debug=True)
    env = dict(os.environ)
    env["MK_ATTN_DEBUG"] = debug_env
    env["MK_ATTN_CHECK_BUILD"] = "1" if check_build else "0"
    r = subprocess.run([sys.executable, os.path.join(ROOT, "tests", "check_mode_run.py")],
                       env=env, capture_output=True, text=True, timeout=600)
    out = r.stdout + r.stderr
    assert r.returncode == 0, out[-3000:]
    want = "libmk_attn_debug.so" if check_build else "libmk_attn.so"
    assert f"library: {want}" in out, out[-3000:]
    assert "check mode run: ok" in out
