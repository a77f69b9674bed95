"""Failure detection on the GPU without a fault: a kernel wait that nothing
ever satisfies runs into its time limit, every CTA unwinds, the launch reports
MK_ERR_TIMEOUT through mk_attn_check_status, and the CUDA context stays usable
(the next ordinary call is correct)."""
import math
import time

import numpy as np
import pytest
import torch

import oracle
from paper_2609_04523_gb300 import binding
from paper_2609_04523_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def test_wait_timeout_is_reported_and_context_survives():
    dev = torch.device("cuda")
    B, Hq, Hkv, S, D = 1, 4, 2, 300, 128
    scale = 1.0 / math.sqrt(D)
    q, k, v, _ = W.make_qkv(B, Hq, Hkv, S, D, seed=900)
    qd, kd, vd = q.to(dev), k.to(dev), v.to(dev)
    o = torch.empty_like(qd)
    lse = torch.empty((B, Hq, S), dtype=torch.float32, device=dev)
    st = torch.cuda.current_stream().cuda_stream
    assert binding.mk_attn_check_status(st) == binding.MK_OK

    t0 = time.perf_counter()
    rc = binding.mk_attn_fwd_stall_test(qd.data_ptr(), kd.data_ptr(), vd.data_ptr(), o.data_ptr(),
                                        lse.data_ptr(), B, Hq, Hkv, S, D, 1, scale, None, st)
    assert rc == binding.MK_OK
    status = binding.mk_attn_check_status(st)
    elapsed = time.perf_counter() - t0
    assert status == binding.MK_ERR_TIMEOUT, binding.mk_attn_error_string(status)
    assert 1.0 < elapsed < 60.0, elapsed          # the 2 s wait limit, then the unwind
    assert binding.mk_attn_check_status(st) == binding.MK_OK  # the status word was cleared

    o2, lse2 = binding.attn_fwd(qd, kd, vd, True, scale)
    assert binding.mk_attn_check_status(st) == binding.MK_OK
    o_ref, lse_ref = oracle.attn_fwd(q, k, v, True, scale)
    err_o = float(np.max(np.abs(o2.float().cpu().numpy() - o_ref)))
    err_lse = float(np.max(np.abs(lse2.double().cpu().numpy() - lse_ref)))
    assert err_o <= 2e-2 and err_lse <= 1e-3, (err_o, err_lse)
