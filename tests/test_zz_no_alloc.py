"""The allocation-free decode entry point, on the GPU.

mk_attn_decode_paged_noalloc serves callers that cannot allocate device
memory (code running under an allocator that another runtime owns, inside
host callbacks, or in plugins that must not grow the device heap): its split
partials go to a fixed 16 MiB array that the library declares in device
memory instead of a caller workspace.  These tests call it through the C ABI
and check it
  - against mk_attn_decode_paged with a workspace: both run the same kernels
    with the same split plan, so the outputs must agree bit for bit (which
    also holds them within the decode tests' tolerances);
  - against the fp64 oracle, within the decode tests' tolerances;
on two calls in a row: the second call has the same sizes but shorter
sequences, so a merge that read partials the first call left in the shared
array would show;
  - that a warm call changes the device's free memory by nothing;
  - that sizes needing more scratch than the array holds are refused before
    anything is launched.

The file name makes pytest collect it last."""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2609_04523_gb300 import binding
from paper_2609_04523_gb300 import workloads as W

pytestmark = pytest.mark.gpu

O_MAX_ABS, O_REL_RMS, LSE_MAX_ABS = 2e-2, 5e-3, 1e-3


def _device_args(inp):
    dev = torch.device("cuda")
    return [t.to(dev).contiguous() for t in
            (inp.q, inp.k_cache, inp.v_cache, inp.page_table, inp.seq_lens)]


def _sizes(inp):
    B, Hq, D = inp.q.shape
    num_pages, page_size, Hkv, _ = inp.k_cache.shape
    return B, Hq, Hkv, D, page_size, inp.page_table.shape[1], num_pages


def _outputs(q):
    o = torch.full_like(q, float("nan"))
    lse = torch.full(tuple(q.shape[:2]), float("nan"), dtype=torch.float32, device=q.device)
    return o, lse


def _call_noalloc(args, inp, o, lse, stream):
    q, kc, vc, pt, sl = args
    B, Hq, Hkv, D, ps, mp, npg = _sizes(inp)
    return binding.mk_attn_decode_paged_noalloc(
        q.data_ptr(), kc.data_ptr(), vc.data_ptr(), pt.data_ptr(), sl.data_ptr(), o.data_ptr(),
        lse.data_ptr(), B, Hq, Hkv, D, ps, mp, npg, inp.scale, stream)


def _call_workspace(args, inp, o, lse, stream):
    q, kc, vc, pt, sl = args
    B, Hq, Hkv, D, ps, mp, npg = _sizes(inp)
    need = binding.mk_attn_decode_workspace_bytes(B, Hq, Hkv, D, ps, mp)
    ws = torch.empty(max(need, 16) // 4 + 4, dtype=torch.float32, device=q.device)
    st = binding.mk_attn_decode_paged(
        q.data_ptr(), kc.data_ptr(), vc.data_ptr(), pt.data_ptr(), sl.data_ptr(), o.data_ptr(),
        lse.data_ptr(), B, Hq, Hkv, D, ps, mp, npg, inp.scale, ws.data_ptr(), ws.numel() * 4,
        stream)
    return st, ws


def _compare(o, lse, o_ref, lse_ref, what):
    o = o.float().cpu().numpy()
    o_ref = np.asarray(o_ref.float().cpu().numpy() if torch.is_tensor(o_ref) else o_ref)
    lse = lse.double().cpu().numpy()
    lse_ref = np.asarray(lse_ref.double().cpu().numpy() if torch.is_tensor(lse_ref) else lse_ref)
    assert np.all(np.isfinite(o)), f"{what}: o has unwritten entries"
    fin = np.isfinite(lse_ref)
    assert np.array_equal(fin, np.isfinite(lse)), f"{what}: empty rows differ"
    d = o - o_ref
    max_abs = float(np.max(np.abs(d)))
    rel = math.sqrt(float(np.sum(d * d)) / max(float(np.sum(o_ref * o_ref)), 1e-300))
    lerr = float(np.max(np.abs(lse[fin] - lse_ref[fin]))) if fin.any() else 0.0
    assert max_abs <= O_MAX_ABS, f"{what}: o max_abs {max_abs:.3e}"
    assert rel <= O_REL_RMS, f"{what}: o rel_rms {rel:.3e}"
    assert lerr <= LSE_MAX_ABS, f"{what}: lse err {lerr:.3e}"


def _shorter(inp, lens):
    """The same decode step with shorter sequences (same sizes and pages)."""
    sl = torch.tensor(lens, dtype=torch.int32)
    assert torch.all(sl <= inp.seq_lens)
    return W.PagedInputs(inp.q, inp.k_cache, inp.v_cache, inp.page_table, sl, inp.scale)


@pytest.mark.parametrize("case", [0, 1])
def test_noalloc_matches_workspace_entry_and_oracle_on_two_calls_in_a_row(case):
    """Two decode steps of the same sizes, both with several KV splits, so
    both go through the static scratch; the second has shorter sequences and
    is checked after the first has left its partials there."""
    first = [W.make_paged([5000, 1, 0, 2100], 16, 4, 128, 64, seed=901),
             W.make_paged([3, 4000, 777], 24, 3, 64, 32, seed=902)][case]
    second = _shorter(first, [[300, 1, 0, 1000], [3, 129, 40]][case])
    stream = torch.cuda.current_stream().cuda_stream
    for n, inp in enumerate((first, second)):
        B, Hq, Hkv, D, ps, mp, _ = _sizes(inp)
        need = binding.mk_attn_decode_workspace_bytes(B, Hq, Hkv, D, ps, mp)
        assert 0 < need <= binding.DECODE_STATIC_SCRATCH_BYTES, f"call {n + 1}: need {need}"
        args = _device_args(inp)
        o_ws, lse_ws = _outputs(args[0])
        st, _ws = _call_workspace(args, inp, o_ws, lse_ws, stream)
        assert st == binding.MK_OK, binding.mk_attn_error_string(st)
        o, lse = _outputs(args[0])
        st = _call_noalloc(args, inp, o, lse, stream)
        assert st == binding.MK_OK, binding.mk_attn_error_string(st)
        assert binding.mk_attn_check_status(stream) == binding.MK_OK
        what = f"case {case} call {n + 1}"
        assert torch.equal(o.view(torch.int16), o_ws.view(torch.int16)), f"{what}: o differs"
        assert torch.equal(lse, lse_ws), f"{what}: lse differs"
        _compare(o, lse, o_ws, lse_ws, what + " vs workspace entry")
        o_ref, lse_ref = oracle.decode_paged(inp.q, inp.k_cache, inp.v_cache, inp.page_table,
                                             inp.seq_lens, inp.scale)
        _compare(o, lse, o_ref, lse_ref, what + " vs oracle")


def test_warm_noalloc_call_allocates_nothing():
    """After a first call (which looks up the scratch address and loads the
    library's decode kernels), a call changes the device's free memory by
    nothing."""
    inp = W.make_paged([3000, 17, 900], 16, 4, 128, 64, seed=904)
    args = _device_args(inp)
    o, lse = _outputs(args[0])
    stream = torch.cuda.current_stream().cuda_stream
    assert _call_noalloc(args, inp, o, lse, stream) == binding.MK_OK
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    assert _call_noalloc(args, inp, o, lse, stream) == binding.MK_OK
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert free1 == free0, f"free device memory moved by {free0 - free1} bytes"
    assert binding.mk_attn_check_status(stream) == binding.MK_OK


def test_noalloc_refuses_sizes_beyond_its_scratch():
    """Sizes whose split partials exceed the static array are refused with
    MK_ERR_SCRATCH_LIMIT and nothing is launched: the outputs stay as they
    were.  The batch is chosen from the planned workspace size on this GPU."""
    Hq, Hkv, D, ps, mp = 8, 1, 128, 16, 64
    B = next((b for b in range(1, 8192)
              if binding.mk_attn_decode_workspace_bytes(b, Hq, Hkv, D, ps, mp)
              > binding.DECODE_STATIC_SCRATCH_BYTES), None)
    if B is None:
        pytest.skip("no batch below 8192 needs more scratch than the static array on this GPU")
    inp = W.make_paged([20] * B, Hq, Hkv, D, ps, seed=903, max_pages=mp)
    args = _device_args(inp)
    o, lse = _outputs(args[0])
    stream = torch.cuda.current_stream().cuda_stream
    st = _call_noalloc(args, inp, o, lse, stream)
    assert st == binding.MK_ERR_SCRATCH_LIMIT
    assert "scratch" in binding.mk_attn_error_string(st)
    assert binding.mk_attn_check_status(stream) == binding.MK_OK
    assert torch.isnan(o.float()).all() and torch.isnan(lse).all()
