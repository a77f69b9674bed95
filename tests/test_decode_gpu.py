"""Paged decode step on the GPU against the fp64 oracle, through the C ABI.

Same bar as the forward pass: o max-abs <= 2e-2 and relative RMS <= 5e-3,
lse max-abs <= 1e-3; a sequence with no cached key must give o = 0 and
lse = -inf exactly."""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2609_04523_gb300 import binding
from paper_2609_04523_gb300 import workloads as W

pytestmark = pytest.mark.gpu

O_MAX_ABS, O_REL_RMS, LSE_MAX_ABS = 2e-2, 5e-3, 1e-3


def run_gpu(inp, scale=None):
    dev = torch.device("cuda")
    args = [t.to(dev) for t in (inp.q, inp.k_cache, inp.v_cache, inp.page_table, inp.seq_lens)]
    o = torch.full_like(args[0], float("nan"))
    lse = torch.full(tuple(inp.q.shape[:2]), float("nan"), dtype=torch.float32, device=dev)
    binding.decode_paged(*args, scale=inp.scale if scale is None else scale, out=o, lse=lse)
    assert binding.mk_attn_check_status(torch.cuda.current_stream().cuda_stream) == binding.MK_OK
    return o.float().cpu().numpy(), lse.double().cpu().numpy()


def check(inp, what):
    o, lse = run_gpu(inp)
    o_ref, lse_ref = oracle.decode_paged(inp.q, inp.k_cache, inp.v_cache, inp.page_table,
                                         inp.seq_lens, inp.scale)
    empty = np.asarray(inp.seq_lens) == 0
    assert np.all(o[empty] == 0.0) and np.all(np.isneginf(lse[empty])), f"{what}: empty rows"
    o, lse, o_ref, lse_ref = o[~empty], lse[~empty], o_ref[~empty], lse_ref[~empty]
    if o.size == 0:
        return
    d = o - o_ref
    max_abs = float(np.max(np.abs(d)))
    rel = math.sqrt(float(np.sum(d * d)) / max(float(np.sum(o_ref * o_ref)), 1e-300))
    lerr = float(np.max(np.abs(lse - lse_ref)))
    assert max_abs <= O_MAX_ABS, f"{what}: o max_abs {max_abs:.3e}"
    assert rel <= O_REL_RMS, f"{what}: o rel_rms {rel:.3e}"
    assert lerr <= LSE_MAX_ABS, f"{what}: lse err {lerr:.3e}"


@pytest.mark.parametrize("D", [64, 128])
@pytest.mark.parametrize("page_size", [16, 32, 64, 128])
@pytest.mark.parametrize("G", [1, 2, 3, 4, 8, 11, 16])
def test_decode_lengths(D, page_size, G):
    """G picks the CTA's head capacity (1, 2, 4, 8); 3 leaves capacity unused,
    11 splits a group into CTAs of 6 and 5 heads, 16 into two full CTAs."""
    lens = [0, 1, page_size - 1, page_size, page_size + 1, 3 * page_size + 7, 1000, 2049]
    Hkv = 2
    inp = W.make_paged(lens, Hkv * G, Hkv, D, page_size, seed=600 + D + page_size + G)
    check(inp, f"D{D} ps{page_size} G{G}")


def test_decode_wide_group():
    """32 query heads per key/value head: four CTAs of 8 heads each."""
    inp = W.make_paged([1, 700, 2500], 64, 2, 128, 32, seed=655)
    check(inp, "G32")


@pytest.mark.parametrize("B", [1, 3, 40])
def test_decode_splits(B):
    """Few sequences: many KV splits per (b, g), merged by log-sum-exp; many
    sequences: a single split writes o and lse directly."""
    rng = np.random.default_rng(B)
    lens = [int(x) for x in rng.integers(1, 6000, size=B)]
    inp = W.make_paged(lens, 16, 4, 128, 64, seed=700 + B)
    check(inp, f"B{B}")


def test_decode_one_long_sequence():
    """One sequence of 131072 cached keys (2048 pages of 64): every split of the
    plan belongs to it, and the merge combines them all."""
    inp = W.make_paged([131072], 8, 2, 128, 64, seed=716)
    check(inp, "L131072")


def test_decode_many_sequences():
    """3000 sequences of 0..199 cached keys (page 16): one split each for most,
    a grid of 3000 sequences in z, empty sequences among them."""
    rng = np.random.default_rng(715)
    lens = [int(x) for x in rng.integers(0, 200, size=3000)]
    inp = W.make_paged(lens, 8, 2, 128, 16, seed=715)
    check(inp, "B3000")


def test_decode_uneven_lengths_with_empty_splits():
    """One long sequence sets max_pages; the short ones leave most of their
    splits empty (lse -inf partials), which the merge must ignore."""
    lens = [9000, 3, 0, 130, 64]
    inp = W.make_paged(lens, 8, 2, 128, 32, seed=710)
    check(inp, "uneven")


def test_decode_large_logits():
    """q and k with sigma 3 (logits 9x larger, sharp softmax rows).  v is
    scaled by 1/4 (exact in bf16) so that o stays at unit scale: the absolute
    bound on o assumes unit-variance values, and bf16 rounding of o alone
    grows with its magnitude."""
    inp = W.make_paged([777, 1500], 8, 8, 64, 16, seed=720, sigma=3.0)
    inp = W.PagedInputs(inp.q, inp.k_cache, inp.v_cache * 0.25, inp.page_table, inp.seq_lens,
                        inp.scale)
    check(inp, "sigma 3 logits")


def test_decode_deterministic():
    inp = W.make_paged([3000, 41, 512], 32, 8, 128, 64, seed=730)
    o1, l1 = run_gpu(inp)
    o2, l2 = run_gpu(inp)
    assert np.array_equal(o1, o2) and np.array_equal(l1, l2)


def _raw(inp, **over):
    dev = torch.device("cuda")
    q, kc, vc, pt, sl = [t.to(dev) for t in (inp.q, inp.k_cache, inp.v_cache, inp.page_table,
                                             inp.seq_lens)]
    o = torch.zeros_like(q)
    lse = torch.zeros(tuple(q.shape[:2]), dtype=torch.float32, device=dev)
    B, Hq, D = q.shape
    npg, ps, Hkv, _ = kc.shape
    kw = dict(D=D, page_size=ps, Hq=Hq, Hkv=Hkv, ws=None, ws_bytes=0)
    kw.update(over)
    need = binding.mk_attn_decode_workspace_bytes(B, kw["Hq"], kw["Hkv"], kw["D"], kw["page_size"],
                                                  pt.shape[1])
    ws = torch.empty(max(need, 16) // 4 + 4, dtype=torch.float32, device=dev)
    ws_ptr = ws.data_ptr() if kw["ws"] is None else kw["ws"]
    ws_bytes = ws.numel() * 4 if kw["ws"] is None else kw["ws_bytes"]
    st = binding.mk_attn_decode_paged(q.data_ptr(), kc.data_ptr(), vc.data_ptr(), pt.data_ptr(),
                                      sl.data_ptr(), o.data_ptr(), lse.data_ptr(), B, kw["Hq"],
                                      kw["Hkv"], kw["D"], kw["page_size"], pt.shape[1], npg, 0.1,
                                      ws_ptr, ws_bytes, torch.cuda.current_stream().cuda_stream)
    return st, o, lse, need


def test_decode_rejected_calls_touch_nothing():
    inp = W.make_paged([100, 5], 8, 2, 128, 32, seed=740)
    for over, want in [(dict(D=96), binding.MK_ERR_UNSUPPORTED),
                       (dict(page_size=8), binding.MK_ERR_UNSUPPORTED),
                       (dict(Hq=7), binding.MK_ERR_INVALID_ARG)]:
        st, o, lse, _ = _raw(inp, **over)
        assert st == want, (over, st)
        torch.cuda.synchronize()
        assert torch.all(o == 0) and torch.all(lse == 0)
    st, o, lse, need = _raw(W.make_paged([4000], 8, 2, 128, 32, seed=741), ws=None)
    if need > 0:  # a split launch without its workspace is refused
        st, o, lse, _ = _raw(W.make_paged([4000], 8, 2, 128, 32, seed=741), ws=0, ws_bytes=0)
        assert st == binding.MK_ERR_INVALID_ARG


def test_decode_device_side_range_errors_are_reported():
    """Page indices or lengths out of range are only visible on the device:
    the launch goes through (no fault: the page is replaced) and the next
    status check reports MK_ERR_INVALID_ARG, then clears."""
    inp = W.make_paged([300, 20], 4, 4, 64, 32, seed=750)
    pt = inp.page_table.clone()
    pt[0, 3] = inp.k_cache.shape[0] + 5
    bad = W.PagedInputs(inp.q, inp.k_cache, inp.v_cache, pt, inp.seq_lens, inp.scale)
    dev = torch.device("cuda")
    args = [t.to(dev) for t in (bad.q, bad.k_cache, bad.v_cache, bad.page_table, bad.seq_lens)]
    binding.decode_paged(*args, scale=bad.scale)
    st = torch.cuda.current_stream().cuda_stream
    assert binding.mk_attn_check_status(st) == binding.MK_ERR_INVALID_ARG
    assert binding.mk_attn_check_status(st) == binding.MK_OK
    sl = inp.seq_lens.clone()
    sl[1] = inp.page_table.shape[1] * 32 + 1
    args[3] = inp.page_table.to(dev)
    args[4] = sl.to(dev)
    binding.decode_paged(*args, scale=bad.scale)
    assert binding.mk_attn_check_status(st) == binding.MK_ERR_INVALID_ARG
    check(inp, "after range errors")


def test_decode_bench_workload():
    """The bench workload (64 sequences of 1024-8192 cached tokens, Hq 32,
    Hkv 8, D 128, page 64, pages in random order), every output row against
    the oracle, in the launch configuration bench.py times."""
    lens = [int(x) for x in np.random.default_rng(2001).integers(1024, 8193, size=64)]
    inp = W.make_paged(lens, 32, 8, 128, 64, seed=2001, spare_pages=64)
    check(inp, "bench workload")
