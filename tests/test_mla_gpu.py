"""Latent (MLA) decode step on the GPU against the fp64 oracle, through the C
ABI.  Same bar as the other attention outputs: o max-abs <= 2e-2 and relative
RMS <= 5e-3, lse max-abs <= 1e-3; a sequence with no cached key gives o = 0
and lse = -inf exactly."""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2609_04523_gb300 import binding
from paper_2609_04523_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def check(inp, what):
    dev = torch.device("cuda")
    args = [t.to(dev) for t in (inp.q, inp.cache, inp.page_table, inp.seq_lens)]
    B, Hq, _ = inp.q.shape
    o = torch.full((B, Hq, binding.MLA_DV), float("nan"), dtype=torch.bfloat16, device=dev)
    lse = torch.full((B, Hq), float("nan"), dtype=torch.float32, device=dev)
    binding.mla_decode_paged(*args, scale=inp.scale, out=o, lse=lse)
    assert binding.mk_attn_check_status(torch.cuda.current_stream().cuda_stream) == binding.MK_OK
    o, lse = o.float().cpu().numpy(), lse.double().cpu().numpy()
    o_ref, lse_ref = oracle.mla_decode(inp.q, inp.cache, inp.page_table, inp.seq_lens, inp.scale,
                                       inp.dv)
    empty = np.asarray(inp.seq_lens) == 0
    assert np.all(o[empty] == 0.0) and np.all(np.isneginf(lse[empty])), f"{what}: empty rows"
    o, lse, o_ref, lse_ref = o[~empty], lse[~empty], o_ref[~empty], lse_ref[~empty]
    if o.size == 0:
        return
    assert np.all(np.isfinite(o)), f"{what}: unwritten outputs"
    d = o - o_ref
    max_abs = float(np.max(np.abs(d)))
    rel = math.sqrt(float(np.sum(d * d)) / float(np.sum(o_ref * o_ref)))
    lerr = float(np.max(np.abs(lse - lse_ref)))
    assert max_abs <= 2e-2, f"{what}: o max_abs {max_abs:.3e}"
    assert rel <= 5e-3, f"{what}: o rel_rms {rel:.3e}"
    assert lerr <= 1e-3, f"{what}: lse err {lerr:.3e}"


@pytest.mark.parametrize("page_size", [16, 32, 64, 128])
@pytest.mark.parametrize("Hq", [16, 128])
def test_mla_lengths(page_size, Hq):
    """Lengths around the 64-key block edges (half a page at page size 128),
    the page edges and an empty sequence."""
    lens = [0, 1, 63, 64, 65, 127, 128, 129, 191, 193, page_size + 3, 700, 2049]
    inp = W.make_mla_paged(lens, Hq, page_size, seed=960 + Hq + page_size)
    check(inp, f"ps{page_size} Hq{Hq}")


@pytest.mark.parametrize("Hq", [1, 129])
def test_mla_one_head_and_one_past_a_group(Hq):
    """One head (127 zero-filled rows of the M = 128 tile), and 129 heads (a
    second group holding a single head)."""
    inp = W.make_mla_paged([0, 1, 300, 1500], Hq, 64, seed=975 + Hq)
    check(inp, f"Hq{Hq}")


def test_mla_one_long_sequence():
    """One sequence of 65536 latent rows (1024 pages of 64), 128 heads: all the
    KV splits belong to it."""
    inp = W.make_mla_paged([65536], 128, 64, seed=977)
    check(inp, "L65536")


def test_mla_two_head_groups():
    """200 heads: a full group of 128 and a partial one of 72."""
    inp = W.make_mla_paged([300, 1500], 200, 64, seed=971)
    check(inp, "Hq200")


@pytest.mark.parametrize("B", [1, 4, 40])
def test_mla_splits(B):
    """Few sequences: many KV splits merged by log-sum-exp; many: one split."""
    rng = np.random.default_rng(980 + B)
    lens = [int(x) for x in rng.integers(1, 6000, size=B)]
    inp = W.make_mla_paged(lens, 32, 64, seed=980 + B)
    check(inp, f"B{B}")


def test_mla_many_sequences():
    """600 sequences of 0..299 latent rows (page 16, 16 heads): a grid of 600
    two-CTA clusters per split, empty sequences among them."""
    rng = np.random.default_rng(985)
    lens = [int(x) for x in rng.integers(0, 300, size=600)]
    inp = W.make_mla_paged(lens, 16, 16, seed=985)
    check(inp, "B600")


def test_mla_large_logits():
    """Row maxima that rise by far more than the lazy-rescale threshold
    between blocks (q and cache ~ N(0, 4))."""
    inp = W.make_mla_paged([900, 3000], 64, 64, seed=990, sigma=2.0)
    inp = W.MlaInputs(inp.q, inp.cache, inp.page_table, inp.seq_lens, inp.scale * 0.5, inp.dv)
    check(inp, "large logits")


def test_mla_rejects_bad_arguments():
    dev = torch.device("cuda")
    A = 1 << 20  # never dereferenced: every call below is rejected on the host
    good = dict(q=A, cache=A, page_table=A, seq_lens=A, o=A, lse=A, B=2, Hq=16, page_size=64,
                max_pages=4, num_pages=8, scale=0.04, workspace=None, workspace_bytes=0,
                stream=None)
    for kw, want in ((dict(q=None), binding.MK_ERR_INVALID_ARG),
                     (dict(page_size=48), binding.MK_ERR_UNSUPPORTED),
                     (dict(o=A + 8), binding.MK_ERR_ALIGNMENT),
                     (dict(scale=float("inf")), binding.MK_ERR_INVALID_ARG)):
        assert binding.mk_attn_mla_decode_paged(**{**good, **kw}) == want, kw
    del dev


def test_mla_bench_workload():
    """The bench workload (64 sequences of 1024-8192 cached tokens, 128 heads,
    page 64, pages in random order), every output row against the oracle, in
    the launch configuration bench.py times."""
    lens = [int(x) for x in np.random.default_rng(2001).integers(1024, 8193, size=64)]
    inp = W.make_mla_paged(lens, 128, 64, seed=2002, spare_pages=64)
    check(inp, "bench workload")


def test_mla_repeated_calls_are_bitwise_stable():
    """Back-to-back calls with KV splits (each a grid of two-CTA clusters that
    exchange partial scores through distributed shared memory) give the same
    bits every time and leave the status word clean: a race in the exchange
    or in the split merge would show up as a differing call."""
    dev = torch.device("cuda")
    inp = W.make_mla_paged([4000, 1, 0, 2500, 63, 65, 129], 128, 16, seed=993)
    args = [t.to(dev).contiguous() for t in (inp.q, inp.cache, inp.page_table, inp.seq_lens)]
    B, Hq, _ = inp.q.shape
    need = binding.mk_attn_mla_decode_workspace_bytes(B, Hq, inp.cache.shape[1], inp.page_table.shape[1])
    assert need > 0, "the case must use several KV splits"
    ws = torch.empty(need // 4 + 4, dtype=torch.float32, device=dev)
    o0 = torch.empty((B, Hq, binding.MLA_DV), dtype=torch.bfloat16, device=dev)
    l0 = torch.empty((B, Hq), dtype=torch.float32, device=dev)
    binding.mla_decode_paged(*args, scale=inp.scale, out=o0, lse=l0, workspace=ws)
    o = torch.empty_like(o0)
    l = torch.empty_like(l0)
    for _ in range(40):
        o.fill_(float("nan"))
        binding.mla_decode_paged(*args, scale=inp.scale, out=o, lse=l, workspace=ws)
        torch.cuda.synchronize()
        assert torch.equal(o.view(torch.int16), o0.view(torch.int16)) and torch.equal(l, l0)
    assert binding.mk_attn_check_status(torch.cuda.current_stream().cuda_stream) == binding.MK_OK
