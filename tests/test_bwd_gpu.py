"""Attention backward on the GPU against the fp64 oracle, through the C ABI.

The GPU forward pass produces o and lse; the GPU backward pass then gives
dq, dk, dv, which are compared element by element with the oracle's exact
gradients of the forward definition.  Tolerance, from a rounding model of the
kernel's arithmetic (P and dS rounded to bf16 as MMA operands, fp32
accumulation, Delta from the bf16 o, bf16 outputs), which predicts a relative
RMS error of about 2.4e-3 and a largest error of about 3.4e-3 of the largest
gradient at these sizes: for each of dq, dk, dv, relative RMS <= 5e-3 and
max |err| <= 1e-2 * max(max |ref|, 1e-3).  The floor covers gradients the
mathematics makes exactly zero (one key: dq = dk = 0), where the kernel's
Delta - dP cancellation leaves rounding residue near 1e-6."""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2609_04523_gb300 import binding
from paper_2609_04523_gb300 import workloads as W

pytestmark = pytest.mark.gpu

REL_RMS, MAX_REL = 5e-3, 1e-2
ABS_FLOOR = 1e-3  # max-abs bound at least 1e-5, for gradients that are exactly zero


def gpu_fwd_bwd(q, k, v, do, causal, scale, cu=None):
    dev = torch.device("cuda")
    qd, kd, vd, dod = (t.to(dev) for t in (q, k, v, do))
    cud = None if cu is None else cu.to(dev)
    o, lse = binding.attn_fwd(qd, kd, vd, causal=causal, scale=scale, cu_seqlens=cud)
    dq = torch.full_like(qd, float("nan"))
    dk = torch.full_like(kd, float("nan"))
    dv = torch.full_like(vd, float("nan"))
    binding.attn_bwd(qd, kd, vd, o, lse, dod, causal=causal, scale=scale, cu_seqlens=cud,
                     dq=dq, dk=dk, dv=dv)
    assert binding.mk_attn_check_status(torch.cuda.current_stream().cuda_stream) == binding.MK_OK
    return dq.float().cpu().numpy(), dk.float().cpu().numpy(), dv.float().cpu().numpy()


def compare(got, ref, what):
    ref = np.asarray(ref, dtype=np.float64)
    got = np.asarray(got, dtype=np.float64).reshape(ref.shape)
    assert np.all(np.isfinite(got)), f"{what}: non-finite (unwritten) entries"
    d = got - ref
    scale = max(float(np.max(np.abs(ref))), ABS_FLOOR)
    max_abs = float(np.max(np.abs(d)))
    assert max_abs <= MAX_REL * scale, f"{what}: max_abs {max_abs:.3e} (max ref {scale:.3e})"
    ref2 = float(np.sum(ref * ref))
    if ref2 > 0.0:  # a gradient the mathematics makes zero has no relative error
        rel = math.sqrt(float(np.sum(d * d)) / ref2)
        assert rel <= REL_RMS, f"{what}: rel_rms {rel:.3e}"


def check(q, k, v, do, causal, scale, cu=None, what=""):
    dq, dk, dv = gpu_fwd_bwd(q, k, v, do, causal, scale, cu)
    rq, rk, rv = oracle.attn_bwd(q, k, v, do, causal, scale,
                                 cu_seqlens=None if cu is None else cu.numpy())
    compare(dq, rq, f"{what} dq")
    compare(dk, rk, f"{what} dk")
    compare(dv, rv, f"{what} dv")


@pytest.mark.parametrize("D", [64, 128])
@pytest.mark.parametrize("causal", [True, False])
@pytest.mark.parametrize("S", [1, 100, 128, 300, 513])
def test_bwd_fixed_length(D, causal, S):
    """Single partial tile, exact tiles and ragged tails; GQA group of 3."""
    B, Hq, Hkv = 2, 6, 2
    q, k, v, _ = W.make_qkv(B, Hq, Hkv, S, D, seed=800 + S + D + int(causal))
    do = W.make_grad_out(q.shape, seed=800 + S + D)
    check(q, k, v, do, causal, 1.0 / math.sqrt(D), what=f"S{S} D{D} causal={causal}")


@pytest.mark.parametrize("G", [1, 4, 8, 16])
def test_bwd_group_sizes(G):
    q, k, v, _ = W.make_qkv(1, 2 * G, 2, 640, 128, seed=850 + G)
    do = W.make_grad_out(q.shape, seed=850 + G)
    check(q, k, v, do, True, 1.0 / math.sqrt(128), what=f"G{G}")


@pytest.mark.parametrize("causal", [True, False])
@pytest.mark.parametrize("D", [64, 128])
def test_bwd_varlen(causal, D):
    """Packed sequences, including lengths below one tile and of one token."""
    lens = [1, 130, 700, 5, 256, 383]
    q, k, v, cu = W.make_qkv(0, 8, 2, 0, D, seed=870 + D + int(causal), lengths=lens)
    do = W.make_grad_out(q.shape, seed=870 + D)
    check(q, k, v, do, causal, 1.0 / math.sqrt(D), cu=cu, what=f"varlen D{D} causal={causal}")


def test_bwd_varlen_more_sequences_than_one_warp_scan():
    """2100 packed sequences, empty ones among them: the backward kernels find a
    unit's sequence by warp scans over cu_seqlens in chunks of 32 sequences."""
    lens = W.many_short_lengths(2100, seed=92)
    q, k, v, cu = W.make_qkv(0, 4, 2, 0, 64, seed=92, lengths=lens)
    do = W.make_grad_out(q.shape, seed=92)
    check(q, k, v, do, True, 0.125, cu=cu, what="varlen 2100 sequences")


@pytest.mark.parametrize("causal", [True, False])
def test_bwd_stages_separately(causal):
    """mk_attn_bwd_stages: dQ alone (which writes Delta into the workspace),
    then dK/dV alone, equal the full call bit for bit; the stand-alone Delta
    kernel followed by dK/dV meets the oracle (its Delta sums in another order,
    so not bitwise).  Outputs of stages not enqueued stay untouched."""
    dev = torch.device("cuda")
    lens = [300, 1, 129, 700]
    q, k, v, cu = W.make_qkv(0, 8, 2, 0, 128, seed=893 + int(causal), lengths=lens)
    do = W.make_grad_out(q.shape, seed=893)
    qd, kd, vd, dod, cud = q.to(dev), k.to(dev), v.to(dev), do.to(dev), cu.to(dev)
    o, lse = binding.attn_fwd(qd, kd, vd, causal=causal, scale=0.09, cu_seqlens=cud)
    need = binding.mk_attn_bwd_workspace_bytes(len(lens), 8, q.shape[0], True)
    ws = torch.empty((need + 15) // 16 * 4, dtype=torch.float32, device=dev)

    def nan_outputs():
        return (torch.full_like(qd, float("nan")), torch.full_like(kd, float("nan")),
                torch.full_like(vd, float("nan")))

    def run(stages, outs):
        binding.attn_bwd(qd, kd, vd, o, lse, dod, causal=causal, scale=0.09, cu_seqlens=cud,
                         dq=outs[0], dk=outs[1], dv=outs[2], workspace=ws, stages=stages)
        assert binding.mk_attn_check_status(torch.cuda.current_stream().cuda_stream) == 0

    full = nan_outputs()
    run(binding.BWD_ALL, full)
    sep = nan_outputs()
    run(binding.BWD_DQ, sep)
    assert torch.isnan(sep[1].float()).all() and torch.isnan(sep[2].float()).all()
    assert torch.equal(sep[0], full[0])
    run(binding.BWD_DKDV, sep)
    assert torch.equal(sep[1], full[1]) and torch.equal(sep[2], full[2])

    ws.fill_(float("nan"))
    via_delta = nan_outputs()
    run(binding.BWD_DELTA, via_delta)
    assert all(torch.isnan(t.float()).all() for t in via_delta)
    run(binding.BWD_DKDV, via_delta)
    assert torch.isnan(via_delta[0].float()).all()
    _, rk, rv = oracle.attn_bwd(q, k, v, do, causal, 0.09, cu_seqlens=cu.numpy())
    compare(via_delta[1].float().cpu().numpy(), rk, "Delta kernel + dK/dV: dk")
    compare(via_delta[2].float().cpu().numpy(), rv, "Delta kernel + dK/dV: dv")


@pytest.mark.parametrize("scale", [-0.09, 0.0, 0.3])
def test_bwd_scales(scale):
    """Negative, zero and large scales (zero scale: dq = dk = 0)."""
    q, k, v, _ = W.make_qkv(1, 4, 4, 260, 64, seed=890)
    do = W.make_grad_out(q.shape, seed=890)
    if scale == 0.0:
        dq, dk, dv = gpu_fwd_bwd(q, k, v, do, True, 0.0)
        assert np.all(dq == 0.0) and np.all(dk == 0.0)
        _, _, rv = oracle.attn_bwd(q, k, v, do, True, 0.0)
        compare(dv, rv, "scale 0 dv")
        return
    check(q, k, v, do, True, scale, what=f"scale {scale}")


def test_bwd_deterministic():
    """No atomics: two calls give bitwise identical gradients."""
    q, k, v, _ = W.make_qkv(2, 8, 2, 777, 128, seed=900)
    do = W.make_grad_out(q.shape, seed=900)
    a = gpu_fwd_bwd(q, k, v, do, True, 0.088)
    b = gpu_fwd_bwd(q, k, v, do, True, 0.088)
    for x, y in zip(a, b):
        assert np.array_equal(x, y)


def test_bwd_causal_gqa_b4_s2048():
    """The bench workload (causal GQA B=4, Hq=32, Hkv=8, S=2048, D=128), every
    gradient element against the full oracle."""
    inp = W.make_config_inputs(2)
    do = W.make_grad_out(inp.q.shape, seed=inp.cfg.seed)
    check(inp.q, inp.k, inp.v, do, True, inp.cfg.scale, what="B4 S2048")


def test_bwd_causal_gqa_b1_s32768_sampled():
    """The long-context workload (causal GQA B=1, Hq=32, Hkv=8, S=32768,
    D=128, N(0, 0.5^2)) at full size: dq on sampled rows (a row's dq depends on
    that row only), dk / dv on the last key tile of every key/value head and on
    a range further back (the oracle visits every query row that sees them),
    and two identities over the whole tensors: sum_j dk_j = 0 (the rows of dS
    sum to zero) and sum_j dv_j = sum over the group's heads of sum_i dO_i."""
    inp = W.make_config_inputs(3)
    c = inp.cfg
    do = W.make_grad_out(inp.q.shape, seed=c.seed)
    dq, dk, dv = gpu_fwd_bwd(inp.q, inp.k, inp.v, do, True, c.scale)
    S, G = c.S, c.Hq // c.Hkv
    rows = [(0, h, i) for h in (0, 13, 31) for i in (0, 1, 127, 128, 4097, 20000, S - 129, S - 1)]
    ref = oracle.attn_bwd_dq_rows(inp.q, inp.k, inp.v, do, True, c.scale, rows)
    compare(np.stack([dq[0, i, h] for _, h, i in rows]), ref, "sampled dq rows")
    ranges = [(0, g, S - 128, S) for g in range(c.Hkv)] + [(0, 5, S - 1024, S - 1016)]
    rk, rv = oracle.attn_bwd_dkv_ranges(inp.q, inp.k, inp.v, do, True, c.scale, ranges)
    gk = np.concatenate([dk[0, j0:j1, g] for _, g, j0, j1 in ranges])
    gv = np.concatenate([dv[0, j0:j1, g] for _, g, j0, j1 in ranges])
    compare(gk, rk, "sampled dk ranges")
    compare(gv, rv, "sampled dv ranges")
    dof = do.double().numpy()[0]
    for g in range(c.Hkv):
        sk = dk[0, :, g].astype(np.float64).sum(axis=0)
        assert np.max(np.abs(sk)) <= 1e-2 * np.max(np.abs(dk[0, :, g])) * math.sqrt(S), "sum of dk"
        want = dof[:, g * G:(g + 1) * G].sum(axis=(0, 1))
        sv = dv[0, :, g].astype(np.float64).sum(axis=0)
        assert np.max(np.abs(sv - want)) <= 1e-2 * np.max(np.abs(want)), "sum of dv"
