"""CUDA path vs the fp64 oracle, element by element, through the C ABI (GPU).

Tolerances (bf16 output, fp32 LSE), over each whole output tensor:
  max |o_gpu - o_ref|                         <= 2e-2
  sqrt(sum (o_gpu - o_ref)^2 / sum o_ref^2)   <= 5e-3
  max |lse_gpu - lse_ref|                     <= 1e-3
The oracle is fp64 and unrounded; the kernel rounds P to bf16 (RNE) before
the P V contraction and o to bf16 at the end, which the bounds absorb.
"""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2609_04523_gb300 import binding
from paper_2609_04523_gb300 import workloads as W
from paper_2609_04523_gb300.build import build_library

pytestmark = pytest.mark.gpu

O_MAX_ABS = 2e-2
O_REL_RMS = 5e-3
LSE_MAX_ABS = 1e-3


@pytest.fixture(scope="module", autouse=True)
def cuda_lib():
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need a CUDA device")
    build_library()
    binding.load_library()


def gpu_attn(q, k, v, causal, scale, cu=None, prefill_nan=True):
    dev = torch.device("cuda")
    qd, kd, vd = q.to(dev), k.to(dev), v.to(dev)
    cud = cu.to(dev) if cu is not None else None
    o = torch.empty_like(qd)
    if cu is None:
        lse = torch.empty((q.shape[0], q.shape[2], q.shape[1]), dtype=torch.float32, device=dev)
    else:
        lse = torch.empty((q.shape[1], q.shape[0]), dtype=torch.float32, device=dev)
    if prefill_nan:
        o.fill_(float("nan"))
        lse.fill_(float("nan"))
    binding.attn_fwd(qd, kd, vd, causal, scale, cud, out=o, lse=lse)
    assert binding.mk_attn_check_status(torch.cuda.current_stream().cuda_stream) == 0
    return o.cpu(), lse.cpu()


def errors(o_gpu, lse_gpu, o_ref, lse_ref):
    og = o_gpu.to(torch.float64).numpy()
    lg = lse_gpu.to(torch.float64).numpy()
    assert np.all(np.isfinite(og)), "non-finite output (unwritten or overflowed row)"
    assert np.all(np.isfinite(lg)), "non-finite lse"
    d = og - o_ref
    max_abs = float(np.max(np.abs(d))) if d.size else 0.0
    denom = float(np.sum(o_ref * o_ref))
    rel_rms = math.sqrt(float(np.sum(d * d)) / denom) if denom > 0 else math.sqrt(float(np.sum(d * d)))
    lse_err = float(np.max(np.abs(lg - lse_ref))) if lg.size else 0.0
    return max_abs, rel_rms, lse_err


def assert_close(o_gpu, lse_gpu, o_ref, lse_ref, what=""):
    max_abs, rel_rms, lse_err = errors(o_gpu, lse_gpu, o_ref, lse_ref)
    assert max_abs <= O_MAX_ABS, f"{what}: max_abs {max_abs:.3e}"
    assert rel_rms <= O_REL_RMS, f"{what}: rel_rms {rel_rms:.3e}"
    assert lse_err <= LSE_MAX_ABS, f"{what}: lse err {lse_err:.3e}"


def check_fixed(B, Hq, Hkv, S, D, causal, seed, scale=None, sigma=1.0):
    q, k, v, _ = W.make_qkv(B, Hq, Hkv, S, D, seed=seed, sigma=sigma)
    scale = 1.0 / math.sqrt(D) if scale is None else scale
    o, lse = gpu_attn(q, k, v, causal, scale)
    o_ref, lse_ref = oracle.attn_fwd(q, k, v, causal, scale)
    assert_close(o, lse, o_ref, lse_ref, f"B{B} Hq{Hq} Hkv{Hkv} S{S} D{D} causal{causal}")


# ------------------------------------------------------------- shape sweep

@pytest.mark.parametrize("D", [64, 128])
@pytest.mark.parametrize("causal", [True, False])
@pytest.mark.parametrize("S", [1, 2, 127, 128, 129, 255, 384])
def test_tile_edges(D, causal, S):
    check_fixed(B=2, Hq=4, Hkv=2, S=S, D=D, causal=causal, seed=S * 7 + D + int(causal))


@pytest.mark.parametrize("D", [64, 128])
@pytest.mark.parametrize("G", [1, 2, 4, 8])
@pytest.mark.parametrize("B", [1, 3])
def test_gqa_groups(D, G, B):
    check_fixed(B=B, Hq=8, Hkv=8 // G, S=300, D=D, causal=True, seed=100 + G * 10 + B + D)


@pytest.mark.parametrize("causal", [True, False])
def test_mqa_one_kv_head_for_64_query_heads(causal):
    """Multi-query attention: G = 64, every query head reads key/value head 0."""
    check_fixed(B=1, Hq=64, Hkv=1, S=300, D=128, causal=causal, seed=170 + int(causal))


@pytest.mark.parametrize("causal", [True, False])
def test_gqa_odd_group(causal):
    """G = 3: units pair consecutive row tiles of one head (no head pairs)."""
    check_fixed(B=2, Hq=6, Hkv=2, S=700, D=128, causal=causal, seed=150 + int(causal))


@pytest.mark.parametrize("causal", [True, False])
def test_varlen_gqa_odd_group(causal):
    lens = [300, 129, 1, 640]
    q, k, v, cu = W.make_qkv(0, 6, 2, 0, 64, seed=160, lengths=lens)
    o, lse = gpu_attn(q, k, v, causal, 0.125, cu)
    o_ref, lse_ref = oracle.attn_fwd(q, k, v, causal, 0.125, cu_seqlens=cu.numpy())
    assert_close(o, lse, o_ref, lse_ref, "varlen G=3")


@pytest.mark.parametrize("D", [64, 128])
def test_long_noncausal(D):
    check_fixed(B=1, Hq=2, Hkv=1, S=1000, D=D, causal=False, seed=200 + D)


# ------------------------------------------------------------------ varlen

@pytest.mark.parametrize("D", [64, 128])
@pytest.mark.parametrize("causal", [True, False])
def test_varlen_edges(D, causal):
    lens = [1, 127, 128, 129, 700, 5]
    q, k, v, cu = W.make_qkv(0, 8, 2, 0, D, seed=300 + D, lengths=lens)
    scale = 1.0 / math.sqrt(D)
    o, lse = gpu_attn(q, k, v, causal, scale, cu)
    o_ref, lse_ref = oracle.attn_fwd(q, k, v, causal, scale, cu_seqlens=cu.numpy())
    assert_close(o, lse, o_ref, lse_ref, "varlen edges")


def test_varlen_random_lengths():
    lens = W.varlen_lengths(77, 6000, 1, 900)
    q, k, v, cu = W.make_qkv(0, 16, 4, 0, 128, seed=77, lengths=lens)
    o, lse = gpu_attn(q, k, v, True, 0.09, cu)
    o_ref, lse_ref = oracle.attn_fwd(q, k, v, True, 0.09, cu_seqlens=cu.numpy())
    assert_close(o, lse, o_ref, lse_ref, "varlen random")


def test_varlen_with_empty_sequences():
    lens = [0, 130, 0, 0, 64, 0]
    q, k, v, cu = W.make_qkv(0, 4, 4, 0, 64, seed=88, lengths=lens)
    o, lse = gpu_attn(q, k, v, True, 0.125, cu)
    o_ref, lse_ref = oracle.attn_fwd(q, k, v, True, 0.125, cu_seqlens=cu.numpy())
    assert_close(o, lse, o_ref, lse_ref, "varlen empty sequences")


@pytest.mark.parametrize("causal", [True, False])
def test_varlen_more_sequences_than_cu_cache(causal):
    """2100 packed sequences: the kernel caches cu_seqlens[0..2047] in shared
    memory and reads the entries past it from global memory.  Lengths 0..39,
    with a 300- and a 129-token sequence past the cache, so ragged tiles and
    empty sequences occur on both sides of it."""
    lens = W.many_short_lengths(2100, seed=91)
    q, k, v, cu = W.make_qkv(0, 4, 2, 0, 64, seed=91, lengths=lens)
    o, lse = gpu_attn(q, k, v, causal, 0.125, cu)
    o_ref, lse_ref = oracle.attn_fwd(q, k, v, causal, 0.125, cu_seqlens=cu.numpy())
    assert_close(o, lse, o_ref, lse_ref, "varlen 2100 sequences")


# ----------------------------------------------------------- special cases

def test_zero_scale_gives_prefix_means():
    q, k, v, _ = W.make_qkv(1, 2, 2, 200, 128, seed=400)
    o, lse = gpu_attn(q, k, v, True, 0.0)
    o_ref, lse_ref = oracle.attn_fwd(q, k, v, True, 0.0)
    assert_close(o, lse, o_ref, lse_ref, "scale 0")
    n = np.arange(1, 201)
    assert np.max(np.abs(lse[0, 0].double().numpy() - np.log(n))) <= LSE_MAX_ABS


@pytest.mark.parametrize("D", [64, 128])
@pytest.mark.parametrize("causal", [True, False])
def test_negative_scale(D, causal):
    """softmax(c q k^T) with c < 0: the row max of c s comes from the row's
    smallest score, and hidden keys must still get weight 0."""
    check_fixed(B=2, Hq=4, Hkv=2, S=300, D=D, causal=causal, seed=410 + D + int(causal),
                scale=-1.0 / math.sqrt(D))


def test_negative_scale_with_rescales():
    """A steep negative scale over 1000 keys: the running max rises by more
    than the lazy-rescale threshold many times along each row."""
    check_fixed(B=1, Hq=2, Hkv=1, S=1000, D=128, causal=False, seed=414, scale=-0.7)


def test_negative_zero_scale():
    q, k, v, _ = W.make_qkv(1, 2, 2, 200, 64, seed=412)
    o, lse = gpu_attn(q, k, v, True, -0.0)
    o_ref, lse_ref = oracle.attn_fwd(q, k, v, True, 0.0)
    assert_close(o, lse, o_ref, lse_ref, "scale -0")


def test_identical_keys():
    q, k, v, _ = W.make_qkv(1, 4, 1, 260, 64, seed=401)
    k = k[:, :1].expand_as(k).contiguous()
    o, lse = gpu_attn(q, k, v, True, 0.125)
    o_ref, lse_ref = oracle.attn_fwd(q, k, v, True, 0.125)
    assert_close(o, lse, o_ref, lse_ref, "identical keys")


@pytest.mark.parametrize("causal", [True, False])
def test_one_hot_values_expose_p(causal):
    """v_j = e_j with S <= D: o_i is the probability row i itself."""
    S, D = 128, 128
    q, k, _, _ = W.make_qkv(1, 2, 2, S, D, seed=402)
    v = torch.zeros(1, S, 2, D, dtype=torch.bfloat16)
    for j in range(S):
        v[:, j, :, j] = 1.0
    o, lse = gpu_attn(q, k, v, causal, 0.2)
    o_ref, lse_ref = oracle.attn_fwd(q, k, v, causal, 0.2)
    assert_close(o, lse, o_ref, lse_ref, "one-hot")
    if causal:
        P = o[0, :, 0].double().numpy()
        assert np.all(np.triu(P, 1) == 0.0), "probability on a hidden key"


def test_adversarial_rows():
    B, H, S, D = 2, 2, 512, 64
    scale = 0.125
    g = torch.Generator("cpu").manual_seed(403)
    q32 = torch.randn(B, S, H, D, generator=g)
    k32 = torch.randn(B, S, H, D, generator=g)
    v = torch.randn(B, S, H, D, generator=g).to(torch.bfloat16)
    planted = W.plant_adversarial_rows(q32, k32, scale, seed=403)
    q, k = q32.to(torch.bfloat16), k32.to(torch.bfloat16)
    o, lse = gpu_attn(q, k, v, False, scale)
    o_ref, lse_ref = oracle.attn_fwd(q, k, v, False, scale)
    assert_close(o, lse, o_ref, lse_ref, "adversarial")
    for (b, h, r, t) in planted:
        assert abs(float(lse[b, h, r]) - 30.0) <= 1e-2
        assert torch.max(torch.abs(o[b, r, h].float() - v[b, t, h].float())) <= 1e-2


def test_large_logits_do_not_overflow():
    """sigma = 4 and scale 1: logits reach the hundreds and rows are nearly
    one-hot, while |o| reaches about 16, where one bf16 ulp is 0.125.  The
    element bound is therefore taken relative to max |o_ref| (1e-2 of it, the
    2e-2 of unit-scale outputs at |o| <= 2); the relative RMS bound is the
    usual one, and the lse bound grows with |lse| (fp32)."""
    q, k, v, _ = W.make_qkv(1, 2, 2, 384, 128, seed=404, sigma=4.0)
    o, lse = gpu_attn(q, k, v, True, 1.0)
    o_ref, lse_ref = oracle.attn_fwd(q, k, v, True, 1.0)
    max_abs, rel_rms, lse_err = errors(o, lse, o_ref, lse_ref)
    o_scale = float(np.max(np.abs(o_ref)))
    assert o_scale > 4.0  # the case really has large outputs
    assert max_abs <= 1e-2 * o_scale, f"max_abs {max_abs:.3e} vs max|o_ref| {o_scale:.3e}"
    assert rel_rms <= O_REL_RMS, f"rel_rms {rel_rms:.3e}"
    assert lse_err <= 1e-4 * float(np.max(np.abs(lse_ref))) + 1e-3


# --------------------------------------------------------------- invariants

def test_gqa_equals_repeated_kv_bitwise():
    q, k, v, _ = W.make_qkv(2, 8, 2, 333, 128, seed=500)
    o1, l1 = gpu_attn(q, k, v, True, 0.1)
    o2, l2 = gpu_attn(q, k.repeat_interleave(4, dim=2), v.repeat_interleave(4, dim=2), True, 0.1)
    assert torch.equal(o1.view(torch.int16), o2.view(torch.int16))
    assert torch.equal(l1, l2)


def test_varlen_equals_separate_calls_bitwise():
    lens = [300, 1, 129, 256]
    q, k, v, cu = W.make_qkv(0, 4, 2, 0, 64, seed=501, lengths=lens)
    o, l = gpu_attn(q, k, v, True, 0.125, cu)
    for b, L in enumerate(lens):
        t0 = int(cu[b])
        sl = slice(t0, t0 + L)
        o1, l1 = gpu_attn(q[sl][None].contiguous(), k[sl][None].contiguous(),
                          v[sl][None].contiguous(), True, 0.125)
        assert torch.equal(o[sl].view(torch.int16), o1[0].view(torch.int16))
        assert torch.equal(l[:, sl], l1[0])


def test_deterministic():
    q, k, v, _ = W.make_qkv(2, 4, 4, 700, 128, seed=502)
    o1, l1 = gpu_attn(q, k, v, True, 0.08)
    o2, l2 = gpu_attn(q, k, v, True, 0.08)
    assert torch.equal(o1.view(torch.int16), o2.view(torch.int16)) and torch.equal(l1, l2)


def test_guard_regions_untouched():
    """Outputs carved out of larger buffers: nothing outside them is written."""
    dev = torch.device("cuda")
    B, S, Hq, Hkv, D = 2, 200, 4, 2, 64
    q, k, v, _ = W.make_qkv(B, Hq, Hkv, S, D, seed=503)
    pad = 4096
    n_o = B * S * Hq * D
    n_l = B * Hq * S
    ob = torch.full((n_o + 2 * pad,), 7.0, dtype=torch.bfloat16, device=dev)
    lb = torch.full((n_l + 2 * pad,), 7.0, dtype=torch.float32, device=dev)
    o = ob[pad:pad + n_o].view(B, S, Hq, D)
    lse = lb[pad:pad + n_l].view(B, Hq, S)
    binding.attn_fwd(q.to(dev), k.to(dev), v.to(dev), True, 0.125, None, out=o, lse=lse)
    torch.cuda.synchronize()
    assert torch.all(ob[:pad] == 7.0) and torch.all(ob[pad + n_o:] == 7.0)
    assert torch.all(lb[:pad] == 7.0) and torch.all(lb[pad + n_l:] == 7.0)
    o_ref, lse_ref = oracle.attn_fwd(q, k, v, True, 0.125)
    assert_close(o.cpu(), lse.cpu(), o_ref, lse_ref, "guarded")


@pytest.mark.parametrize("offset_bytes", [16, 32])
def test_output_pointer_alignment(offset_bytes):
    """o at a 16-byte (not 32-byte) and at a 32-byte aligned address: the
    epilogue switches between 16- and 32-byte stores; both must agree."""
    dev = torch.device("cuda")
    B, S, Hq, Hkv, D = 1, 260, 4, 2, 128
    q, k, v, _ = W.make_qkv(B, Hq, Hkv, S, D, seed=505)
    n_o = B * S * Hq * D
    base = torch.zeros(n_o + 64, dtype=torch.bfloat16, device=dev)
    assert base.data_ptr() % 256 == 0
    o = base[offset_bytes // 2: offset_bytes // 2 + n_o].view(B, S, Hq, D)
    lse = torch.empty((B, Hq, S), dtype=torch.float32, device=dev)
    binding.attn_fwd(q.to(dev), k.to(dev), v.to(dev), True, 0.1, None, out=o, lse=lse)
    assert binding.mk_attn_check_status(torch.cuda.current_stream().cuda_stream) == 0
    o_ref, lse_ref = oracle.attn_fwd(q, k, v, True, 0.1)
    assert_close(o.cpu(), lse.cpu(), o_ref, lse_ref, f"o offset {offset_bytes}")


def test_rejected_call_leaves_outputs_untouched():
    dev = torch.device("cuda")
    q, k, v, _ = W.make_qkv(1, 4, 2, 64, 64, seed=504)
    qd, kd, vd = q.to(dev), k.to(dev), v.to(dev)
    o = torch.full_like(qd, 3.0)
    lse = torch.full((1, 4, 64), 3.0, dtype=torch.float32, device=dev)
    st = binding.mk_attn_fwd(qd.data_ptr(), kd.data_ptr(), vd.data_ptr(), o.data_ptr(),
                             lse.data_ptr(), 1, 4, 3, 64, 64, 1, 0.1, None,
                             torch.cuda.current_stream().cuda_stream)
    assert st == binding.MK_ERR_INVALID_ARG
    torch.cuda.synchronize()
    assert torch.all(o == 3.0) and torch.all(lse == 3.0)


# ------------------------------------------------------- the five configs

def _config_parity(n, full: bool, n_rows: int = 4096):
    inp = W.make_config_inputs(n)
    c = inp.cfg
    cu = inp.cu_seqlens
    o, lse = gpu_attn(inp.q, inp.k, inp.v, c.causal, c.scale, cu)
    if full:
        o_ref, lse_ref = oracle.attn_fwd(inp.q, inp.k, inp.v, c.causal, c.scale,
                                         cu_seqlens=None if cu is None else cu.numpy())
        assert_close(o, lse, o_ref, lse_ref, c.name)
        return
    rows = W.sample_rows(inp.lengths, c.Hq, n_rows, seed=c.seed)
    # every row of the last query tile of every head is in the sample
    for b, L in enumerate(inp.lengths):
        last0 = ((L - 1) // W.TILE) * W.TILE
        in_last = rows[(rows[:, 0] == b) & (rows[:, 2] >= last0)]
        assert len({(int(h), int(i)) for _, h, i in in_last}) == c.Hq * (L - last0)
    o_ref, lse_ref = oracle.attn_rows(inp.q, inp.k, inp.v, c.causal, c.scale, rows,
                                      cu_seqlens=None if cu is None else cu.numpy())
    og = np.empty_like(o_ref)
    lg = np.empty_like(lse_ref)
    starts = np.cumsum([0] + list(inp.lengths))
    for n_, (b, h, i) in enumerate(rows):
        if cu is None:
            og[n_] = o[b, i, h].double().numpy()
            lg[n_] = float(lse[b, h, i])
        else:
            t = int(starts[b] + i)
            og[n_] = o[t, h].double().numpy()
            lg[n_] = float(lse[h, t])
    assert_close(torch.from_numpy(og), torch.from_numpy(lg), o_ref, lse_ref, c.name + " (rows)")
    assert torch.all(torch.isfinite(o.float())) and torch.all(torch.isfinite(lse))


def test_config1_full():
    _config_parity(1, full=True)


def test_config2_full():
    _config_parity(2, full=True)


def test_config3_sampled_rows():
    """S = 32768 (about 8.8 TFLOP in fp64, minutes of host time): the last
    query tile of all 32 heads (4096 rows that see 32641-32768 keys each),
    the first row, and 4095 uniform random rows."""
    _config_parity(3, full=False, n_rows=8192)


def test_config4_full():
    _config_parity(4, full=True)


def test_config5_full():
    """Every row of the varlen workload (about 1.5 TFLOP in fp64)."""
    _config_parity(5, full=True)


def test_varlen_causal_beyond_schedule_table():
    """One causal sequence with more than 1024 tile pairs (over 262144 tokens):
    the longest-first varlen schedule table covers up to 1024 pairs, so this
    launch is scheduled in sequence order.  Sampled rows against the oracle;
    every row written."""
    lens = [262144 + 300, 5, 1000]
    Hq = 2
    q, k, v, cu = W.make_qkv(0, Hq, 1, 0, 64, seed=520, lengths=lens)
    o, lse = gpu_attn(q, k, v, True, 0.125, cu)
    rows = W.sample_rows(lens, Hq, 256, seed=520)
    o_ref, lse_ref = oracle.attn_rows(q, k, v, True, 0.125, rows, cu_seqlens=cu.numpy())
    starts = np.cumsum([0] + lens)
    og = np.stack([o[int(starts[b] + i), h].double().numpy() for b, h, i in rows])
    lg = np.array([float(lse[h, int(starts[b] + i)]) for b, h, i in rows])
    assert_close(torch.from_numpy(og), torch.from_numpy(lg), o_ref, lse_ref, "varlen > 1024 pairs")
    assert torch.all(torch.isfinite(o.float())) and torch.all(torch.isfinite(lse))
