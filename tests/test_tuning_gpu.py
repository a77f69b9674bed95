"""Every launch knob of the autotuner keeps the results: the forward, backward
and decode kernels under non-default tunings, against the fp64 oracle (the
parity tolerances of their own tests) and, where a knob cannot change any
arithmetic (CTA count, unit schedule), bitwise against the default tuning."""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2609_04523_gb300 import autotune, binding
from paper_2609_04523_gb300 import workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def restore():
    yield
    binding.set_tuning()


def fwd(q, k, v, causal, scale, cu=None):
    dev = torch.device("cuda")
    o, lse = binding.attn_fwd(q.to(dev), k.to(dev), v.to(dev), causal=causal, scale=scale,
                              cu_seqlens=None if cu is None else cu.to(dev))
    assert binding.mk_attn_check_status(torch.cuda.current_stream().cuda_stream) == binding.MK_OK
    return o.float().cpu().numpy(), lse.double().cpu().numpy()


def check_fwd(o, lse, o_ref, lse_ref):
    d = o - o_ref
    assert float(np.max(np.abs(d))) <= 2e-2
    assert math.sqrt(float(np.sum(d * d)) / float(np.sum(o_ref * o_ref))) <= 5e-3
    assert float(np.max(np.abs(lse - lse_ref))) <= 1e-3


KNOBS = [dict(ctas=1), dict(ctas=37), dict(ctas=300), dict(schedule=binding.SCHED_SNAKE),
         dict(schedule=binding.SCHED_ROUND_ROBIN),
         dict(schedule=binding.SCHED_BLOCKED), dict(ctas=64, schedule=binding.SCHED_BLOCKED),
         dict(schedule=binding.SCHED_DYNAMIC), dict(ctas=1, schedule=binding.SCHED_DYNAMIC),
         dict(ctas=37, schedule=binding.SCHED_DYNAMIC)]


@pytest.mark.parametrize("knob", KNOBS, ids=lambda d: "-".join(f"{k}{v}" for k, v in d.items()))
def test_forward_and_backward_bitwise_under_schedule_knobs(knob):
    """Each unit is computed whole by one CTA, so the CTA count and the
    schedule decide only where a unit runs: outputs are bitwise equal."""
    lens = [300, 1, 900, 129]
    q, k, v, cu = W.make_qkv(0, 8, 2, 0, 128, seed=931, lengths=lens)
    do = W.make_grad_out(q.shape, seed=931)
    dev = torch.device("cuda")
    args = [t.to(dev) for t in (q, k, v, do)]
    cud = cu.to(dev)

    def run():
        o, lse = binding.attn_fwd(*args[:3], causal=True, scale=0.09, cu_seqlens=cud)
        g = binding.attn_bwd(*args[:3], o, lse, args[3], causal=True, scale=0.09, cu_seqlens=cud)
        assert binding.mk_attn_check_status(torch.cuda.current_stream().cuda_stream) == 0
        return [t.cpu() for t in (o, lse, *g)]

    base = run()
    with binding.tuning(**knob):
        got = run()
    for a, b in zip(base, got):
        assert torch.equal(a, b)


def errors(o, lse, o_ref, lse_ref):
    d = o - o_ref
    return (float(np.max(np.abs(d))), math.sqrt(float(np.sum(d * d)) / float(np.sum(o_ref * o_ref))),
            float(np.max(np.abs(lse - lse_ref))))


@pytest.mark.parametrize("tau", [0.0, 1.0, 16.0])
def test_forward_rescale_threshold(tau):
    """The lazy rescale is exact in real arithmetic for every threshold; in
    the kernel a larger threshold lets P span up to 2^tau within one tile
    before its MMA, and the largest error grows with it (on these inputs
    0.015 at the default 8, 0.025 at 16).  On rows with large, often-rising
    logits (q, k ~ N(0, 4), scale 0.3: nearly one-hot softmax rows, where
    bf16 rounding of the dominant weight and of o alone reaches about 2e-2):
    relative RMS <= 5e-3, lse <= 1e-3 and max |err| <= max(2e-2, 2x the
    default's).  Config 1 keeps the plain tolerance."""
    B, Hq, Hkv, S, D = 2, 4, 2, 700, 64
    q, k, _, _ = W.make_qkv(B, Hq, Hkv, S, D, seed=940, sigma=2.0)
    v = W.make_qkv(B, Hq, Hkv, S, D, seed=941)[2]
    for causal in (True, False):
        ref = oracle.attn_fwd(q, k, v, causal, 0.3)
        base = errors(*fwd(q, k, v, causal, 0.3), *ref)
        with binding.tuning(rescale_log2=tau):
            got = errors(*fwd(q, k, v, causal, 0.3), *ref)
        assert got[1] <= 5e-3 and got[2] <= 1e-3, (tau, causal, got)
        assert got[0] <= max(2e-2, 2.0 * base[0]), (tau, causal, got, base)
    inp = W.make_config_inputs(1)
    with binding.tuning(rescale_log2=tau):
        o, lse = fwd(inp.q, inp.k, inp.v, True, inp.cfg.scale)
    check_fwd(o, lse, *oracle.attn_fwd(inp.q, inp.k, inp.v, True, inp.cfg.scale))


@pytest.mark.parametrize("plan", [dict(split_ctas_per_sm=1, split_min_pages=1),
                                  dict(split_ctas_per_sm=64, split_min_pages=1),
                                  dict(split_ctas_per_sm=12, split_min_pages=4096)])
def test_decode_split_plans(plan):
    """Decode under other KV-split plans (one split, many short splits):
    parity with the oracle."""
    lens = [5000, 1, 0, 2100, 64]
    inp = W.make_paged(lens, 16, 4, 128, 64, seed=950)
    dev = torch.device("cuda")
    args = [t.to(dev) for t in (inp.q, inp.k_cache, inp.v_cache, inp.page_table, inp.seq_lens)]
    with binding.tuning(**plan):
        o, lse = binding.decode_paged(*args, scale=inp.scale)
        assert binding.mk_attn_check_status(torch.cuda.current_stream().cuda_stream) == 0
    o_ref, lse_ref = oracle.decode_paged(inp.q, inp.k_cache, inp.v_cache, inp.page_table,
                                         inp.seq_lens, inp.scale)
    o, lse = o.float().cpu().numpy(), lse.double().cpu().numpy()
    live = np.asarray(lens) > 0
    assert np.all(o[~live] == 0) and np.all(np.isneginf(lse[~live]))
    d = o[live] - o_ref[live]
    assert float(np.max(np.abs(d))) <= 2e-2
    assert float(np.max(np.abs(lse[live] - lse_ref[live]))) <= 1e-3


@pytest.mark.parametrize("waves", [1, 24])
def test_mla_split_plans(waves):
    """The latent decode step under one and many KV splits: parity."""
    inp = W.make_mla_paged([3000, 1, 0, 700], 64, 64, seed=955)
    dev = torch.device("cuda")
    args = [t.to(dev) for t in (inp.q, inp.cache, inp.page_table, inp.seq_lens)]
    with binding.tuning(mla_split_ctas_per_sm=waves):
        o, lse = binding.mla_decode_paged(*args, scale=inp.scale)
        assert binding.mk_attn_check_status(torch.cuda.current_stream().cuda_stream) == 0
    o_ref, lse_ref = oracle.mla_decode(inp.q, inp.cache, inp.page_table, inp.seq_lens, inp.scale,
                                       inp.dv)
    o, lse = o.float().cpu().numpy(), lse.double().cpu().numpy()
    live = np.asarray(inp.seq_lens) > 0
    assert np.all(o[~live] == 0) and np.all(np.isneginf(lse[~live]))
    d = o[live] - o_ref[live]
    assert float(np.max(np.abs(d))) <= 2e-2
    assert float(np.max(np.abs(lse[live] - lse_ref[live]))) <= 1e-3


def test_sweep_returns_sorted_rows_and_restores_tuning():
    binding.set_tuning(ctas=99)
    rows = autotune.sweep("prefill", 1, space={"ctas": [0, 2], "schedule": [0, 2]}, steps=2,
                          warmup=1)
    assert len(rows) == 4 and all(r["ms"] > 0 for r in rows)
    assert rows == sorted(rows, key=lambda r: r["ms"])
    assert binding.mk_attn_get_tuning().ctas == 99


def test_dynamic_schedule_counters_reset_over_many_launches_and_two_streams():
    """MK_SCHED_DYNAMIC claims units from per-launch device counters that each
    launch's last CTA zeroes.  1100 launches wrap the 1024-slot ring, so every
    slot is reused; launches alternate between two streams so that some run at
    once.  Every output must equal the snake schedule's bit for bit (a counter
    left non-zero would skip units)."""
    dev = torch.device("cuda")
    q, k, v, _ = W.make_qkv(1, 4, 2, 2048, 64, seed=932)
    q, k, v = q.to(dev), k.to(dev), v.to(dev)
    with binding.tuning(schedule=binding.SCHED_SNAKE):
        o_ref, lse_ref = binding.attn_fwd(q, k, v, causal=True, scale=0.125)
    streams = [torch.cuda.Stream(), torch.cuda.Stream()]
    for st in streams:
        st.wait_stream(torch.cuda.current_stream())
    outs = []
    with binding.tuning(ctas=5, schedule=binding.SCHED_DYNAMIC):
        for i in range(1100):
            st = streams[i % 2]
            with torch.cuda.stream(st):
                o = torch.empty_like(q)
                lse = torch.empty((1, 4, 2048), dtype=torch.float32, device=dev)
                binding.attn_fwd(q, k, v, causal=True, scale=0.125, out=o, lse=lse, stream=st)
            if i % 50 == 0 or i >= 1090:
                outs.append((st, o, lse))
        torch.cuda.synchronize()
    assert binding.mk_attn_check_status(torch.cuda.current_stream().cuda_stream) == 0
    for _, o, lse in outs:
        assert torch.equal(o, o_ref) and torch.equal(lse, lse_ref)
