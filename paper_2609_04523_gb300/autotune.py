"""Config autotuner: a plain sweep over the library's launch knobs.

The paper's Autotuning Agent (Section 2.1) searches a kernel's configuration
space by timing candidates on the target hardware and keeping the fastest
correct one.  Here the search space is the runtime tuning of the C library
(mk_attn_tuning: persistent CTA count, unit schedule, the forward's lazy
rescale threshold, decode's KV-split plan); tile shapes and pipeline depths
are fixed at compile time by TMEM and shared-memory capacity.  Every
candidate runs the real kernels through the C ABI and is timed with CUDA
events on the launching stream, L2 flushed before each timed call; results
never differ beyond rounding between candidates (the GPU tests check parity
under each knob).

    python -m paper_2609_04523_gb300.autotune --workload prefill --config 2 --out sweep.json
"""
from __future__ import annotations

import argparse
import itertools
import json
import statistics

from . import binding
from . import workloads as W

FLUSH_BYTES = 256 << 20

# The default search space per workload: every combination is timed.
SPACES = {
    "prefill": dict(ctas=[0, 148, 144, 136, 128, 114, 76],
                    schedule=[binding.SCHED_SNAKE, binding.SCHED_ROUND_ROBIN,
                              binding.SCHED_BLOCKED, binding.SCHED_DYNAMIC],
                    rescale_log2=[0.0, 4.0, 8.0, 12.0]),
    "backward": dict(ctas=[0, 148, 136, 114],
                     schedule=[binding.SCHED_SNAKE, binding.SCHED_ROUND_ROBIN,
                               binding.SCHED_BLOCKED]),
    "decode": dict(split_ctas_per_sm=[3, 6, 12, 24, 48], split_min_pages=[1, 2, 4, 8, 16]),
    "mla": dict(mla_split_ctas_per_sm=[1, 2, 3, 4, 6, 8, 12, 16, 24]),
}


def candidates(space: dict):
    names = sorted(space)
    for values in itertools.product(*(space[n] for n in names)):
        yield dict(zip(names, values))


# GPU cycles of torch's bounded spin kernel before the timed calls: about 5 ms.
HEAD_START_CYCLES = 10_000_000


def time_call(fn, steps: int, warmup: int, flush, stream) -> float:
    """Mean CUDA-event time of fn() in ms, L2 flushed before each call.  All
    calls are enqueued behind a short GPU spin and synchronised once, so the
    host stays ahead and no call's events include GPU idle time."""
    import torch
    for _ in range(warmup):
        flush.zero_()
        fn()
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    torch.cuda.synchronize()
    torch.cuda._sleep(HEAD_START_CYCLES)
    for a, b in zip(starts, ends):
        flush.zero_()
        a.record(stream)
        fn()
        b.record(stream)
    torch.cuda.synchronize()
    return statistics.mean(a.elapsed_time(b) for a, b in zip(starts, ends))


def make_step(workload: str, config: int, dev):
    """Returns (step, work, unit): one call of the workload on resident
    inputs and its work per call (FLOPs, or bytes for decode)."""
    import numpy as np
    import torch
    if workload == "mla":
        lens = [int(x) for x in np.random.default_rng(2001).integers(1024, 8193, size=64)]
        inp = W.make_mla_paged(lens, 128, 64, seed=2002, spare_pages=64)
        args = [t.to(dev) for t in (inp.q, inp.cache, inp.page_table, inp.seq_lens)]

        def step():  # the workspace follows the current split plan
            binding.mla_decode_paged(*args, scale=inp.scale)
        return step, W.mla_decode_bytes(lens, 128), "GB/s"
    if workload == "decode":
        lens = [int(x) for x in np.random.default_rng(2001).integers(1024, 8193, size=64)]
        inp = W.make_paged(lens, 32, 8, 128, 64, seed=2001, spare_pages=64)
        args = [t.to(dev) for t in (inp.q, inp.k_cache, inp.v_cache, inp.page_table,
                                    inp.seq_lens)]
        o = torch.empty_like(args[0])
        lse = torch.empty(tuple(inp.q.shape[:2]), dtype=torch.float32, device=dev)

        def step():  # the workspace follows the current split plan
            binding.decode_paged(*args, scale=inp.scale, out=o, lse=lse)
        return step, W.decode_bytes(lens, 32, 8, 128), "GB/s"
    inp = W.make_config_inputs(config)
    c = inp.cfg
    q, k, v = inp.q.to(dev), inp.k.to(dev), inp.v.to(dev)
    cu = None if inp.cu_seqlens is None else inp.cu_seqlens.to(dev)
    flops = W.attn_flops(inp.lengths, c.Hq, c.D, c.causal)
    o, lse = binding.attn_fwd(q, k, v, c.causal, c.scale, cu)
    if workload == "prefill":
        def step():
            binding.attn_fwd(q, k, v, c.causal, c.scale, cu, out=o, lse=lse)
        return step, flops, "TFLOP/s"
    do = W.make_grad_out(q.shape, seed=c.seed).to(dev)
    dq, dk, dv = torch.empty_like(q), torch.empty_like(k), torch.empty_like(v)

    def step():
        binding.attn_bwd(q, k, v, o, lse, do, c.causal, c.scale, cu, dq=dq, dk=dk, dv=dv)
    return step, 2.5 * flops, "TFLOP/s"


def sweep(workload: str = "prefill", config: int = 2, space: dict | None = None,
          steps: int = 10, warmup: int = 3):
    """Times every candidate of `space` (default SPACES[workload]); returns the
    rows sorted fastest first.  The process-wide tuning is restored after."""
    import torch
    dev = torch.device("cuda")
    stream = torch.cuda.current_stream(dev)
    flush = torch.empty(FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    step, work, unit = make_step(workload, config, dev)
    scale = 1e12 if unit == "TFLOP/s" else 1e9
    rows = []
    for cand in candidates(space or SPACES[workload]):
        with binding.tuning(**cand):
            ms = time_call(step, steps, warmup, flush, stream)
            st = binding.mk_attn_check_status(stream.cuda_stream)
        if st != binding.MK_OK:
            raise RuntimeError(f"kernel status {st} under {cand}")
        rows.append({**cand, "ms": ms, "value": work / (ms * 1e-3) / scale, "unit": unit})
    rows.sort(key=lambda r: r["ms"])
    return rows


def main():
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    ap.add_argument("--workload", default="prefill", choices=sorted(SPACES))
    ap.add_argument("--config", type=int, default=2)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--out", default=None)
    args = ap.parse_args()
    rows = sweep(args.workload, args.config, steps=args.steps)
    default = next((r for r in rows if all(r.get(k) == v for k, v in binding.DEFAULT_TUNING.items()
                                            if k in r)), None)
    out = {"workload": args.workload, "config": args.config, "best": rows[0], "default": default,
           "rows": rows}
    text = json.dumps(out, indent=1)
    if args.out:
        with open(args.out, "w") as f:
            f.write(text)
    print(json.dumps({"best": rows[0], "default": default}))


if __name__ == "__main__":
    main()
