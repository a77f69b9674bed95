"""One call of every kernel family through the binding, each checked against
the fp64 oracle; run by tests/test_check_mode_gpu.py in a child process whose
environment selects the check mode (MK_ATTN_DEBUG) and/or the check build
(MK_ATTN_CHECK_BUILD), both of which are read once per process.

Every entry point must return MK_OK (under MK_ATTN_DEBUG that is the device
status after a synchronisation), and every result must meet the parity
tolerances.  Prints the loaded library and "check mode run: ok"."""
import math
import os
import sys

import numpy as np
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import oracle  # noqa: E402
from paper_2609_04523_gb300 import binding  # noqa: E402
from paper_2609_04523_gb300 import workloads as W  # noqa: E402


def close(what, got, ref, max_abs, rel_rms=5e-3):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    d = got - ref
    ma = float(np.max(np.abs(d)))
    rr = math.sqrt(float(np.sum(d * d)) / max(float(np.sum(ref * ref)), 1e-300))
    if not (ma <= max_abs and rr <= rel_rms):
        raise SystemExit(f"{what}: max_abs {ma:.3e} rel_rms {rr:.3e}")


def main():
    dev = torch.device("cuda")
    lib = binding.load_library()
    print("library:", os.path.basename(binding.library_path()))
    stream = torch.cuda.current_stream().cuda_stream

    # forward, fixed length and varlen, and the backward pass
    q, k, v, _ = W.make_qkv(2, 8, 2, 300, 128, seed=61)
    do = W.make_grad_out(q.shape, seed=61)
    o, lse = binding.attn_fwd(q.to(dev), k.to(dev), v.to(dev), True, 0.09)
    o_ref, lse_ref = oracle.attn_fwd(q, k, v, True, 0.09)
    close("fwd o", o.cpu().float(), o_ref, 2e-2)
    close("fwd lse", lse.cpu().double(), lse_ref, 1e-3, 1.0)
    dq, dk, dv = binding.attn_bwd(q.to(dev), k.to(dev), v.to(dev), o, lse, do.to(dev),
                                  True, 0.09)
    for name, got, ref in zip(("dq", "dk", "dv"), (dq, dk, dv),
                              oracle.attn_bwd(q, k, v, do, True, 0.09)):
        close("bwd " + name, got.cpu().float(), ref, 1e-2 * max(float(np.max(np.abs(ref))), 1e-3))
    lens = [300, 1, 129, 0, 640]
    q, k, v, cu = W.make_qkv(0, 4, 2, 0, 64, seed=62, lengths=lens)
    o, lse = binding.attn_fwd(q.to(dev), k.to(dev), v.to(dev), True, 0.125, cu.to(dev))
    o_ref, lse_ref = oracle.attn_fwd(q, k, v, True, 0.125, cu_seqlens=cu.numpy())
    close("varlen fwd o", o.cpu().float(), o_ref, 2e-2)

    # paged decode, with a workspace and without
    inp = W.make_paged([0, 70, 1500, 3000], 8, 2, 128, 64, seed=63)
    args = [t.to(dev) for t in (inp.q, inp.k_cache, inp.v_cache, inp.page_table, inp.seq_lens)]
    o, lse = binding.decode_paged(*args, scale=inp.scale)
    o_ref, lse_ref = oracle.decode_paged(inp.q, inp.k_cache, inp.v_cache, inp.page_table,
                                         inp.seq_lens, inp.scale)
    close("decode o", o.cpu().float()[1:], o_ref[1:], 2e-2)
    B, Hq, D = inp.q.shape
    npg, ps, Hkv, _ = inp.k_cache.shape
    o2 = torch.empty_like(o)
    l2 = torch.empty_like(lse)
    st = binding.mk_attn_decode_paged_noalloc(
        args[0].data_ptr(), args[1].data_ptr(), args[2].data_ptr(), args[3].data_ptr(),
        args[4].data_ptr(), o2.data_ptr(), l2.data_ptr(), B, Hq, Hkv, D, ps,
        inp.page_table.shape[1], npg, inp.scale, stream)
    if st != binding.MK_OK:
        raise SystemExit(f"noalloc decode: status {st}")
    close("noalloc decode o", o2.cpu().float()[1:], o_ref[1:], 2e-2)

    # latent (MLA) decode
    mi = W.make_mla_paged([0, 200, 900], 16, 64, seed=64)
    margs = [t.to(dev) for t in (mi.q, mi.cache, mi.page_table, mi.seq_lens)]
    o, lse = binding.mla_decode_paged(*margs, scale=mi.scale)
    o_ref, _ = oracle.mla_decode(mi.q, mi.cache, mi.page_table, mi.seq_lens, mi.scale, mi.dv)
    close("mla o", o.cpu().float()[1:], o_ref[1:], 2e-2)

    torch.cuda.synchronize()
    st = binding.mk_attn_check_status(stream)
    if st != binding.MK_OK:
        raise SystemExit(f"final status {st}")
    del lib
    print("check mode run: ok")


if __name__ == "__main__":
    main()
