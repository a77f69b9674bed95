"""Entry points captured in a CUDA graph and replayed.

Serving stacks capture decode (and often prefill) steps in CUDA graphs.  Each
test runs a call eagerly, captures the same call (same buffers) with
torch.cuda.graph, poisons the outputs, replays the graph twice and requires
the replayed outputs to equal the eager ones bit for bit.  The decode and
latent decode calls use several KV splits, so the captured graph holds the
merge kernel's dependent launch as well."""
import pytest
import torch

from paper_2609_04523_gb300 import binding
from paper_2609_04523_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def _capture_and_replay(fn, outs):
    """fn() enqueues the call on the current stream and writes `outs`."""
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        fn()  # warm-up outside the capture (first-call set-up happens here)
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    ref = [t.clone() for t in outs]
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        fn()
    for _ in range(2):
        for t in outs:
            t.fill_(float("nan"))
        graph.replay()
        torch.cuda.synchronize()
        for t, r in zip(outs, ref):
            assert torch.equal(t, r), "replayed output differs from the eager one"
    assert binding.mk_attn_check_status(torch.cuda.current_stream().cuda_stream) == binding.MK_OK


def test_forward_captured():
    dev = torch.device("cuda")
    q, k, v, cu = W.make_qkv(0, 8, 2, 0, 128, seed=941, lengths=[700, 1, 333, 1500])
    q, k, v, cu = q.to(dev), k.to(dev), v.to(dev), cu.to(dev)
    o = torch.empty_like(q)
    lse = torch.empty((8, q.shape[0]), dtype=torch.float32, device=dev)
    _capture_and_replay(
        lambda: binding.attn_fwd(q, k, v, causal=True, scale=0.088, cu_seqlens=cu, out=o, lse=lse),
        [o, lse])


def test_backward_captured():
    dev = torch.device("cuda")
    q, k, v, _ = W.make_qkv(2, 8, 4, 640, 128, seed=942)
    q, k, v = q.to(dev), k.to(dev), v.to(dev)
    do = W.make_grad_out(q.shape, seed=942).to(dev)
    o, lse = binding.attn_fwd(q, k, v, causal=True, scale=0.088)
    dq, dk, dv = torch.empty_like(q), torch.empty_like(k), torch.empty_like(v)
    need = binding.mk_attn_bwd_workspace_bytes(2, 8, 640, False)
    ws = torch.empty(need // 4 + 4, dtype=torch.float32, device=dev)
    _capture_and_replay(
        lambda: binding.attn_bwd(q, k, v, o, lse, do, causal=True, scale=0.088,
                                 dq=dq, dk=dk, dv=dv, workspace=ws),
        [dq, dk, dv])


def test_decode_with_splits_captured():
    dev = torch.device("cuda")
    inp = W.make_paged([5000, 3, 2600, 0, 1200], 16, 4, 128, 64, seed=943)
    args = [t.to(dev).contiguous() for t in (inp.q, inp.k_cache, inp.v_cache, inp.page_table,
                                            inp.seq_lens)]
    B, Hq, D = inp.q.shape
    _, ps, Hkv, _ = inp.k_cache.shape
    need = binding.mk_attn_decode_workspace_bytes(B, Hq, Hkv, D, ps, inp.page_table.shape[1])
    assert need > 0, "the case must use several KV splits"
    ws = torch.empty(need // 4 + 4, dtype=torch.float32, device=dev)
    o = torch.empty_like(args[0])
    lse = torch.empty((B, Hq), dtype=torch.float32, device=dev)
    _capture_and_replay(
        lambda: binding.decode_paged(*args, scale=inp.scale, out=o, lse=lse, workspace=ws),
        [o, lse])


def test_latent_decode_with_splits_captured():
    dev = torch.device("cuda")
    inp = W.make_mla_paged([4000, 1, 0, 2500], 16, 64, seed=944)
    args = [t.to(dev).contiguous() for t in (inp.q, inp.cache, inp.page_table, inp.seq_lens)]
    B, Hq, _ = inp.q.shape
    need = binding.mk_attn_mla_decode_workspace_bytes(B, Hq, inp.cache.shape[1],
                                                      inp.page_table.shape[1])
    assert need > 0, "the case must use several KV splits"
    ws = torch.empty(need // 4 + 4, dtype=torch.float32, device=dev)
    o = torch.empty((B, Hq, 512), dtype=torch.bfloat16, device=dev)
    lse = torch.empty((B, Hq), dtype=torch.float32, device=dev)
    _capture_and_replay(
        lambda: binding.mla_decode_paged(*args, scale=inp.scale, out=o, lse=lse, workspace=ws),
        [o, lse])
