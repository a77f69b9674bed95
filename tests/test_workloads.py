"""The seeded input generators (no GPU)."""
import numpy as np
import torch

from paper_2609_04523_gb300 import workloads as W


def test_make_qkv_is_deterministic():
    a = W.make_qkv(2, 4, 2, 33, 16, seed=7)
    b = W.make_qkv(2, 4, 2, 33, 16, seed=7)
    for x, y in zip(a[:3], b[:3]):
        assert x.dtype == torch.bfloat16
        assert torch.equal(x.view(torch.int16), y.view(torch.int16))
    c = W.make_qkv(2, 4, 2, 33, 16, seed=8)
    assert not torch.equal(a[0], c[0])


def test_shapes_fixed_and_varlen():
    q, k, v, cu = W.make_qkv(3, 8, 2, 40, 64, seed=1)
    assert q.shape == (3, 40, 8, 64) and k.shape == (3, 40, 2, 64) and cu is None
    q, k, v, cu = W.make_qkv(0, 8, 2, 0, 64, seed=1, lengths=[5, 9])
    assert q.shape == (14, 8, 64) and v.shape == (14, 2, 64)
    assert cu.dtype == torch.int32 and cu.tolist() == [0, 5, 14]


def test_varlen_lengths_recipe():
    lens = W.varlen_lengths(1005, 32768)
    assert sum(lens) == 32768
    assert all(512 <= L <= 4096 for L in lens[:-1])
    assert 1 <= lens[-1] <= 4096
    assert lens == W.varlen_lengths(1005, 32768)


def test_config_table():
    assert [c.index for c in W.CONFIGS] == [1, 2, 3, 4, 5]
    c2 = W.config(2)
    assert (c2.B, c2.Hq, c2.Hkv, c2.S, c2.D, c2.causal) == (4, 32, 8, 2048, 128, True)
    assert abs(W.config(1).scale - 0.125) < 1e-15


def test_config1_inputs_and_flops():
    inp = W.make_config_inputs(1)
    assert inp.q.shape == (1, 128, 2, 64)
    assert W.attn_flops([128], 2, 64, True) == 4 * 2 * 64 * 128 * 128 / 2
    assert W.attn_flops([2048] * 4, 32, 128, True) == 137438953472.0
    assert W.attn_pairs([3], 1, True) == 6 and W.attn_pairs([3], 2, False) == 18


def test_adversarial_rows_have_the_stated_gap():
    """Config 4's recipe on a reduced shape: the planted logit is exactly 30
    and at least 29.5 above every other logit of its row."""
    g = torch.Generator("cpu").manual_seed(3)
    B, S, H, D = 2, 1024, 2, 64
    scale = 1 / 8
    q32 = torch.randn(B, S, H, D, generator=g)
    k32 = torch.randn(B, S, H, D, generator=g)
    planted = W.plant_adversarial_rows(q32, k32, scale, seed=3)
    assert len(planted) == B * H * 4
    q = q32.to(torch.bfloat16).double()
    k = k32.to(torch.bfloat16).double()
    for (b, h, r, t) in planted:
        s = scale * (k[b, :, h] @ q[b, r, h])
        assert float(s[t]) == 30.0
        others = torch.cat([s[:t], s[t + 1:]])
        assert 30.0 - float(others.max()) >= 29.5


def test_sample_rows_cover_last_tiles():
    lens = [300, 129, 7]
    rows = W.sample_rows(lens, 4, 50, seed=0)
    assert rows.shape[1] == 3 and len(rows) >= 50
    for b, L in enumerate(lens):
        last0 = ((L - 1) // 128) * 128
        got = {int(i) for (bb, h, i) in rows if bb == b}
        assert set(range(last0, L)) <= got
        assert all(0 <= i < L for (bb, h, i) in rows if bb == b)


def test_many_short_lengths():
    """Seeded, 0..39 with empty sequences among them, 300 at n - 50 and 129 last."""
    a = W.many_short_lengths(2100, seed=91)
    assert a == W.many_short_lengths(2100, seed=91)
    assert len(a) == 2100 and a[2050] == 300 and a[-1] == 129
    rest = [x for i, x in enumerate(a) if i not in (2050, 2099)]
    assert min(rest) == 0 and max(rest) <= 39
    assert W.many_short_lengths(2100, seed=92) != a
