"""Pins of the fp64 oracle: facts fixed by mathematics, not by the oracle itself.

Each check takes an oracle library handle, so that tests/test_oracle_mutants.py
can run the same checks against oracles with planted mistakes and show that
each mistake fails at least one of them.  A check raises AssertionError when
the oracle disagrees with the fact it pins.

The attention definition being pinned is the reference operation of the
paper's attention kernels (Section 2.1 and Section 3.1; Table 2, Flash and GQA
Attention): softmax(scale * q k^T + causal mask) v with the row log-sum-exp.
"""
from __future__ import annotations

import math

import numpy as np
import torch

import oracle
from oracle import brute
from paper_2609_04523_gb300 import workloads as W

TIGHT = 1e-12  # fp64 agreement between formulations of the same definition


def _bits(t: torch.Tensor) -> np.ndarray:
    return t.contiguous().view(torch.int16).numpy().view(np.uint16)


def _f64(t: torch.Tensor) -> np.ndarray:
    return t.to(torch.float64).numpy()


def _run(lib, q, k, v, causal, scale, cu=None):
    return oracle.attn_fwd(q, k, v, causal, scale, cu_seqlens=cu, n_threads=2, lib=lib)


def _close(a, b, tol, what):
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    assert a.shape == b.shape, f"{what}: shape {a.shape} vs {b.shape}"
    if a.size == 0:
        return
    assert not np.any(np.isnan(a)), f"{what}: NaN in result"
    with np.errstate(invalid="ignore"):
        err = float(np.max(np.abs(a - b)))
    assert err <= tol, f"{what}: max abs error {err:.3e} > {tol:.1e}"


# --------------------------------------------------------------- brute force

def check_brute_force_tiny(lib):
    """Tiny inputs, all flags: the oracle equals the explicit-P formulation."""
    cases = [
        dict(B=2, Hq=2, Hkv=2, S=5, D=4, causal=True),
        dict(B=1, Hq=4, Hkv=2, S=7, D=8, causal=True),
        dict(B=2, Hq=6, Hkv=3, S=6, D=3, causal=False),
        dict(B=1, Hq=8, Hkv=1, S=9, D=16, causal=False),
        dict(B=3, Hq=4, Hkv=4, S=1, D=5, causal=True),
    ]
    for n, c in enumerate(cases):
        q, k, v, _ = W.make_qkv(c["B"], c["Hq"], c["Hkv"], c["S"], c["D"], seed=11 + n)
        scale = 1.0 / math.sqrt(c["D"]) * (1.0 + 0.5 * n)
        o, lse = _run(lib, q, k, v, c["causal"], scale)
        ob, lseb = brute.attn_fwd(_bits(q), _bits(k), _bits(v), c["causal"], scale)
        _close(o, ob, TIGHT, f"brute case {n} o")
        _close(lse, lseb, TIGHT, f"brute case {n} lse")


def check_brute_force_varlen(lib):
    lens = [3, 1, 8, 5]
    q, k, v, cu = W.make_qkv(0, 4, 2, 0, 8, seed=21, lengths=lens)
    for causal in (True, False):
        o, lse = _run(lib, q, k, v, causal, 0.3, cu.numpy())
        ob, lseb = brute.attn_fwd(_bits(q), _bits(k), _bits(v), causal, 0.3, cu.numpy())
        _close(o, ob, TIGHT, f"varlen brute o causal={causal}")
        _close(lse, lseb, TIGHT, f"varlen brute lse causal={causal}")


def check_library_sdpa(lib):
    """Library special case: PyTorch's fp64 scaled_dot_product_attention on CPU
    (K/V repeated per group for GQA), and scipy's logsumexp of the logit
    matrix for the LSE."""
    from scipy.special import logsumexp
    for causal in (True, False):
        B, Hq, Hkv, S, D = 2, 6, 2, 12, 16
        q, k, v, _ = W.make_qkv(B, Hq, Hkv, S, D, seed=31 + int(causal))
        scale = 0.2
        o, lse = _run(lib, q, k, v, causal, scale)
        G = Hq // Hkv
        qt = torch.from_numpy(_f64(q)).permute(0, 2, 1, 3)
        kt = torch.from_numpy(_f64(k)).permute(0, 2, 1, 3).repeat_interleave(G, dim=1)
        vt = torch.from_numpy(_f64(v)).permute(0, 2, 1, 3).repeat_interleave(G, dim=1)
        ref = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, is_causal=causal,
                                                               scale=scale)
        _close(o, ref.permute(0, 2, 1, 3).numpy(), 1e-12, f"sdpa o causal={causal}")
        logits = scale * torch.matmul(qt, kt.transpose(-1, -2)).numpy()
        if causal:
            logits = np.where(np.triu(np.ones((S, S), dtype=bool), 1), -np.inf, logits)
        _close(lse, logsumexp(logits, axis=-1), 1e-12, f"scipy logsumexp causal={causal}")


# --------------------------------------------------------------- closed forms

def check_identical_keys(lib):
    """All keys equal: P is uniform over the visible keys, so o_i is the mean of
    the visible values and lse_i = scale*q_i.k + ln(#visible)."""
    B, Hq, Hkv, S, D = 1, 4, 2, 37, 8
    q, k, v, _ = W.make_qkv(B, Hq, Hkv, S, D, seed=41)
    k = k[:, :1].expand_as(k).contiguous()  # every key equals key 0 of its head
    scale = 0.7
    G = Hq // Hkv
    for causal in (True, False):
        o, lse = _run(lib, q, k, v, causal, scale)
        vf, qf, kf = _f64(v), _f64(q), _f64(k)
        for h in range(Hq):
            g = h // G
            for i in range(S):
                n = i + 1 if causal else S
                _close(o[0, i, h], vf[0, :n, g].mean(axis=0), 1e-12, "identical keys o")
                want = scale * float(qf[0, i, h] @ kf[0, 0, g]) + math.log(n)
                _close(lse[0, h, i], want, 1e-12, "identical keys lse")


def check_single_key(lib):
    """S = 1: o = v_0 and lse = scale*q_0.k_0, causal or not."""
    B, Hq, Hkv, D = 3, 4, 1, 16
    q, k, v, _ = W.make_qkv(B, Hq, Hkv, 1, D, seed=51)
    for causal in (True, False):
        o, lse = _run(lib, q, k, v, causal, 0.37)
        for b in range(B):
            for h in range(Hq):
                _close(o[b, 0, h], _f64(v)[b, 0, 0], 0.0, "single key o")
                want = 0.37 * float(_f64(q)[b, 0, h] @ _f64(k)[b, 0, 0])
                _close(lse[b, h, 0], want, 1e-14, "single key lse")


def check_zero_scale(lib):
    """scale = 0: every visible logit is 0, so o_i is the visible-prefix mean
    of v and lse_i = ln(#visible)."""
    B, Hq, Hkv, S, D = 2, 2, 1, 20, 8
    q, k, v, _ = W.make_qkv(B, Hq, Hkv, S, D, seed=61)
    for causal in (True, False):
        o, lse = _run(lib, q, k, v, causal, 0.0)
        for b in range(B):
            for i in range(S):
                n = i + 1 if causal else S
                _close(o[b, i, 1], _f64(v)[b, :n, 0].mean(axis=0), 1e-12, "scale 0 o")
                _close(lse[b, 1, i], math.log(n), 1e-14, "scale 0 lse")


def check_negative_scale(lib):
    """scale < 0: scale * q.k = |scale| * (-q).k, and negating a bf16 value is
    exact, so the oracle at (q, -c) equals the oracle at (-q, c) exactly; the
    explicit-P formulation agrees at the negative scale too."""
    B, Hq, Hkv, S, D = 2, 4, 2, 19, 16
    q, k, v, _ = W.make_qkv(B, Hq, Hkv, S, D, seed=131)
    for causal in (False, True):
        o, lse = _run(lib, q, k, v, causal, -0.4)
        o2, lse2 = _run(lib, -q, k, v, causal, 0.4)
        _close(o, o2, 0.0, f"negated scale vs negated q o (causal {causal})")
        _close(lse, lse2, 0.0, f"negated scale vs negated q lse (causal {causal})")
        ob, lseb = brute.attn_fwd(_bits(q), _bits(k), _bits(v), causal, -0.4)
        _close(o, ob, TIGHT, f"negative scale brute o (causal {causal})")
        _close(lse, lseb, TIGHT, f"negative scale brute lse (causal {causal})")


def check_one_hot_values(lib):
    """v_j = e_j (S <= D): o_i is row i of P itself.  Its entries are >= 0,
    sum to 1, vanish on hidden keys, and follow exp(s_ij - lse_i)."""
    B, Hq, Hkv, S, D = 1, 2, 2, 10, 16
    q, k, _, _ = W.make_qkv(B, Hq, Hkv, S, D, seed=71)
    v = torch.zeros(B, S, Hkv, D, dtype=torch.bfloat16)
    for j in range(S):
        v[:, j, :, j] = 1.0
    scale = 0.45
    for causal in (True, False):
        o, lse = _run(lib, q, k, v, causal, scale)
        for h in range(Hq):
            P = o[0, :, h, :S]
            assert np.all(P >= 0.0), "one-hot: negative probability"
            _close(P.sum(axis=1), np.ones(S), 1e-13, "one-hot row sums")
            _close(o[0, :, h, S:], np.zeros((S, D - S)), 0.0, "one-hot unused columns")
            logits = scale * _f64(q)[0, :, h] @ _f64(k)[0, :, h].T
            want = np.exp(logits - lse[0, h][:, None])
            if causal:
                want = np.where(np.triu(np.ones((S, S), dtype=bool), 1), 0.0, want)
                _close(np.triu(P, 1), np.zeros((S, S)), 0.0, "one-hot hidden keys")
            _close(P, want, 1e-12, "one-hot P = exp(s - lse)")


def check_adversarial_rows(lib):
    """Rows with one logit `gap` above the rest: o ~ v_target, within the
    weight left on the other keys, and lse = gap + ln(1 + sum_j e^(s_j - gap))."""
    B, H, S, D = 2, 3, 64, 16
    scale = 0.125
    g = torch.Generator("cpu").manual_seed(81)
    q32 = torch.randn(B, S, H, D, generator=g)
    k32 = torch.randn(B, S, H, D, generator=g)
    v = torch.randn(B, S, H, D, generator=g).to(torch.bfloat16)
    planted = W.plant_adversarial_rows(q32, k32, scale, seed=81)
    q, k = q32.to(torch.bfloat16), k32.to(torch.bfloat16)
    o, lse = _run(lib, q, k, v, False, scale)
    qf, kf, vf = _f64(q), _f64(k), _f64(v)
    for (b, h, r, t) in planted:
        s = scale * kf[b, :, h] @ qf[b, r, h]
        assert abs(s[t] - 30.0) == 0.0, "planted logit is not exactly 30"
        others = np.delete(s, t)
        assert 30.0 - others.max() >= 29.5, "gap below 29.5"
        rest = np.exp(others - 30.0).sum()
        _close(o[b, r, h], vf[b, t, h], 2.0 * rest * np.abs(vf[b, :, h]).max() + 1e-15,
               "adversarial o")
        _close(lse[b, h, r], 30.0 + math.log1p(rest), 1e-12, "adversarial lse")


# ----------------------------------------------------------------- invariants

def check_gqa_equals_repeated_mha(lib):
    B, Hq, Hkv, S, D = 2, 8, 2, 19, 8
    q, k, v, _ = W.make_qkv(B, Hq, Hkv, S, D, seed=91)
    G = Hq // Hkv
    for causal in (True, False):
        o, lse = _run(lib, q, k, v, causal, 0.3)
        o2, lse2 = _run(lib, q, k.repeat_interleave(G, dim=2), v.repeat_interleave(G, dim=2),
                        causal, 0.3)
        _close(o, o2, 0.0, "GQA vs repeated MHA o")
        _close(lse, lse2, 0.0, "GQA vs repeated MHA lse")


def check_varlen_equals_separate(lib):
    lens = [5, 1, 17, 9]
    Hq, Hkv, D = 4, 2, 8
    q, k, v, cu = W.make_qkv(0, Hq, Hkv, 0, D, seed=101, lengths=lens)
    for causal in (True, False):
        o, lse = _run(lib, q, k, v, causal, 0.4, cu.numpy())
        for b, L in enumerate(lens):
            t0 = int(cu[b])
            sl = slice(t0, t0 + L)
            o1, lse1 = _run(lib, q[sl][None], k[sl][None], v[sl][None], causal, 0.4)
            _close(o[sl], o1[0], 0.0, "varlen vs separate o")
            _close(lse[:, sl], lse1[0], 0.0, "varlen vs separate lse")


def check_key_permutation(lib):
    """Non-causal attention does not depend on the order of the (key, value) pairs."""
    B, Hq, Hkv, S, D = 1, 2, 1, 23, 8
    q, k, v, _ = W.make_qkv(B, Hq, Hkv, S, D, seed=111)
    perm = torch.from_numpy(np.random.default_rng(5).permutation(S))
    o, lse = _run(lib, q, k, v, False, 0.5)
    o2, lse2 = _run(lib, q, k[:, perm], v[:, perm], False, 0.5)
    _close(o, o2, 1e-13, "permutation o")
    _close(lse, lse2, 1e-13, "permutation lse")


def check_causal_is_truncated_noncausal(lib):
    """Causal row i equals the last row of non-causal attention over keys 0..i."""
    B, Hq, Hkv, S, D = 1, 2, 2, 13, 8
    q, k, v, _ = W.make_qkv(B, Hq, Hkv, S, D, seed=121)
    o, lse = _run(lib, q, k, v, True, 0.6)
    for i in (0, 1, 6, 12):
        o1, lse1 = _run(lib, q[:, :i + 1], k[:, :i + 1], v[:, :i + 1], False, 0.6)
        _close(o[:, i], o1[:, i], 0.0, "causal vs truncated o")
        _close(lse[:, :, i], lse1[:, :, i], 0.0, "causal vs truncated lse")


def check_logit_shift(lib):
    """Adding c to every logit of a row (through one extra dimension with
    q_extra = c/scale, k_extra = 1) leaves o unchanged and adds c to lse."""
    B, H, S, D = 1, 2, 15, 7
    q, k, v, _ = W.make_qkv(B, H, H, S, D, seed=131)
    scale, c = 0.125, 2.0
    q2 = torch.cat([q, torch.full((B, S, H, 1), c / scale, dtype=torch.bfloat16)], dim=3)
    k2 = torch.cat([k, torch.ones((B, S, H, 1), dtype=torch.bfloat16)], dim=3)
    v2 = torch.cat([v, torch.zeros((B, S, H, 1), dtype=torch.bfloat16)], dim=3)
    for causal in (True, False):
        o, lse = _run(lib, q, k, v, causal, scale)
        o2, lse2 = _run(lib, q2, k2, v2, causal, scale)
        _close(o2[..., :D], o, 1e-13, "shift o")
        _close(lse2, lse + c, 1e-13, "shift lse")


def check_value_affine(lib):
    """o is linear in v, and adding a constant to every value adds it to o
    (the weights of a row sum to one)."""
    B, Hq, Hkv, S, D = 1, 2, 1, 16, 8
    q, k, v, _ = W.make_qkv(B, Hq, Hkv, S, D, seed=141)
    for causal in (True, False):
        o, _ = _run(lib, q, k, v, causal, 0.3)
        o2, _ = _run(lib, q, k, (v.float() * 2).to(torch.bfloat16), causal, 0.3)
        _close(o2, 2 * o, 0.0, "linear in v")
        o3, _ = _run(lib, q, k, torch.full_like(v, 3.0), causal, 0.3)
        _close(o3, np.full(o3.shape, 3.0), 1e-13, "constant values")


def check_rows_match_full(lib):
    lens = [40, 7, 130]
    Hq, Hkv, D = 4, 2, 8
    q, k, v, cu = W.make_qkv(0, Hq, Hkv, 0, D, seed=151, lengths=lens)
    o, lse = _run(lib, q, k, v, True, 0.3, cu.numpy())
    rows = W.sample_rows(lens, Hq, 60, seed=3)
    orow, lrow = oracle.attn_rows(q, k, v, True, 0.3, rows, cu_seqlens=cu.numpy(),
                                  n_threads=2, lib=lib)
    for n, (b, h, i) in enumerate(rows):
        t = int(cu[b]) + int(i)
        _close(orow[n], o[t, h], 0.0, "rows vs full o")
        _close(lrow[n], lse[h, t], 0.0, "rows vs full lse")


# ------------------------------------------------------- paged decode step

def _decode(lib, inp):
    return oracle.decode_paged(inp.q, inp.k_cache, inp.v_cache, inp.page_table, inp.seq_lens,
                               inp.scale, n_threads=2, lib=lib)


def _gather(cache, page_table, L, page_size):
    """The first L cached positions of one sequence, contiguous: [L, Hkv, D]."""
    rows = [cache[int(page_table[j // page_size]), j % page_size] for j in range(L)]
    return torch.stack(rows) if rows else cache[:0, 0]


def check_decode_equals_prefill_last_row(lib):
    """A decode step is the last row of causal attention over the same keys:
    gather each sequence's pages into a packed varlen batch, put the decode
    query at its last position, and ask the (separately pinned) prefill
    definition for that row."""
    lens, Hq, Hkv, D, ps = [1, 7, 16, 33, 50], 6, 2, 8, 16
    inp = W.make_paged(lens, Hq, Hkv, D, ps, seed=140)
    o, lse = _decode(lib, inp)
    k = torch.cat([_gather(inp.k_cache, inp.page_table[b], L, ps) for b, L in enumerate(lens)])
    v = torch.cat([_gather(inp.v_cache, inp.page_table[b], L, ps) for b, L in enumerate(lens)])
    q = torch.zeros((sum(lens), Hq, D), dtype=torch.bfloat16)
    starts = np.cumsum([0] + lens)
    for b, L in enumerate(lens):
        q[starts[b] + L - 1] = inp.q[b]
    rows = np.array([(b, h, L - 1) for b, L in enumerate(lens) for h in range(Hq)], dtype=np.int64)
    o_ref, lse_ref = oracle.attn_rows(q, k, v, True, inp.scale, rows, cu_seqlens=starts,
                                      n_threads=2, lib=lib)
    _close(o.reshape(-1, D), o_ref, TIGHT, "decode vs prefill last row o")
    _close(lse.reshape(-1), lse_ref, TIGHT, "decode vs prefill last row lse")


def check_decode_page_permutation(lib):
    """Where the pages sit in the cache does not matter: relabelling the
    physical pages (and the page table with them) changes nothing."""
    lens, Hq, Hkv, D, ps = [40, 3, 64], 4, 4, 8, 8
    inp = W.make_paged(lens, Hq, Hkv, D, ps, seed=141, spare_pages=5)
    o, lse = _decode(lib, inp)
    n = inp.k_cache.shape[0]
    perm = torch.from_numpy(np.random.default_rng(7).permutation(n))  # new slot of page i
    inv = torch.empty_like(perm)
    inv[perm] = torch.arange(n)
    pt = inp.page_table.clone()
    pt[pt >= 0] = perm[pt[pt >= 0].long()].int()
    moved = W.PagedInputs(inp.q, inp.k_cache[inv], inp.v_cache[inv], pt, inp.seq_lens, inp.scale)
    o2, lse2 = _decode(lib, moved)
    _close(o, o2, 0.0, "page permutation o")
    _close(lse, lse2, 0.0, "page permutation lse")


def check_decode_single_key(lib):
    """One cached key: o = v_0 and lse = scale * q . k_0."""
    Hq, Hkv, D, ps = 4, 2, 16, 16
    inp = W.make_paged([1, 1], Hq, Hkv, D, ps, seed=142)
    o, lse = _decode(lib, inp)
    for b in range(2):
        pg = int(inp.page_table[b, 0])
        for h in range(Hq):
            g = h // (Hq // Hkv)
            k0 = _f64(inp.k_cache[pg, 0, g])
            v0 = _f64(inp.v_cache[pg, 0, g])
            _close(o[b, h], v0, TIGHT, "single key o")
            _close(lse[b, h], inp.scale * float(np.dot(_f64(inp.q[b, h]), k0)), TIGHT, "single key lse")


def check_decode_identical_keys(lib):
    """All cached keys equal: the weights are uniform, so o is the mean of the
    values and lse = scale * q . k + ln L."""
    Hq, Hkv, D, ps, L = 2, 1, 8, 8, 21
    inp = W.make_paged([L], Hq, Hkv, D, ps, seed=143)
    kc = inp.k_cache.clone()
    kc[:] = kc[int(inp.page_table[0, 0]), 0]
    inp = W.PagedInputs(inp.q, kc, inp.v_cache, inp.page_table, inp.seq_lens, inp.scale)
    o, lse = _decode(lib, inp)
    v = _f64(_gather(inp.v_cache, inp.page_table[0], L, ps))[:, 0]
    k0 = _f64(kc[0, 0, 0])
    for h in range(Hq):
        _close(o[0, h], v.mean(axis=0), 1e-12, "identical keys o")
        _close(lse[0, h], inp.scale * float(np.dot(_f64(inp.q[0, h]), k0)) + math.log(L), 1e-12,
               "identical keys lse")


def check_decode_empty_sequence(lib):
    """No cached key: o = 0 and lse = -inf (the defensive reading)."""
    inp = W.make_paged([0, 9], 2, 2, 8, 8, seed=144)
    o, lse = _decode(lib, inp)
    assert np.all(o[0] == 0.0), "empty sequence o"
    assert np.all(np.isneginf(lse[0])), "empty sequence lse"
    assert np.all(np.isfinite(lse[1])), "non-empty sequence lse"


ALL_CHECKS = [
    check_brute_force_tiny,
    check_brute_force_varlen,
    check_library_sdpa,
    check_identical_keys,
    check_single_key,
    check_zero_scale,
    check_negative_scale,
    check_one_hot_values,
    check_adversarial_rows,
    check_gqa_equals_repeated_mha,
    check_varlen_equals_separate,
    check_key_permutation,
    check_causal_is_truncated_noncausal,
    check_logit_shift,
    check_value_affine,
    check_rows_match_full,
    check_decode_equals_prefill_last_row,
    check_decode_page_permutation,
    check_decode_single_key,
    check_decode_identical_keys,
    check_decode_empty_sequence,
]
