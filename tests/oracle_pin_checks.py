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


# --------------------------------------------------------------- backward pass

def _bwd(lib, q, k, v, do, causal, scale, cu=None):
    return oracle.attn_bwd(q, k, v, do, causal, scale, cu_seqlens=cu, n_threads=2, lib=lib)


def _fwd_loss_f64(q, k, v, do, causal, scale, seqs):
    """sum(o * do) for fp64 q [T,Hq,D], k/v [T,Hkv,D], do [T,Hq,D], through
    the brute-force explicit-P forward (no gradient formula involved)."""
    Hq, Hkv = q.shape[1], k.shape[1]
    G = Hq // Hkv
    loss = 0.0
    for t0, L in seqs:
        for h in range(Hq):
            g = h // G
            P = brute.probability_matrix(q[t0:t0 + L, h], k[t0:t0 + L, g], causal, scale)
            loss += float(np.sum((P @ v[t0:t0 + L, g]) * do[t0:t0 + L, h]))
    return loss


def check_bwd_finite_differences(lib):
    """Directional derivatives of sum(o * dO) by central differences of the
    brute-force forward (fp64, step 1e-5) equal <grad, direction> from the
    oracle's dq, dk, dv: fixed length and varlen, causal or not, GQA."""
    rng = np.random.default_rng(5)
    cases = [
        dict(B=1, Hq=4, Hkv=2, S=6, D=4, causal=True, lens=None),
        dict(B=2, Hq=3, Hkv=1, S=5, D=3, causal=False, lens=None),
        dict(B=0, Hq=2, Hkv=2, S=0, D=4, causal=True, lens=[3, 1, 4]),
    ]
    for n, c in enumerate(cases):
        q, k, v, cu = W.make_qkv(c["B"], c["Hq"], c["Hkv"], c["S"], c["D"], seed=61 + n,
                                 lengths=c["lens"])
        do = W.make_grad_out(q.shape, seed=61 + n)
        scale = 0.45
        cu_np = None if cu is None else cu.numpy()
        dq, dk, dv = _bwd(lib, q, k, v, do, c["causal"], scale, cu_np)
        if cu is None:
            B, S = c["B"], c["S"]
            seqs = [(b * S, S) for b in range(B)]
            flat = lambda t: _f64(t).reshape(B * S, t.shape[2], t.shape[3])
        else:
            seqs = [(int(cu[b]), int(cu[b + 1] - cu[b])) for b in range(len(cu) - 1)]
            flat = _f64
        x = [flat(q), flat(k), flat(v)]
        g = [dq.reshape(x[0].shape), dk.reshape(x[1].shape), dv.reshape(x[2].shape)]
        dof = flat(do)
        eps = 1e-5
        for t in range(4):
            dirs = [rng.standard_normal(a.shape) for a in x]
            plus = [a + eps * d for a, d in zip(x, dirs)]
            minus = [a - eps * d for a, d in zip(x, dirs)]
            fd = (_fwd_loss_f64(*plus, dof, c["causal"], scale, seqs) -
                  _fwd_loss_f64(*minus, dof, c["causal"], scale, seqs)) / (2 * eps)
            an = sum(float(np.sum(gg * d)) for gg, d in zip(g, dirs))
            assert abs(fd - an) <= 1e-7 * max(1.0, abs(an)), \
                f"bwd finite differences case {n}: {fd!r} vs {an!r}"
            # one operand at a time, so that a mistake in one gradient cannot
            # hide behind another
            for w in range(3):
                pl = list(x)
                mi = list(x)
                pl[w] = x[w] + eps * dirs[w]
                mi[w] = x[w] - eps * dirs[w]
                fd_w = (_fwd_loss_f64(*pl, dof, c["causal"], scale, seqs) -
                        _fwd_loss_f64(*mi, dof, c["causal"], scale, seqs)) / (2 * eps)
                an_w = float(np.sum(g[w] * dirs[w]))
                assert abs(fd_w - an_w) <= 1e-7 * max(1.0, abs(an_w)), \
                    f"bwd finite differences case {n} operand {w}: {fd_w!r} vs {an_w!r}"


def check_bwd_torch_autograd(lib):
    """Library special case: reverse-mode autograd of PyTorch's fp64
    scaled_dot_product_attention on CPU (K/V repeated per group for GQA, so
    autograd sums each group's gradients)."""
    for causal in (True, False):
        B, Hq, Hkv, S, D = 2, 6, 2, 11, 8
        q, k, v, _ = W.make_qkv(B, Hq, Hkv, S, D, seed=71 + int(causal))
        do = W.make_grad_out(q.shape, seed=71 + int(causal))
        scale = 0.3
        dq, dk, dv = _bwd(lib, q, k, v, do, causal, scale)
        G = Hq // Hkv
        qt = torch.from_numpy(_f64(q)).permute(0, 2, 1, 3).requires_grad_()
        kt = torch.from_numpy(_f64(k)).permute(0, 2, 1, 3).requires_grad_()
        vt = torch.from_numpy(_f64(v)).permute(0, 2, 1, 3).requires_grad_()
        o = torch.nn.functional.scaled_dot_product_attention(
            qt, kt.repeat_interleave(G, dim=1), vt.repeat_interleave(G, dim=1),
            is_causal=causal, scale=scale)
        o.backward(torch.from_numpy(_f64(do)).permute(0, 2, 1, 3))
        _close(dq, qt.grad.permute(0, 2, 1, 3).numpy(), 1e-12, f"autograd dq causal={causal}")
        _close(dk, kt.grad.permute(0, 2, 1, 3).numpy(), 1e-12, f"autograd dk causal={causal}")
        _close(dv, vt.grad.permute(0, 2, 1, 3).numpy(), 1e-12, f"autograd dv causal={causal}")


def check_bwd_zero_scale(lib):
    """scale = 0: P is uniform over the visible keys and no logit depends on
    q or k, so dq = dk = 0 exactly and dv_j = sum over the group's heads and
    the rows i that see j of dO_i / |K_i|."""
    B, Hq, Hkv, S, D = 2, 4, 2, 9, 4
    q, k, v, _ = W.make_qkv(B, Hq, Hkv, S, D, seed=81)
    do = W.make_grad_out(q.shape, seed=81)
    G = Hq // Hkv
    dof = _f64(do)
    for causal in (True, False):
        dq, dk, dv = _bwd(lib, q, k, v, do, causal, 0.0)
        assert np.all(dq == 0.0) and np.all(dk == 0.0), "scale 0: dq, dk not zero"
        want = np.zeros_like(dv)
        for b in range(B):
            for g in range(Hkv):
                for j in range(S):
                    rows = range(j, S) if causal else range(S)
                    for h in range(g * G, (g + 1) * G):
                        for i in rows:
                            want[b, j, g] += dof[b, i, h] / ((i + 1) if causal else S)
        _close(dv, want, 1e-13, f"scale 0 dv causal={causal}")


def check_bwd_single_key(lib):
    """S = 1: P = 1 whatever the logit, so dq = dk = 0 and dv_0 is the sum of
    dO_0 over the group's heads."""
    B, Hq, Hkv, D = 2, 6, 3, 8
    q, k, v, _ = W.make_qkv(B, Hq, Hkv, 1, D, seed=91)
    do = W.make_grad_out(q.shape, seed=91)
    for causal in (True, False):
        dq, dk, dv = _bwd(lib, q, k, v, do, causal, 0.8)
        _close(dq, np.zeros_like(dq), 1e-15, "single key dq")
        _close(dk, np.zeros_like(dk), 1e-15, "single key dk")
        want = _f64(do).reshape(B, 1, Hkv, Hq // Hkv, D).sum(axis=3)
        _close(dv, want, 1e-14, "single key dv")


def check_bwd_sum_identities(lib):
    """Every row of dS sums to zero (sum_j P_ij (dP_ij - Delta_i) = Delta_i -
    Delta_i), so sum_j dk_j = 0 for each (sequence, key/value head); and the
    rows of P sum to one, so sum_j dv_j = sum over the group's heads and all
    rows of dO_i."""
    lens = [7, 1, 12]
    q, k, v, cu = W.make_qkv(0, 6, 2, 0, 8, seed=101, lengths=lens)
    do = W.make_grad_out(q.shape, seed=101)
    G = 3
    for causal in (True, False):
        dq, dk, dv = _bwd(lib, q, k, v, do, causal, 0.6, cu.numpy())
        dof = _f64(do)
        for b in range(len(lens)):
            t0, t1 = int(cu[b]), int(cu[b + 1])
            for g in range(2):
                _close(dk[t0:t1, g].sum(axis=0), np.zeros(8), 1e-12, "sum of dk")
                want = dof[t0:t1, g * G:(g + 1) * G].sum(axis=(0, 1))
                _close(dv[t0:t1, g].sum(axis=0), want, 1e-12, "sum of dv")
        assert np.max(np.abs(dk)) > 1e-3, "dk identically zero"


def check_bwd_gqa_equals_repeated_mha(lib):
    """GQA equals MHA on K/V repeated per group, with dk, dv summed over the
    group's copies."""
    B, Hq, Hkv, S, D = 2, 8, 2, 10, 4
    q, k, v, _ = W.make_qkv(B, Hq, Hkv, S, D, seed=111)
    do = W.make_grad_out(q.shape, seed=111)
    G = Hq // Hkv
    kr = k.repeat_interleave(G, dim=2).contiguous()
    vr = v.repeat_interleave(G, dim=2).contiguous()
    for causal in (True, False):
        dq, dk, dv = _bwd(lib, q, k, v, do, causal, 0.5)
        dq2, dk2, dv2 = _bwd(lib, q, kr, vr, do, causal, 0.5)
        _close(dq, dq2, 1e-13, "gqa dq")
        _close(dk, dk2.reshape(B, S, Hkv, G, D).sum(axis=3), 1e-13, "gqa dk")
        _close(dv, dv2.reshape(B, S, Hkv, G, D).sum(axis=3), 1e-13, "gqa dv")


def check_bwd_varlen_equals_separate(lib):
    """A packed varlen batch equals one fixed-length call per sequence."""
    lens = [5, 9, 1, 4]
    q, k, v, cu = W.make_qkv(0, 4, 2, 0, 8, seed=121, lengths=lens)
    do = W.make_grad_out(q.shape, seed=121)
    for causal in (True, False):
        dq, dk, dv = _bwd(lib, q, k, v, do, causal, 0.4, cu.numpy())
        for b, L in enumerate(lens):
            t0 = int(cu[b])
            sl = slice(t0, t0 + L)
            e = _bwd(lib, q[sl][None].contiguous(), k[sl][None].contiguous(),
                     v[sl][None].contiguous(), do[sl][None].contiguous(), causal, 0.4)
            _close(dq[sl], e[0][0], 1e-13, "varlen dq")
            _close(dk[sl], e[1][0], 1e-13, "varlen dk")
            _close(dv[sl], e[2][0], 1e-13, "varlen dv")


def check_bwd_sampled_match_full(lib):
    """The sampled forms (dq on rows, dk / dv on key ranges) equal the same
    rows of the full backward pass."""
    for causal in (True, False):
        lens = [13, 6, 20]
        q, k, v, cu = W.make_qkv(0, 6, 3, 0, 8, seed=131, lengths=lens)
        do = W.make_grad_out(q.shape, seed=131)
        dq, dk, dv = _bwd(lib, q, k, v, do, causal, 0.35, cu.numpy())
        rows = [(0, 0, 0), (0, 5, 12), (1, 2, 3), (2, 4, 19), (2, 1, 7)]
        got = oracle.attn_bwd_dq_rows(q, k, v, do, causal, 0.35, rows, cu_seqlens=cu.numpy(),
                                      n_threads=2, lib=lib)
        for r, (b, h, i) in enumerate(rows):
            _close(got[r], dq[int(cu[b]) + i, h], 1e-13, "sampled dq row")
        ranges = [(0, 1, 0, 13), (2, 0, 17, 20), (1, 2, 2, 3), (2, 2, 5, 11)]
        gk, gv = oracle.attn_bwd_dkv_ranges(q, k, v, do, causal, 0.35, ranges,
                                            cu_seqlens=cu.numpy(), n_threads=2, lib=lib)
        at = 0
        for b, g, j0, j1 in ranges:
            t0 = int(cu[b])
            _close(gk[at:at + j1 - j0], dk[t0 + j0:t0 + j1, g], 1e-13, "sampled dk range")
            _close(gv[at:at + j1 - j0], dv[t0 + j0:t0 + j1, g], 1e-13, "sampled dv range")
            at += j1 - j0


# ------------------------------------------------- latent (MLA) decode step

def _mla(lib, inp):
    return oracle.mla_decode(inp.q, inp.cache, inp.page_table, inp.seq_lens, inp.scale, inp.dv,
                             n_threads=2, lib=lib)


def _mla_rows(inp, b):
    """The cached latent rows of sequence b, in position order, fp64."""
    L = int(inp.seq_lens[b])
    ps = inp.cache.shape[1]
    c = _f64(inp.cache)
    return np.stack([c[int(inp.page_table[b, j // ps]), j % ps] for j in range(L)]) if L else \
        np.zeros((0, c.shape[2]))


def check_mla_library_sdpa(lib):
    """Library special case: torch's fp64 scaled_dot_product_attention with
    K = the gathered latent rows and V = their first dv components (SDPA
    allows a value dimension other than the key's), one key/value head
    broadcast over the query heads; scipy's logsumexp for the LSE."""
    from scipy.special import logsumexp
    for dqk, dv, ps, lens in ((40, 32, 4, [9, 1, 13]), (576, 512, 64, [70, 3])):
        inp = W.make_mla_paged(lens, 5, ps, seed=161 + dqk, dqk=dqk, dv=dv)
        o, lse = _mla(lib, inp)
        for b, L in enumerate(lens):
            c = torch.from_numpy(_mla_rows(inp, b))
            q = torch.from_numpy(_f64(inp.q[b]))[None, :, None, :]     # [1, Hq, 1, dqk]
            k = c[None, None].expand(1, q.shape[1], L, dqk)
            v = c[None, None, :, :dv].expand(1, q.shape[1], L, dv)
            ref = torch.nn.functional.scaled_dot_product_attention(q, k, v, scale=inp.scale)
            _close(o[b], ref[0, :, 0].numpy(), 1e-12, f"mla sdpa o dqk={dqk}")
            logits = inp.scale * (q[0, :, 0] @ c.T).numpy()
            _close(lse[b], logsumexp(logits, axis=1), 1e-12, f"mla lse dqk={dqk}")


def check_mla_brute_force(lib):
    """The explicit probability matrix over the gathered rows: o = P V."""
    inp = W.make_mla_paged([6, 11], 3, 4, seed=171, dqk=24, dv=16)
    o, lse = _mla(lib, inp)
    for b in range(2):
        c = _mla_rows(inp, b)
        P = brute.probability_matrix(_f64(inp.q[b]), c, False, inp.scale)
        _close(o[b], P @ c[:, :16], TIGHT, "mla brute o")


def check_mla_closed_forms(lib):
    """One key: o = its first dv components, lse = scale q.c.  Scale 0: o is
    the mean of the rows' first dv components, lse = ln L.  No key: o = 0,
    lse = -inf.  Rows permuted across pages: same result."""
    inp = W.make_mla_paged([1, 0, 37], 4, 8, seed=181, dqk=48, dv=32)
    o, lse = _mla(lib, inp)
    c0 = _mla_rows(inp, 0)
    _close(o[0], np.repeat(c0[:, :32], 4, axis=0), 0.0, "mla single key o")
    _close(lse[0], inp.scale * (_f64(inp.q[0]) @ c0[0]), 1e-13, "mla single key lse")
    assert np.all(o[1] == 0.0) and np.all(np.isneginf(lse[1])), "mla empty sequence"
    z = W.MlaInputs(inp.q, inp.cache, inp.page_table, inp.seq_lens, 0.0, inp.dv)
    oz, lz = _mla(lib, z)
    c2 = _mla_rows(inp, 2)
    _close(oz[2], np.repeat(c2[:, :32].mean(axis=0, keepdims=True), 4, axis=0), 1e-13, "mla scale 0 o")
    _close(lz[2], np.full(4, math.log(37)), 1e-13, "mla scale 0 lse")
    # move sequence 2's pages to other physical pages (copying the rows)
    ps, n = 8, (37 + 7) // 8
    cache = inp.cache.clone()
    pt = inp.page_table.clone()
    free = [p for p in range(cache.shape[0]) if p not in set(int(x) for x in pt[pt >= 0])]
    moved = list(reversed([int(pt[2, j]) for j in range(n)]))
    for j in range(n):
        dst = moved[j]
        cache[dst] = inp.cache[int(pt[2, j])]
        pt[2, j] = dst
    o2, lse2 = _mla(lib, W.MlaInputs(inp.q, cache, pt, inp.seq_lens, inp.scale, inp.dv))
    _close(o2[2], o[2], TIGHT, "mla page permutation o")
    _close(lse2[2], lse[2], TIGHT, "mla page permutation lse")
    del free


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
    check_bwd_finite_differences,
    check_bwd_torch_autograd,
    check_bwd_zero_scale,
    check_bwd_single_key,
    check_bwd_sum_identities,
    check_bwd_gqa_equals_repeated_mha,
    check_bwd_varlen_equals_separate,
    check_bwd_sampled_match_full,
    check_mla_library_sdpa,
    check_mla_brute_force,
    check_mla_closed_forms,
]
