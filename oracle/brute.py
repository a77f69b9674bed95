"""Brute-force explicit-softmax-matrix attention in fp64 (TEST INFRASTRUCTURE).

A second, deliberately different formulation of the same definition as
``mk_oracle.c``, for tiny inputs only: it forms the whole logit matrix of a
(sequence, head) pair, writes -inf where the causal mask or the sequence end
hides a key, normalises every row of the matrix into the probability matrix
P, and takes O = P V and lse = ln(sum_j exp(s_ij)).  The tests use it as one
of the pins of the C oracle (brute force on tiny inputs) and to expose P
itself (row sums, one-hot checks).

Only tests/ may import it.
"""
from __future__ import annotations

import numpy as np


def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to fp64."""
    u32 = bits.astype(np.uint32) << np.uint32(16)
    return u32.view(np.float32).astype(np.float64)


def probability_matrix(q: np.ndarray, k: np.ndarray, causal: bool, scale: float) -> np.ndarray:
    """P for one (sequence, head): q [L,D], k [L,D] in fp64 -> P [L,L]."""
    L = q.shape[0]
    logits = scale * (q @ k.T)
    if causal:
        hidden = np.triu(np.ones((L, L), dtype=bool), k=1)  # key j > query i
        logits = np.where(hidden, -np.inf, logits)
    row_max = logits.max(axis=1, keepdims=True)
    e = np.exp(logits - row_max)
    return e / e.sum(axis=1, keepdims=True)


def log_sum_exp_rows(q: np.ndarray, k: np.ndarray, causal: bool, scale: float) -> np.ndarray:
    L = q.shape[0]
    logits = scale * (q @ k.T)
    if causal:
        logits = np.where(np.triu(np.ones((L, L), dtype=bool), k=1), -np.inf, logits)
    row_max = logits.max(axis=1)
    return row_max + np.log(np.exp(logits - row_max[:, None]).sum(axis=1))


def attn_fwd(q_bits, k_bits, v_bits, causal: bool, scale: float, cu_seqlens=None):
    """Same interface and layouts as ``oracle.attn_fwd`` (uint16 bf16 bits in)."""
    q = bf16_bits_to_f64(np.asarray(q_bits))
    k = bf16_bits_to_f64(np.asarray(k_bits))
    v = bf16_bits_to_f64(np.asarray(v_bits))
    if cu_seqlens is None:
        B, S, Hq, D = q.shape
        Hkv = k.shape[2]
        seqs = [(b * S, S) for b in range(B)]
        q = q.reshape(B * S, Hq, D)
        k = k.reshape(B * S, Hkv, D)
        v = v.reshape(B * S, Hkv, D)
        lse = np.zeros((B, Hq, S))
    else:
        _, Hq, D = q.shape
        Hkv = k.shape[1]
        cu = [int(c) for c in cu_seqlens]
        seqs = [(cu[b], cu[b + 1] - cu[b]) for b in range(len(cu) - 1)]
        lse = np.zeros((Hq, q.shape[0]))
    group = Hq // Hkv
    o = np.zeros_like(q)
    for b, (t0, L) in enumerate(seqs):
        if L == 0:
            continue
        for h in range(Hq):
            g = h // group
            qs, ks, vs = q[t0:t0 + L, h], k[t0:t0 + L, g], v[t0:t0 + L, g]
            P = probability_matrix(qs, ks, causal, scale)
            o[t0:t0 + L, h] = P @ vs
            row_lse = log_sum_exp_rows(qs, ks, causal, scale)
            if cu_seqlens is None:
                lse[b, h] = row_lse
            else:
                lse[h, t0:t0 + L] = row_lse
    if cu_seqlens is None:
        o = o.reshape(len(seqs), -1, Hq, D)
    return o, lse
