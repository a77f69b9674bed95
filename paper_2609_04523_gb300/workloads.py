"""Seeded synthetic inputs for the attention forward pass.

This module is the one piece shared by the CUDA path's tests and bench and by
the oracle side: it draws inputs and does work accounting, and holds none of
the attention arithmetic.  Everything is generated on the CPU so that the
oracle and the GPU see identical bf16 bits.

The paper evaluates its attention kernels (Table 2, Flash Attention and GQA
Attention rows; ragged attention) on workloads from a benchmark suite that is
not available here and whose shapes the paper does not print.  The five
configurations below stand in for them; their shapes, value distributions and
structure are synthetic.

Recipe (every config): ``torch.Generator('cpu').manual_seed(1000 + n)`` for
config n (1-based); fp32 ``randn`` for q, then k, then v, each multiplied by
sigma, then rounded to bf16 (round-to-nearest-even).
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np
import torch

TILE = 128  # rows per query tile and keys per key/value block of the kernels


@dataclass(frozen=True)
class AttnConfig:
    index: int             # 1-based config number
    name: str
    B: int                 # batch (fixed length) or number of sequences (varlen)
    Hq: int
    Hkv: int
    S: int                 # sequence length, or total tokens T for varlen
    D: int
    causal: bool
    sigma: float
    varlen: bool = False
    adversarial: bool = False
    len_range: tuple = (512, 4096)
    description: str = ""

    @property
    def scale(self) -> float:
        return 1.0 / math.sqrt(self.D)

    @property
    def seed(self) -> int:
        return 1000 + self.index


CONFIGS = [
    AttnConfig(1, "causal_mha_b1_h2_s128_d64", B=1, Hq=2, Hkv=2, S=128, D=64,
               causal=True, sigma=1.0,
               description="causal MHA fwd, B=1, Hq=Hkv=2, S=128, D=64, N(0,1)"),
    AttnConfig(2, "causal_gqa_b4_hq32_hkv8_s2048_d128", B=4, Hq=32, Hkv=8, S=2048, D=128,
               causal=True, sigma=1.0,
               description="causal GQA fwd, B=4, Hq=32, Hkv=8, S=2048, D=128, N(0,1)"),
    AttnConfig(3, "causal_gqa_b1_hq32_hkv8_s32768_d128", B=1, Hq=32, Hkv=8, S=32768, D=128,
               causal=True, sigma=0.5,
               description="causal GQA long-context fwd, B=1, Hq=32, Hkv=8, S=32768, D=128, N(0,0.5^2)"),
    AttnConfig(4, "noncausal_mha_b16_h16_s1024_d64_adv", B=16, Hq=16, Hkv=16, S=1024, D=64,
               causal=False, sigma=1.0, adversarial=True,
               description="non-causal MHA fwd, B=16, Hq=Hkv=16, S=1024, D=64, N(0,1), "
                           "4 adversarial rows per (b,h) with one logit 30 above the rest"),
    AttnConfig(5, "causal_gqa_varlen_hq64_hkv8_d128_t32768", B=0, Hq=64, Hkv=8, S=32768, D=128,
               causal=True, sigma=1.0, varlen=True,
               description="causal GQA varlen packed fwd, Hq=64, Hkv=8, D=128, 32768 tokens, "
                           "lengths ~ U{512..4096}, last truncated"),
]


def config(n: int) -> AttnConfig:
    return CONFIGS[n - 1]


# ----------------------------------------------------------------- lengths

def varlen_lengths(seed: int, total: int, lo: int = 512, hi: int = 4096) -> list[int]:
    """Lengths drawn uniformly from lo..hi (inclusive) until they reach `total`;
    the last one is truncated so that they sum to exactly `total` (it may fall
    below lo, down to 1)."""
    rng = np.random.default_rng(seed)
    lens: list[int] = []
    acc = 0
    while acc < total:
        L = int(rng.integers(lo, hi + 1))
        L = min(L, total - acc)
        lens.append(L)
        acc += L
    return lens


def many_short_lengths(n: int, seed: int) -> list[int]:
    """n lengths drawn uniformly from 0..39 (empty sequences included), with a
    300-token sequence at index n - 50 and a 129-token one last, when n > 50."""
    rng = np.random.default_rng(seed)
    lens = [int(x) for x in rng.integers(0, 40, size=n)]
    if n > 50:
        lens[n - 50] = 300
        lens[n - 1] = 129
    return lens


def cu_from_lengths(lens) -> torch.Tensor:
    cu = [0]
    for L in lens:
        cu.append(cu[-1] + int(L))
    return torch.tensor(cu, dtype=torch.int32)


# ----------------------------------------------------------------- tensors

def randn_bf16(shape, gen: torch.Generator, sigma: float = 1.0) -> torch.Tensor:
    return (torch.randn(shape, generator=gen, dtype=torch.float32) * sigma).to(torch.bfloat16)


def make_qkv(B: int, Hq: int, Hkv: int, S: int, D: int, seed: int, sigma: float = 1.0,
             lengths=None):
    """Seeded bf16 q, k, v (and int32 cu_seqlens when `lengths` is given).

    Fixed length: q [B,S,Hq,D], k/v [B,S,Hkv,D].  Varlen (lengths given):
    q [T,Hq,D], k/v [T,Hkv,D] with T = sum(lengths)."""
    g = torch.Generator("cpu").manual_seed(seed)
    if lengths is None:
        qs, ks = (B, S, Hq, D), (B, S, Hkv, D)
        cu = None
    else:
        T = int(sum(lengths))
        qs, ks = (T, Hq, D), (T, Hkv, D)
        cu = cu_from_lengths(lengths)
    q = randn_bf16(qs, g, sigma)
    k = randn_bf16(ks, g, sigma)
    v = randn_bf16(ks, g, sigma)
    return q, k, v, cu


def make_grad_out(shape, seed: int, sigma: float = 1.0) -> torch.Tensor:
    """Seeded bf16 output gradient dO for the backward pass (layout of q):
    N(0, sigma^2) drawn from its own generator, so that q, k, v of the same
    seed are unchanged."""
    g = torch.Generator("cpu").manual_seed(seed + 7919)
    return randn_bf16(tuple(shape), g, sigma)


def plant_adversarial_rows(q32: torch.Tensor, k32: torch.Tensor, scale: float, seed: int,
                           n_rows: int = 4, gap: float = 30.0, noise: float = 1e-3):
    """Makes, in each (b, h), `n_rows` query rows whose logit row has one entry
    `gap` above the rest (fp32 tensors [B,S,H,D], modified in place, before bf16
    rounding).

    For a = 0..n_rows-1, with distinct rows r_a and distinct target keys t_a
    drawn from the seed: column a of k is set to noise*N(0,1) for every key,
    k[t_a, a] = 1, and q[r_a] = 0 except q[r_a, a] = gap/scale.  Then logit
    (r_a, t_a) is exactly `gap` and every other logit of row r_a is
    gap*noise*N(0,1).  Returns the list of (b, h, r_a, t_a)."""
    B, S, H, D = q32.shape
    if n_rows > D or n_rows > S:
        raise ValueError("too many adversarial rows for this shape")
    rng = np.random.default_rng(seed + 7919)
    g = torch.Generator("cpu").manual_seed(seed + 7919)
    planted = []
    for b in range(B):
        for h in range(H):
            rows = rng.choice(S, n_rows, replace=False)
            tgts = rng.choice(S, n_rows, replace=False)
            for a in range(n_rows):
                k32[b, :, h, a] = torch.randn(S, generator=g) * noise
                k32[b, int(tgts[a]), h, a] = 1.0
                q32[b, int(rows[a]), h, :] = 0.0
                q32[b, int(rows[a]), h, a] = gap / scale
                planted.append((b, h, int(rows[a]), int(tgts[a])))
    return planted


@dataclass
class Inputs:
    cfg: AttnConfig
    q: torch.Tensor
    k: torch.Tensor
    v: torch.Tensor
    cu_seqlens: torch.Tensor | None
    lengths: list = field(default_factory=list)
    adversarial: list = field(default_factory=list)

    @property
    def B(self) -> int:
        return len(self.lengths) if self.cfg.varlen else self.cfg.B

    @property
    def S(self) -> int:
        return self.cfg.S


def make_config_inputs(n: int) -> Inputs:
    """Inputs of config n (1-based), bit-identical on every call."""
    c = config(n)
    g = torch.Generator("cpu").manual_seed(c.seed)
    if c.varlen:
        lens = varlen_lengths(c.seed, c.S, *c.len_range)
        T = sum(lens)
        q = randn_bf16((T, c.Hq, c.D), g, c.sigma)
        k = randn_bf16((T, c.Hkv, c.D), g, c.sigma)
        v = randn_bf16((T, c.Hkv, c.D), g, c.sigma)
        return Inputs(c, q, k, v, cu_from_lengths(lens), lens)
    qs, ks = (c.B, c.S, c.Hq, c.D), (c.B, c.S, c.Hkv, c.D)
    if not c.adversarial:
        q = randn_bf16(qs, g, c.sigma)
        k = randn_bf16(ks, g, c.sigma)
        v = randn_bf16(ks, g, c.sigma)
        return Inputs(c, q, k, v, None, [c.S] * c.B)
    q32 = torch.randn(qs, generator=g, dtype=torch.float32) * c.sigma
    k32 = torch.randn(ks, generator=g, dtype=torch.float32) * c.sigma
    v = randn_bf16(ks, g, c.sigma)
    planted = plant_adversarial_rows(q32, k32, c.scale, c.seed)
    return Inputs(c, q32.to(torch.bfloat16), k32.to(torch.bfloat16), v, None,
                  [c.S] * c.B, planted)


# ---------------------------------------------------------- work accounting

def attn_flops(lengths, Hq: int, D: int, causal: bool) -> float:
    """Algorithmic FLOPs of the forward pass, FlashAttention convention:
    two contractions of 2*D flops per (query, key) pair, i.e. 4*D*L^2 per
    sequence and head, halved for causal."""
    total = 0.0
    for L in lengths:
        f = 4.0 * Hq * D * float(L) * float(L)
        total += f / 2.0 if causal else f
    return total


def attn_pairs(lengths, Hq: int, causal: bool) -> int:
    """Exact count of visible (query, key) pairs, summed over heads."""
    n = 0
    for L in lengths:
        n += Hq * (L * (L + 1) // 2 if causal else L * L)
    return n


def attn_bytes(T: int, Hq: int, Hkv: int, D: int) -> int:
    """Minimal HBM traffic: read q, k, v once (bf16), write o (bf16) and lse (fp32)."""
    return 2 * T * Hq * D + 2 * 2 * T * Hkv * D + 2 * T * Hq * D + 4 * T * Hq


def sample_rows(lengths, Hq: int, n: int, seed: int, tile: int = TILE) -> np.ndarray:
    """A deterministic row sample (b, h, i) for checks at full size: every row
    of the last query tile of every head of every sequence (the rows that see
    the most keys), the first row of every sequence, plus uniform random rows,
    `n` in total at least."""
    rng = np.random.default_rng(seed)
    rows = []
    for b, L in enumerate(lengths):
        if L <= 0:
            continue
        last0 = ((L - 1) // tile) * tile
        for h in range(Hq):
            rows += [(b, h, i) for i in range(last0, L)]
        rows.append((b, int(rng.integers(0, Hq)), 0))
    total = sum(lengths)
    cum = np.cumsum([0] + list(lengths))
    while len(rows) < n:
        t = int(rng.integers(0, total))
        b = int(np.searchsorted(cum, t, side="right") - 1)
        rows.append((b, int(rng.integers(0, Hq)), int(t - cum[b])))
    return np.asarray(rows, dtype=np.int64)


# ------------------------------------------------------------ paged decode

@dataclass
class PagedInputs:
    """One decode step against a paged K/V cache (see make_paged)."""
    q: torch.Tensor           # bf16 [B, Hq, D]
    k_cache: torch.Tensor     # bf16 [num_pages, page_size, Hkv, D]
    v_cache: torch.Tensor     # bf16 [num_pages, page_size, Hkv, D]
    page_table: torch.Tensor  # int32 [B, max_pages]
    seq_lens: torch.Tensor    # int32 [B]
    scale: float


def make_paged(seq_lens, Hq: int, Hkv: int, D: int, page_size: int, seed: int,
               sigma: float = 1.0, spare_pages: int = 3, max_pages: int | None = None) -> PagedInputs:
    """Seeded decode inputs: each sequence's ceil(L/page_size) logical pages
    get distinct physical pages in a random order (with `spare_pages` unused
    pages mixed in), the way a cache allocator hands them out.  Unused
    page-table entries are -1.  Pure data generation: no attention arithmetic."""
    g = torch.Generator("cpu").manual_seed(seed)
    lens = [int(x) for x in seq_lens]
    need = [(L + page_size - 1) // page_size for L in lens]
    mp = max(1, max(need) if max_pages is None else max_pages)
    num_pages = sum(need) + spare_pages
    perm = torch.randperm(num_pages, generator=g).tolist()
    pt = torch.full((len(lens), mp), -1, dtype=torch.int32)
    at = 0
    for b, n in enumerate(need):
        for j in range(n):
            pt[b, j] = perm[at]
            at += 1
    q = randn_bf16((len(lens), Hq, D), g, sigma)
    kc = randn_bf16((num_pages, page_size, Hkv, D), g, sigma)
    vc = randn_bf16((num_pages, page_size, Hkv, D), g, sigma)
    return PagedInputs(q, kc, vc, pt, torch.tensor(lens, dtype=torch.int32), 1.0 / math.sqrt(D))


@dataclass
class MlaInputs:
    q: torch.Tensor           # bf16 [B, Hq, dqk]
    cache: torch.Tensor       # bf16 [num_pages, page_size, dqk]: latent (dv) + rope (dqk - dv)
    page_table: torch.Tensor  # int32 [B, max_pages], unused entries -1
    seq_lens: torch.Tensor    # int32 [B]
    scale: float
    dv: int


def make_mla_paged(seq_lens, Hq: int, page_size: int, seed: int, dqk: int = 576, dv: int = 512,
                   sigma: float = 1.0, spare_pages: int = 3,
                   max_pages: int | None = None) -> MlaInputs:
    """Seeded inputs of a latent (MLA) decode step: one shared latent cache,
    pages handed out in a random order as in make_paged.  The scale is
    1/sqrt(dqk).  Pure data generation: no attention arithmetic."""
    g = torch.Generator("cpu").manual_seed(seed)
    lens = [int(x) for x in seq_lens]
    need = [(L + page_size - 1) // page_size for L in lens]
    mp = max(1, max(need) if max_pages is None else max_pages)
    num_pages = sum(need) + spare_pages
    perm = torch.randperm(num_pages, generator=g).tolist()
    pt = torch.full((len(lens), mp), -1, dtype=torch.int32)
    at = 0
    for b, n in enumerate(need):
        for j in range(n):
            pt[b, j] = perm[at]
            at += 1
    q = randn_bf16((len(lens), Hq, dqk), g, sigma)
    cache = randn_bf16((num_pages, page_size, dqk), g, sigma)
    return MlaInputs(q, cache, pt, torch.tensor(lens, dtype=torch.int32), 1.0 / math.sqrt(dqk), dv)


def mla_decode_bytes(seq_lens, Hq: int, dqk: int = 576, dv: int = 512) -> int:
    """Minimal HBM traffic of one latent decode step: every cached latent row
    read once (bf16), q read, o written (bf16), lse written."""
    keys = int(sum(int(x) for x in seq_lens))
    B = len(seq_lens)
    return 2 * keys * dqk + 2 * B * Hq * dqk + 2 * B * Hq * dv + 4 * B * Hq


def mla_decode_flops(seq_lens, Hq: int, dqk: int = 576, dv: int = 512) -> float:
    """Matmul FLOPs of one latent decode step: 2 (dqk + dv) per head and key."""
    return 2.0 * (dqk + dv) * Hq * float(sum(int(x) for x in seq_lens))


def decode_bytes(seq_lens, Hq: int, Hkv: int, D: int) -> int:
    """Minimal HBM traffic of one decode step: every cached key and value of
    every sequence read once, q read and o written once (bf16), lse written."""
    keys = int(sum(int(x) for x in seq_lens))
    B = len(seq_lens)
    return 2 * 2 * keys * Hkv * D + 2 * 2 * B * Hq * D + 4 * B * Hq
