// fmha_bwd.cu -- attention backward pass for GB300 (sm_103a) and its C ABI.
//
// Gradients of the forward definition (softmax(scale * q k^T + causal mask) v)
// with respect to q, k and v, for an output gradient dO -- the training step
// of the paper's attention kernels (the forward rows of Table 2; the GDN row's
// forward + backward step shows the training context).  With P_ij =
// exp(scale * q_i.k_j - lse_i) over the visible keys:
//   dv_j    = sum_{h in group} sum_i P_ij dO_i
//   dP_ij   = dO_i . v_j,   Delta_i = sum_j P_ij dP_ij = dO_i . o_i
//   dS_ij   = P_ij (dP_ij - Delta_i)
//   dq_i    = scale * sum_j dS_ij k_j
//   dk_j    = scale * sum_{h in group} sum_i dS_ij q_i
//
// Kernels, all deterministic (no atomics), launched dQ first:
//   delta_kernel   Delta_i = dO_i . o_i from the forward's bf16 o (fp32); only
//                  for callers that want Delta without dQ (the dQ kernel
//                  computes it for its own rows and stores it).
//   bwd_kernel<D, false> (dK/dV): a unit is (sequence, key/value head g,
//                  128-key tile); it holds K and V and streams the Q and dO
//                  tiles of every query head of g's group (causal: the query
//                  tiles at or after the key tile), with S^T = K Q^T and
//                  dP^T = V dO^T in TMEM (lanes = keys), P^T and dS^T written
//                  back to TMEM as bf16, dV += P^T dO and dK += dS^T Q.
//   bwd_kernel<D, true> (dQ): a unit is (sequence, query head, 128-row query
//                  tile); it holds Q and dO (and computes the tile's Delta
//                  from dO and o, writing it for the dK/dV kernel), streams K
//                  and V tiles, with S = Q K^T, dP = dO V^T, dS to TMEM and
//                  dQ += dS K.
// dQ recomputes S and dP instead of accumulating partial dQ tiles across
// CTAs, which keeps the result deterministic and needs no fp32 scratch.
//
// Both kernel modes share one structure: persistent CTAs (one per SM), units
// dealt heaviest first in snake order, 10 warps:
//   warps 0-3, 4-7  elementwise warpgroups: warp w owns TMEM lanes
//                   32 (w % 4) .. + 31 (one key row, or one query row), and
//                   warpgroup w / 4 owns columns 64 (w / 4) .. + 63 of S and dP
//   warp 8          tcgen05 MMA issuer
//   warp 9          TMA producer (and, for dK/dV, the per-column lse / Delta
//                   vectors of each streamed query tile)
// TMEM (512 columns): S at 0, dP at 128, accumulators at 256 (dV, then dK at
// 256 + D; or dQ).  A warpgroup writes its bf16 half of P (or dS) into the
// first 32 columns of its own 64-column half of S (or dP), so the two
// warpgroups never touch each other's columns; the MMA reads the 128-key
// operand from columns 0..31 and 64..95.
// MMA order per streamed tile n (software pipeline):
//   dV += P(n) dO(n);  S(n+1);  dK += dS(n) Q(n);  dP(n+1)
// so the exponentials of tile n+1 (which need S(n+1) only) overlap dK(n) and
// dP(n+1), and dS(n+1) overlaps dV(n+1) and S(n+2).  tcgen05 MMAs issued by
// one thread run in order, so S(n+1) overwriting P(n) after dV(n) has read
// it (and dP(n+1) overwriting dS(n) after dK(n)) needs no extra wait.
#include <cuda.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>
#include <mutex>

#include "mk_attn.h"
#include "ptx.cuh"
#include "tma_host.h"

namespace mk {
namespace bwd {

constexpr int kTile = 128;
constexpr int kEwThreads = 256;  // two elementwise warpgroups
constexpr int kMmaWarp = 8;
constexpr int kLoadWarp = 9;
constexpr int kThreads = 320;
constexpr int kBoxCols = 64;
constexpr int kBoxBytes = kTile * kBoxCols * 2;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColS = 0;
constexpr uint32_t kColP = 128;
constexpr uint32_t kColAcc = 256;
constexpr float kLog2e = 1.4426950408889634f;

__device__ int g_status = 0;  // MK_ERR_TIMEOUT once a wait ran out

// 32 lanes x 16 columns of 32-bit words from registers into TMEM (the warp's
// lane quarter), asynchronous until tcgen05.wait::st.
__device__ __forceinline__ void tmem_st_x16(uint32_t taddr, const uint32_t *r) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
      "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
      "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
      : "memory");
}

// Ring depths: Y1 is the load on the critical path (its slot frees only when
// the last MMA of an iteration has read it), so it gets the deeper ring where
// shared memory allows: at D = 128 the dQ kernel has room for three Y1
// stages, the dK/dV kernel (which also stages lse / Delta vectors per Y1
// stage) for two.
template <int D, bool DQ>
struct Cfg {
  static_assert(D == 64 || D == 128, "head dimension 64 or 128");
  static constexpr int kStages1 = (D == 128) ? (DQ ? 3 : 2) : 4;
  static constexpr int kStages2 = (D == 128) ? 2 : 4;
  static constexpr int kHalves = D / kBoxCols;
  static constexpr int kTileBytes = kTile * D * 2;
  static constexpr int kOffX1 = 0;               // K (dK/dV) or Q (dQ)
  static constexpr int kOffX2 = kTileBytes;      // V (dK/dV) or dO (dQ)
  static constexpr int kOffY1 = 2 * kTileBytes;  // Y1 ring: Q (dK/dV) or K (dQ)
  static constexpr int kOffY2 = kOffY1 + kStages1 * kTileBytes;  // Y2 ring: dO or V
  // dK/dV: [stage][lse2 | delta][128]; dQ: [warpgroup][128] halves of Delta
  static constexpr int kOffVec = kOffY2 + kStages2 * kTileBytes;
  static constexpr int kOffCtl = kOffVec + (DQ ? 2 * kTile * 4 : kStages1 * 2 * kTile * 4);
  static constexpr int kSmemBytes = kOffCtl + 256 + 1024;
  static_assert(kSmemBytes <= 232448, "shared memory per CTA");
};

// Streamed operands have a ring each: Y1 (Q for dK/dV, K for dQ) and Y2 (dO,
// or V).  Y2's last reader (dV, or dP) finishes long before Y1's (dK, or dQ),
// so separate barriers let the producer refill Y2 early and leave only Y1's
// load on the critical path.
struct Ctl {
  uint64_t fixed_full, fixed_empty;
  uint64_t y1_full[4], y1_empty[4], y2_full[4], y2_empty[4];
  uint64_t s_full, dp_full, p_full, dp_free, ds_full, acc_full, mma_drained;
  uint64_t dx_full;  // dQ: both warpgroups' halves of the unit's Delta are in shared memory
  uint32_t tmem_base;
  int abort;
};
static_assert(sizeof(Ctl) <= 256, "control block");

struct Params {
  const float *lse;          // [B, Hq, S] or [Hq, T]
  float *delta;              // same layout: written by the dQ kernel, read by dK/dV
  const uint16_t *o;         // bf16, layout of q (the dQ kernel's Delta)
  uint16_t *dq, *dk, *dv;    // bf16, layouts of q, k, v
  const int32_t *cu_seqlens;
  int B, Hq, Hkv, S, G;      // S: tokens per sequence, or total tokens T (varlen)
  int causal, varlen;
  int n_tiles;               // fixed length: 128-row tiles per sequence
  int n_units;
  int schedule;              // MK_SCHED_*
  float scale, scale_log2;
};

// A work unit: sequence b (token range [seq_start, seq_start + len)), head
// (key/value head for dK/dV, query head for dQ) and the unit's own tile.
struct Unit {
  int valid;
  int b, head, tile;
  int seq_start, len;
};

__device__ __forceinline__ int clamp_tok(int x, int T) { return x < 0 ? 0 : (x > T ? T : x); }
__device__ __forceinline__ int tiles_of(int L) { return (L + kTile - 1) / kTile; }

// Unit u.  Fixed length: units are numbered heaviest first when causal (dK/dV:
// key tile 0 first, it is seen by every query tile; dQ: the last query tile
// first), heads innermost so that consecutive units share K/V in L2.
// Varlen: tile rank u / H in sequence order (a warp scan over cu_seqlens,
// called by all 32 lanes), head u % H.
template <bool DQ>
__device__ __forceinline__ Unit map_unit(const Params &p, int u) {
  Unit w;
  const int H = DQ ? p.Hq : p.Hkv;
  if (!p.varlen) {
    const int per_level = p.B * H;
    const int level = u / per_level, rem = u - level * per_level;
    w.valid = u < p.n_units;
    w.b = rem / H;
    w.head = rem % H;
    w.tile = (DQ && p.causal) ? p.n_tiles - 1 - level : level;
    w.seq_start = w.b * p.S;
    w.len = p.S;
    return w;
  }
  const int lane = lane_id();
  w.valid = 0;
  w.b = w.head = w.tile = w.seq_start = w.len = 0;
  const int rank = u / H;
  w.head = u % H;
  int carry = 0;
  for (int base = 0; base < p.B; base += 32) {
    const int b = base + lane;
    int s0 = 0, s1 = 0, nt = 0;
    if (b < p.B) {
      s0 = clamp_tok(p.cu_seqlens[b], p.S);
      s1 = clamp_tok(p.cu_seqlens[b + 1], p.S);
      if (s1 < s0) s1 = s0;
      nt = tiles_of(s1 - s0);
    }
    int incl = nt;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl += y;
    }
    const int excl = incl - nt;
    const bool mine = b < p.B && rank >= carry + excl && rank < carry + incl;
    const unsigned m = __ballot_sync(0xffffffffu, mine);
    if (m) {
      const int src = __ffs(m) - 1;
      w.valid = 1;
      w.b = base + src;
      w.tile = rank - carry - __shfl_sync(0xffffffffu, excl, src);
      w.seq_start = __shfl_sync(0xffffffffu, s0, src);
      w.len = __shfl_sync(0xffffffffu, s1 - s0, src);
      break;
    }
    carry += __shfl_sync(0xffffffffu, incl, 31);
  }
  return w;
}

// Streamed tiles of a unit: dK/dV visits (query head hh of the group, query
// tile qt) for qt from first_q; dQ visits key tiles 0 .. n_kv - 1.
template <bool DQ>
__device__ __forceinline__ int unit_iters(const Params &p, const Unit &w, int &first_q) {
  const int nt = tiles_of(w.len);
  if constexpr (DQ) {
    first_q = 0;
    return p.causal ? min(w.tile + 1, nt) : nt;
  } else {
    first_q = p.causal ? w.tile : 0;
    return p.G * (nt - first_q);
  }
}

// Unit of this CTA in round k (MK_SCHED_*; snake by default, as in the
// forward kernel); an index >= n_units means no unit.
__device__ __forceinline__ int unit_of_round(int k, int schedule, int n_units) {
  const int G = gridDim.x, c = blockIdx.x;
  if (schedule == MK_SCHED_BLOCKED) {
    const int per = (n_units + G - 1) / G;
    return k < per ? c * per + k : n_units;
  }
  if (schedule == MK_SCHED_ROUND_ROBIN) return k * G + c;
  return (k & 1) ? (k + 1) * G - 1 - c : k * G + c;
}

__device__ __forceinline__ void prefetch_l2(const void *ptr) {
  asm volatile("prefetch.global.L2 [%0];" ::"l"(ptr));
}

__device__ __forceinline__ void drain_wait(uint64_t *bar, uint32_t parity) {
  int local_abort = 0;
  mbar_wait(bar, parity, &local_abort);
}

// Index of (sequence start + position pos, query head h) in lse / delta.
__device__ __forceinline__ int64_t row_index(const Params &p, const Unit &w, int h, int pos) {
  return p.varlen ? (int64_t)h * p.S + w.seq_start + pos
                  : ((int64_t)w.b * p.Hq + h) * p.S + pos;
}

template <int D, bool DQ>
__global__ void __launch_bounds__(kThreads, 1)
    bwd_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
               const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_do,
               const Params p) {
  using C = Cfg<D, DQ>;
  constexpr int NS1 = C::kStages1;
  constexpr int NS2 = C::kStages2;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw_addr = smem_addr(smem_raw);
  uint8_t *smem = smem_raw + ((1024u - (raw_addr & 1023u)) & 1023u);
  Ctl *ctl = reinterpret_cast<Ctl *>(smem + C::kOffCtl);
  float *vec = reinterpret_cast<float *>(smem + C::kOffVec);
  const int warp = threadIdx.x / 32;

  if (threadIdx.x == 0) {
    mbar_init(&ctl->fixed_full, 1);
    // dQ: the fixed tiles are free once the MMAs are done with them and the
    // elementwise warps have read the dO tile for Delta.
    mbar_init(&ctl->fixed_empty, DQ ? 2 : 1);
    for (int s = 0; s < NS1; ++s) {
      // Y1 of dK/dV: the TMA bytes plus one arrival per producer lane for
      // the lse / Delta vectors the lanes write.
      mbar_init(&ctl->y1_full[s], DQ ? 1 : 33);
      mbar_init(&ctl->y1_empty[s], 1);
    }
    for (int s = 0; s < NS2; ++s) {
      mbar_init(&ctl->y2_full[s], 1);
      mbar_init(&ctl->y2_empty[s], 1);
    }
    mbar_init(&ctl->s_full, 1);
    mbar_init(&ctl->dp_full, 1);
    mbar_init(&ctl->p_full, kEwThreads);
    mbar_init(&ctl->dp_free, kEwThreads);
    mbar_init(&ctl->ds_full, kEwThreads);
    mbar_init(&ctl->acc_full, 1);
    mbar_init(&ctl->mma_drained, 1);
    mbar_init(&ctl->dx_full, kEwThreads);
    ctl->abort = 0;
    fence_mbar_init();
  }
  if (warp == kMmaWarp) {
    tmem_alloc(&ctl->tmem_base, kTmemCols);
    tmem_relinquish_alloc_permit();
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem = ctl->tmem_base;
  volatile int *abort = &ctl->abort;

  if (warp == kLoadWarp) {
    // ------------------------------------------------------------ producer
    if (elect_one()) {
      tma_prefetch_desc(&tm_q);
      tma_prefetch_desc(&tm_k);
      tma_prefetch_desc(&tm_v);
      tma_prefetch_desc(&tm_do);
    }
    const uint64_t pol = l2_policy_evict_last();
    const int lane = lane_id();
    uint32_t n_unit = 0, it = 0;
    bool ok = true;
    auto load_tile = [&](uint8_t *dst, const CUtensorMap *map, uint64_t *bar, int head, int row0) {
#pragma unroll
      for (int hb = 0; hb < C::kHalves; ++hb)
        tma_load_3d(dst + hb * kBoxBytes, map, bar, hb * kBoxCols, head, row0, pol);
    };
    for (int k = 0; ok && k * (int)gridDim.x < p.n_units; ++k) {
      const int u = unit_of_round(k, p.schedule, p.n_units);
      if (u >= p.n_units) continue;
      const Unit w = map_unit<DQ>(p, u);
      if (!w.valid) continue;
      int first_q = 0;
      const int N = unit_iters<DQ>(p, w, first_q);
      ok = mbar_wait_all(&ctl->fixed_empty, (n_unit & 1) ^ 1, abort);
      if (!ok) break;
      if (elect_one()) {
        mbar_arrive_expect_tx(&ctl->fixed_full, 2 * C::kTileBytes);
        const int row0 = w.seq_start + w.tile * kTile;
        if constexpr (DQ) {
          load_tile(smem + C::kOffX1, &tm_q, &ctl->fixed_full, w.head, row0);
          load_tile(smem + C::kOffX2, &tm_do, &ctl->fixed_full, w.head, row0);
        } else {
          load_tile(smem + C::kOffX1, &tm_k, &ctl->fixed_full, w.head, row0);
          load_tile(smem + C::kOffX2, &tm_v, &ctl->fixed_full, w.head, row0);
        }
      }
      __syncwarp();
      ++n_unit;
      const int nq = tiles_of(w.len) - first_q;
      // dK/dV: lse in base 2 and Delta of the 128 query positions of streamed
      // tile n, 4 per lane, loaded one tile ahead so that their latency
      // overlaps the wait for a free slot; positions past the sequence end get
      // lse2 = +inf (P = 0) and Delta = 0, so they contribute nothing.
      float l2v[kTile / 32], dlv[kTile / 32];
      auto fetch_vec = [&](int n) {
        const int h = w.head * p.G + n / nq;
        const int qt = first_q + n % nq;
#pragma unroll
        for (int e = 0; e < kTile / 32; ++e) {
          const int pos = qt * kTile + e * 32 + lane;
          l2v[e] = INFINITY;
          dlv[e] = 0.f;
          if (pos < w.len) {
            const int64_t ri = row_index(p, w, h, pos);
            l2v[e] = p.lse[ri] * kLog2e;
            dlv[e] = p.delta[ri];
          }
        }
      };
      if constexpr (!DQ) fetch_vec(0);
      for (int n = 0; n < N; ++n) {
        const int s1 = it % NS1, s2 = it % NS2;
        uint8_t *y1 = smem + C::kOffY1 + s1 * C::kTileBytes;
        uint8_t *y2 = smem + C::kOffY2 + s2 * C::kTileBytes;
        // Head and token row of the streamed tiles: dQ streams the key tiles
        // of the query head's key/value head; dK/dV streams the query tiles
        // of each head of the group.
        const int head = DQ ? w.head / p.G : w.head * p.G + n / nq;
        const int row0 = w.seq_start + (DQ ? n : first_q + n % nq) * kTile;
        // Y1 first: S needs it a whole elementwise phase before dP needs Y2.
        ok = mbar_wait_all(&ctl->y1_empty[s1], ((it / NS1) & 1) ^ 1, abort);
        if (!ok) break;
        if (elect_one()) {
          mbar_arrive_expect_tx(&ctl->y1_full[s1], C::kTileBytes);
          load_tile(y1, DQ ? &tm_k : &tm_q, &ctl->y1_full[s1], head, row0);
        }
        __syncwarp();
        if constexpr (!DQ) {
          float *lv = vec + s1 * 2 * kTile;
#pragma unroll
          for (int e = 0; e < kTile / 32; ++e) {
            lv[e * 32 + lane] = l2v[e];
            lv[kTile + e * 32 + lane] = dlv[e];
          }
          mbar_arrive(&ctl->y1_full[s1]);  // every lane: its vector writes are released
        }
        ok = mbar_wait_all(&ctl->y2_empty[s2], ((it / NS2) & 1) ^ 1, abort);
        if (!ok) break;
        if (elect_one()) {
          mbar_arrive_expect_tx(&ctl->y2_full[s2], C::kTileBytes);
          load_tile(y2, DQ ? &tm_v : &tm_do, &ctl->y2_full[s2], head, row0);
        }
        __syncwarp();
        if constexpr (!DQ) {
          if (n + 1 < N) fetch_vec(n + 1);
        }
        ++it;
      }
    }
    // Teardown: the loads issued land before the CTA exits.
    if (n_unit > 0) drain_wait(&ctl->fixed_full, (n_unit - 1) & 1);
    for (uint32_t n = (it > (uint32_t)NS1 ? it - NS1 : 0); n < it; ++n)
      drain_wait(&ctl->y1_full[n % NS1], (n / NS1) & 1);
    for (uint32_t n = (it > (uint32_t)NS2 ? it - NS2 : 0); n < it; ++n)
      drain_wait(&ctl->y2_full[n % NS2], (n / NS2) & 1);
  } else if (warp == kMmaWarp) {
    // ---------------------------------------------------------- MMA issuer
    constexpr uint32_t idesc_ss = idesc_bf16_f32(kTile, kTile, false, false);
    constexpr uint32_t idesc_ts = idesc_bf16_f32(kTile, D, false, true);
    constexpr uint32_t kLbo = (D > kBoxCols) ? kBoxBytes : 1024;
    const uint32_t sX1 = smem_addr(smem + C::kOffX1), sX2 = smem_addr(smem + C::kOffX2);
    const uint32_t sY1 = smem_addr(smem + C::kOffY1), sY2 = smem_addr(smem + C::kOffY2);
    // dQ: dS(i) (bf16, 64 columns: keys 0..63 from warpgroup 0, 64..127 from
    // warpgroup 1) goes to buffer i % 2 after the dQ accumulator.
    constexpr uint32_t kColDs = kColAcc + D;
    uint32_t n_unit = 0, it = 0, n_p = 0, n_ds = 0;
    bool ok = true;
    // D[tmem col] = X[smem] Y[smem]^T, both K-major (head dim contiguous).
    auto issue_xy = [&](uint32_t col, uint32_t x_addr, uint32_t y_addr) {
      const uint64_t a0 = sdesc_sw128(x_addr, 16, 1024);
      const uint64_t b0 = sdesc_sw128(y_addr, 16, 1024);
#pragma unroll
      for (int kk = 0; kk < D / 16; ++kk) {
        const uint32_t off = ((kk >> 2) * kBoxBytes + (kk & 3) * 32) >> 4;
        umma_ss(tmem + col, a0 + off, b0 + off, idesc_ss, kk > 0 ? 1u : 0u);
      }
    };
    // acc[tmem col] (+)= A[tmem a_col] Y[smem], Y MN-major (128 rows x D):
    // the 128-wide contraction runs over the rows of Y; its bf16 A operand
    // sits in columns a_col + 0..31 (rows 0..63 of Y) and a_col + 32 + gap ..
    // gap: 32 when the two 32-column halves sit in place in S / dP (columns
    // a_col + 0..31 and + 64..95), 0 for a packed 64-column dS buffer.
    auto issue_acc = [&](uint32_t col, uint32_t a_col, uint32_t gap, uint32_t y_addr,
                         bool accumulate) {
      const uint64_t b0 = sdesc_sw128(y_addr, kLbo, 1024);
#pragma unroll
      for (int kk = 0; kk < kTile / 16; ++kk) {
        const uint32_t a = tmem + a_col + kk * 8 + (kk >= 4 ? gap : 0);
        umma_ts(tmem + col, a, b0 + (uint64_t)(kk * 128), idesc_ts,
                (accumulate || kk > 0) ? 1u : 0u);
      }
    };
    for (int k = 0; ok && k * (int)gridDim.x < p.n_units; ++k) {
      const int u = unit_of_round(k, p.schedule, p.n_units);
      if (u >= p.n_units) continue;
      const Unit w = map_unit<DQ>(p, u);
      if (!w.valid) continue;
      int first_q = 0;
      const int N = unit_iters<DQ>(p, w, first_q);
      ok = mbar_wait_all(&ctl->fixed_full, n_unit & 1, abort);
      if (!ok) break;
      const uint32_t it0 = it;
      auto y1_of = [&](uint32_t i) { return sY1 + (i % NS1) * C::kTileBytes; };
      auto y2_of = [&](uint32_t i) { return sY2 + (i % NS2) * C::kTileBytes; };
      ok = mbar_wait_all(&ctl->y1_full[it0 % NS1], (it0 / NS1) & 1, abort);
      if (!ok) break;
      tc_fence_after_sync();
      if (elect_one()) {
        issue_xy(kColS, sX1, y1_of(it0));
        umma_commit(&ctl->s_full);
      }
      __syncwarp();
      ok = mbar_wait_all(&ctl->y2_full[it0 % NS2], (it0 / NS2) & 1, abort);
      if (!ok) break;
      tc_fence_after_sync();
      if (elect_one()) {
        issue_xy(kColP, sX2, y2_of(it0));
        umma_commit(&ctl->dp_full);
        if constexpr (DQ) umma_commit(&ctl->y2_empty[it0 % NS2]);  // V read by dP only
        if (N == 1) umma_commit(&ctl->fixed_empty);
      }
      __syncwarp();
      for (int n = 0; ok && n < N; ++n) {
        const uint32_t i = it0 + n;
        const bool more = n + 1 < N;
        ok = mbar_wait_all(&ctl->p_full, n_p & 1, abort);
        ++n_p;
        if (!ok) break;
        tc_fence_after_sync();
        if constexpr (!DQ) {
          if (elect_one()) {
            issue_acc(kColAcc, kColS, 32, y2_of(i), n > 0);  // dV += P dO
            umma_commit(&ctl->y2_empty[i % NS2]);  // dO(n) no longer read
          }
          __syncwarp();
        }
        if (more) {
          ok = mbar_wait_all(&ctl->y1_full[(i + 1) % NS1], ((i + 1) / NS1) & 1, abort);
          if (!ok) break;
          tc_fence_after_sync();
          if (elect_one()) {
            issue_xy(kColS, sX1, y1_of(i + 1));
            umma_commit(&ctl->s_full);
          }
          __syncwarp();
        }
        if constexpr (DQ) {
          // dP(n) has been read into registers and dS(n) goes to its own
          // buffer, so dP(n+1) need not wait for dQ(n).
          ok = mbar_wait_all(&ctl->dp_free, (n_ds & 1), abort);
          if (!ok) break;
          if (more) {
            ok = mbar_wait_all(&ctl->y2_full[(i + 1) % NS2], ((i + 1) / NS2) & 1, abort);
            if (!ok) break;
            tc_fence_after_sync();
            if (elect_one()) {
              issue_xy(kColP, sX2, y2_of(i + 1));
              umma_commit(&ctl->dp_full);
              umma_commit(&ctl->y2_empty[(i + 1) % NS2]);  // V read by dP only
              if (n + 2 == N) umma_commit(&ctl->fixed_empty);
            }
            __syncwarp();
          }
        }
        ok = mbar_wait_all(&ctl->ds_full, n_ds & 1, abort);
        ++n_ds;
        if (!ok) break;
        if (!DQ && more) ok = mbar_wait_all(&ctl->y2_full[(i + 1) % NS2], ((i + 1) / NS2) & 1, abort);
        if (!ok) break;
        tc_fence_after_sync();
        if (elect_one()) {
          if constexpr (DQ) {
            issue_acc(kColAcc, kColDs + (i & 1) * 64, 0, y1_of(i), n > 0);  // dQ += dS K
          } else {
            issue_acc(kColAcc + D, kColP, 32, y1_of(i), n > 0);  // dK += dS Q
          }
          umma_commit(&ctl->y1_empty[i % NS1]);
          if (!DQ && more) {
            issue_xy(kColP, sX2, y2_of(i + 1));
            umma_commit(&ctl->dp_full);
            if (n + 2 == N) umma_commit(&ctl->fixed_empty);
          }
          if (!more) umma_commit(&ctl->acc_full);
        }
        __syncwarp();
      }
      it = it0 + N;
      ++n_unit;
    }
    if (elect_one()) umma_commit(&ctl->mma_drained);
    __syncwarp();
    drain_wait(&ctl->mma_drained, 0);
  } else {
    // ------------------------------------------------------ elementwise
    const int wg = warp / 4;                  // column half
    const int row = (warp % 4) * 32 + lane_id();  // TMEM lane: key row (dK/dV) or query row (dQ)
    const uint32_t t_row = tmem + ((uint32_t)((warp % 4) * 32) << 16);
    const int col0 = wg * 64;
    const float c2 = p.scale_log2;
    uint32_t n_unit = 0, it = 0, n_s = 0;
    bool ok = true;
    constexpr uint32_t kColAcc2 = DQ ? kColAcc : kColAcc + D;
    static_assert(!DQ || kColAcc + D + 128 <= kTmemCols, "dS buffers");
    for (int k = 0; ok && k * (int)gridDim.x < p.n_units; ++k) {
      const int u = unit_of_round(k, p.schedule, p.n_units);
      if (u >= p.n_units) continue;
      const Unit w = map_unit<DQ>(p, u);
      if (!w.valid) continue;
      int first_q = 0;
      const int N = unit_iters<DQ>(p, w, first_q);
      const int nq = tiles_of(w.len) - first_q;
      // dQ: this thread's query row, its lse (base 2) and Delta = dO . o.
      // The lse and this warpgroup's half of the o row are loaded here (the
      // previous unit prefetched them into L2) and used in the first key
      // tile: lse for P, and o, with the dO tile in shared memory, for Delta,
      // which the first dS needs and the dK/dV kernel reads back.
      const int qpos = w.tile * kTile + row;
      float row_l2 = INFINITY, row_dl = 0.f, lse_raw = INFINITY;
      int64_t ri = 0;
      uint4 ov[DQ ? D / 16 : 1];
      if constexpr (DQ) {
        if (qpos < w.len) {
          ri = row_index(p, w, w.head, qpos);
          lse_raw = p.lse[ri];
          const uint16_t *orow = p.o + (((int64_t)w.seq_start + qpos) * p.Hq + w.head) * D + wg * (D / 2);
#pragma unroll
          for (int c8 = 0; c8 < D / 16; ++c8) ov[c8] = *reinterpret_cast<const uint4 *>(orow + c8 * 8);
        }
      }
      for (int n = 0; n < N; ++n) {
        const uint32_t i = it + n;
        if constexpr (DQ) {
          if (n == N - 1) {  // last key tile: bring the next unit's o and lse rows into L2
            const int un = unit_of_round(k + 1, p.schedule, p.n_units);
            if (un < p.n_units) {
              const Unit wn = map_unit<DQ>(p, un);
              const int qn = wn.tile * kTile + row;
              if (wn.valid && qn < wn.len) {
                prefetch_l2(p.o + (((int64_t)wn.seq_start + qn) * p.Hq + wn.head) * D + wg * (D / 2));
                if (wg == 0) prefetch_l2(p.lse + row_index(p, wn, wn.head, qn));
              }
            }
          }
        }
        ok = mbar_wait_all(&ctl->s_full, n_s & 1, abort);
        if (!ok) break;
        tc_fence_after_sync();
        float x[64];
        {
          uint32_t raw[2][32];
          tmem_ld_32x32b_x32(t_row + kColS + col0, raw[0]);
          tmem_ld_32x32b_x32(t_row + kColS + col0 + 32, raw[1]);
          tmem_ld_wait();
          reg_fence(raw[0]);
          reg_fence(raw[1]);
#pragma unroll
          for (int c = 0; c < 64; ++c) x[c] = __uint_as_float(raw[c / 32][c % 32]);
        }
        // P = 2^(s * scale * log2 e - lse2), hidden pairs 0.
        const float *lv = vec + (i % NS1) * 2 * kTile;
        if constexpr (DQ) {
          // S(n) is in registers: S(n+1) may overwrite it.
          tc_fence_before_sync();
          mbar_arrive(&ctl->p_full);
          if (n == 0) row_l2 = lse_raw * kLog2e;
          const int kpos0 = n * kTile + col0;  // key position of column 0 of this half
          const int lim = p.causal ? min(w.len, qpos + 1) : w.len;  // keys [0, lim)
          const bool mask = kpos0 + 64 > lim;
#pragma unroll
          for (int c = 0; c < 64; ++c) {
            const float e = ex2_approx(fmaf(x[c], c2, -row_l2));
            x[c] = (!mask || kpos0 + c < lim) ? e : 0.f;
          }
          if (n == 0) {
            ok = mbar_wait_all(&ctl->fixed_full, (n_unit & 1), abort);  // the dO tile has landed
            if (!ok) break;
            float part = 0.f;
            if (qpos < w.len) {
              const uint8_t *dorow = smem + C::kOffX2;
#pragma unroll
              for (int c8 = 0; c8 < D / 16; ++c8) {  // this warpgroup's D/2 components, 8 at a time
                const int e0 = wg * (D / 2) + c8 * 8;
                const int chunk = (e0 % kBoxCols) / 8;
                const uint4 dv4 = *reinterpret_cast<const uint4 *>(
                    dorow + (e0 / kBoxCols) * kBoxBytes + row * 128 + ((chunk ^ (row & 7)) << 4));
                const uint32_t aw[4] = {dv4.x, dv4.y, dv4.z, dv4.w};
                const uint32_t bw[4] = {ov[c8].x, ov[c8].y, ov[c8].z, ov[c8].w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                  part = fmaf(__uint_as_float(aw[e] << 16), __uint_as_float(bw[e] << 16), part);
                  part = fmaf(__uint_as_float(aw[e] & 0xffff0000u), __uint_as_float(bw[e] & 0xffff0000u), part);
                }
              }
            }
            // The two warpgroups' halves meet in vec.  A warpgroup writes the
            // next unit's half only after this unit's dQ accumulation, which
            // needs both warpgroups' first dS: no overwrite.  The exchange is
            // an mbarrier with a bounded wait, so a warpgroup that unwinds on
            // a timeout cannot leave the other one waiting for ever.
            vec[wg * kTile + row] = part;
            mbar_arrive(&ctl->dx_full);
            ok = mbar_wait_all(&ctl->dx_full, n_unit & 1, abort);
            if (!ok) break;
            // Every elementwise thread has read the dO tile: release it.
            if (threadIdx.x == 0) mbar_arrive(&ctl->fixed_empty);
            row_dl = vec[row] + vec[kTile + row];
            if (wg == 0 && qpos < w.len &&
                dbg_in_range(ri, (int64_t)p.Hq * (p.varlen ? p.S : (int64_t)p.B * p.S),
                             &g_status))
              p.delta[ri] = row_dl;
          }
        } else {
          // The producer lanes wrote this slot's vectors before arriving on
          // its full barrier; that phase has completed (the MMA waited for it
          // before S) and cannot advance before this iteration ends.
          ok = mbar_wait_all(&ctl->y1_full[i % NS1], (i / NS1) & 1, abort);
          if (!ok) break;
          const int qt = first_q + n % nq;
          const bool diag = p.causal && qt == w.tile;  // key row > query column hidden
#pragma unroll
          for (int c = 0; c < 64; c += 4) {
            const float4 l4 = *reinterpret_cast<const float4 *>(lv + col0 + c);
            x[c] = ex2_approx(fmaf(x[c], c2, -l4.x));
            x[c + 1] = ex2_approx(fmaf(x[c + 1], c2, -l4.y));
            x[c + 2] = ex2_approx(fmaf(x[c + 2], c2, -l4.z));
            x[c + 3] = ex2_approx(fmaf(x[c + 3], c2, -l4.w));
          }
          if (diag) {
#pragma unroll
            for (int c = 0; c < 64; ++c) x[c] = (row > col0 + c) ? 0.f : x[c];
          }
          // P^T (bf16) into the first 32 columns of this half of S, in two
          // stores so that the first one's latency overlaps the second pack.
          uint32_t pk[32];
#pragma unroll
          for (int c = 0; c < 16; ++c) pk[c] = pack_bf16x2(x[2 * c], x[2 * c + 1]);
          tmem_st_x16(t_row + kColS + col0, pk);
#pragma unroll
          for (int c = 16; c < 32; ++c) pk[c] = pack_bf16x2(x[2 * c], x[2 * c + 1]);
          tmem_st_x16(t_row + kColS + col0 + 16, pk + 16);
          tmem_st_wait();
          tc_fence_before_sync();
          mbar_arrive(&ctl->p_full);
        }
        ok = mbar_wait_all(&ctl->dp_full, n_s & 1, abort);
        ++n_s;
        if (!ok) break;
        tc_fence_after_sync();
        {
          uint32_t raw[2][32];
          tmem_ld_32x32b_x32(t_row + kColP + col0, raw[0]);
          tmem_ld_32x32b_x32(t_row + kColP + col0 + 32, raw[1]);
          tmem_ld_wait();
          reg_fence(raw[0]);
          reg_fence(raw[1]);
          if constexpr (DQ) {  // dP(n) is in registers: dP(n+1) may overwrite it
            tc_fence_before_sync();
            mbar_arrive(&ctl->dp_free);
          }
          // dK/dV: dS^T in place of dP^T; dQ: dS into buffer i % 2.  Two
          // stores of 32 keys each, the first overlapping the second half.
          const uint32_t t_ds = t_row + (DQ ? kColAcc + D + (i & 1) * 64 + wg * 32 : kColP + col0);
          uint32_t pk[32];
#pragma unroll
          for (int hh = 0; hh < 2; ++hh) {
#pragma unroll
            for (int c = hh * 32; c < hh * 32 + 32; c += 4) {
              float4 d4;
              if constexpr (DQ) {
                d4 = make_float4(row_dl, row_dl, row_dl, row_dl);
              } else {
                d4 = *reinterpret_cast<const float4 *>(lv + kTile + col0 + c);
              }
              const float ds0 = x[c] * (__uint_as_float(raw[c / 32][c % 32]) - d4.x);
              const float ds1 = x[c + 1] * (__uint_as_float(raw[c / 32][c % 32 + 1]) - d4.y);
              const float ds2 = x[c + 2] * (__uint_as_float(raw[c / 32][c % 32 + 2]) - d4.z);
              const float ds3 = x[c + 3] * (__uint_as_float(raw[c / 32][c % 32 + 3]) - d4.w);
              pk[c / 2] = pack_bf16x2(ds0, ds1);
              pk[c / 2 + 1] = pack_bf16x2(ds2, ds3);
            }
            tmem_st_x16(t_ds + hh * 16, pk + hh * 16);
          }
          tmem_st_wait();
        }
        tc_fence_before_sync();
        mbar_arrive(&ctl->ds_full);
      }
      if (!ok) break;
      it += N;
      // ------------------------------------------------------ epilogue
      ok = mbar_wait_all(&ctl->acc_full, n_unit & 1, abort);
      ++n_unit;
      if (!ok) break;
      tc_fence_after_sync();
      const int pos = w.tile * kTile + row;
      const int64_t tok = (int64_t)w.seq_start + pos;
      // Check build: the row lies inside its output (tokens x heads rows).
      const bool valid = pos < w.len &&
                         dbg_in_range(tok, p.varlen ? (int64_t)p.S : (int64_t)p.B * p.S,
                                      &g_status) &&
                         dbg_in_range(w.head, DQ ? p.Hq : p.Hkv, &g_status);
      // This warpgroup stores columns wg * D/2 .. + D/2 of its row.
      auto store_acc = [&](uint32_t col, uint16_t *base, int heads, int head, float mul) {
        uint4 *dst = reinterpret_cast<uint4 *>(base + (tok * heads + head) * (int64_t)D + wg * (D / 2));
#pragma unroll
        for (int c = 0; c < D / 64; ++c) {
          uint32_t raw[32];
          tmem_ld_32x32b_x32(t_row + col + wg * (D / 2) + c * 32, raw);
          tmem_ld_wait();
          reg_fence(raw);
          uint32_t v[16];
#pragma unroll
          for (int e = 0; e < 16; ++e)
            v[e] = pack_bf16x2(__uint_as_float(raw[2 * e]) * mul, __uint_as_float(raw[2 * e + 1]) * mul);
          if (valid) {
#pragma unroll
            for (int e = 0; e < 4; ++e)
              dst[c * 4 + e] = make_uint4(v[4 * e], v[4 * e + 1], v[4 * e + 2], v[4 * e + 3]);
          }
        }
      };
      if constexpr (DQ) {
        store_acc(kColAcc2, p.dq, p.Hq, w.head, p.scale);
      } else {
        store_acc(kColAcc, p.dv, p.Hkv, w.head, 1.f);
        store_acc(kColAcc2, p.dk, p.Hkv, w.head, p.scale);
      }
      tc_fence_before_sync();
    }
    if (!ok) *abort = 1;
  }

  tc_fence_before_sync();
  __syncthreads();
  if (warp == kMmaWarp) {
    tc_fence_after_sync();
    tmem_dealloc(tmem, kTmemCols);
  }
  if (threadIdx.x == 0 && ctl->abort) atomicExch(&g_status, (int)MK_ERR_TIMEOUT);
}

// Delta_i = dO_i . o_i in fp32, one half-warp per (token, query head) row:
// block (x, y) takes tokens 16 x .. 16 x + 15 of query head y, so that the
// Delta writes of a block are contiguous in the layout of lse.
template <int D>
__global__ void __launch_bounds__(256) delta_kernel(const uint16_t *o, const uint16_t *dO,
                                                    float *delta, int tokens, int Hq, int S,
                                                    int varlen) {
  const int tok = blockIdx.x * 16 + (int)(threadIdx.x >> 4);
  const int h = blockIdx.y;
  const int l16 = threadIdx.x & 15;
  float acc = 0.f;
  if (tok < tokens && l16 * 8 < D) {
    const int64_t off = ((int64_t)tok * Hq + h) * D + l16 * 8;
    const uint4 a = *reinterpret_cast<const uint4 *>(o + off);
    const uint4 b = *reinterpret_cast<const uint4 *>(dO + off);
    const uint32_t aw[4] = {a.x, a.y, a.z, a.w}, bw[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      acc = fmaf(__uint_as_float(aw[e] << 16), __uint_as_float(bw[e] << 16), acc);
      acc = fmaf(__uint_as_float(aw[e] & 0xffff0000u), __uint_as_float(bw[e] & 0xffff0000u), acc);
    }
  }
#pragma unroll
  for (int off = 8; off > 0; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
  if (tok < tokens && l16 == 0) {
    int64_t idx;
    if (varlen) {
      idx = (int64_t)h * S + tok;
    } else {
      const int b = tok / S;
      idx = ((int64_t)b * Hq + h) * S + (tok - b * S);
    }
    delta[idx] = acc;
  }
}

// ------------------------------------------------------------------- host

struct DeviceInfo {
  std::once_flag once;
  int sm_count = 0;
  cudaError_t attr_err[4] = {cudaSuccess, cudaSuccess, cudaSuccess, cudaSuccess};
};
static DeviceInfo g_devices[64];

template <int D, bool DQ>
static void kernel_setup(DeviceInfo &di) {
  const int vi = (D == 128 ? 2 : 0) + (DQ ? 1 : 0);
  di.attr_err[vi] = cudaFuncSetAttribute(bwd_kernel<D, DQ>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         Cfg<D, DQ>::kSmemBytes);
}

template <int D>
static int launch(const void *q, const void *k, const void *v, const void *o, const void *dO,
                  Params p, int64_t tokens, int stages, cudaStream_t st) {
  CUtensorMap tq, tk, tv, tdo;
  if (!encode_tokens_heads_dim(&tq, q, tokens, p.Hq, D, kTile) ||
      !encode_tokens_heads_dim(&tk, k, tokens, p.Hkv, D, kTile) ||
      !encode_tokens_heads_dim(&tv, v, tokens, p.Hkv, D, kTile) ||
      !encode_tokens_heads_dim(&tdo, dO, tokens, p.Hq, D, kTile))
    return MK_ERR_CUDA;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return MK_ERR_CUDA;
  DeviceInfo &di = g_devices[dev];
  std::call_once(di.once, [&] {
    if (cudaDeviceGetAttribute(&di.sm_count, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      di.sm_count = 0;
    kernel_setup<64, false>(di);
    kernel_setup<64, true>(di);
    kernel_setup<128, false>(di);
    kernel_setup<128, true>(di);
  });
  const int v0 = D == 128 ? 2 : 0;
  if (di.sm_count <= 0 || di.attr_err[v0] != cudaSuccess || di.attr_err[v0 + 1] != cudaSuccess)
    return MK_ERR_CUDA;
  mark_launched(kFamBwd);
  // The dQ kernel computes Delta for its own rows; the separate Delta kernel
  // runs only when Delta is asked for without dQ.
  if ((stages & MK_BWD_DELTA) && !(stages & MK_BWD_DQ)) {
    const dim3 grid((unsigned)((tokens + 15) / 16), (unsigned)p.Hq);
    delta_kernel<D><<<grid, 256, 0, st>>>(
        reinterpret_cast<const uint16_t *>(o), reinterpret_cast<const uint16_t *>(dO),
        const_cast<float *>(p.delta), (int)tokens, p.Hq, p.S, p.varlen);
    if (cudaGetLastError() != cudaSuccess) return MK_ERR_CUDA;
  }
  // dK/dV units: (sequence, key/value head, key tile); dQ units: (sequence,
  // query head, query tile).  Varlen: upper bounds (T + 127 B) / 128 tiles.
  const int64_t tiles = p.varlen ? ((int64_t)p.S + 127LL * p.B) / kTile : (int64_t)p.B * p.n_tiles;
  const mk_attn_tuning tune = current_tuning();
  const int ctas = tune.ctas > 0 ? tune.ctas : di.sm_count;
  p.schedule = tune.schedule;
  Params pk = p, pq = p;
  pk.n_units = (int)(tiles * p.Hkv);
  pq.n_units = (int)(tiles * p.Hq);
  if (stages & MK_BWD_DQ) {
    const int gq = pq.n_units < ctas ? pq.n_units : ctas;
    bwd_kernel<D, true><<<gq, kThreads, Cfg<D, true>::kSmemBytes, st>>>(tq, tk, tv, tdo, pq);
    if (cudaGetLastError() != cudaSuccess) return MK_ERR_CUDA;
  }
  if (stages & MK_BWD_DKDV) {
    const int gk = pk.n_units < ctas ? pk.n_units : ctas;
    bwd_kernel<D, false><<<gk, kThreads, Cfg<D, false>::kSmemBytes, st>>>(tq, tk, tv, tdo, pk);
    if (cudaGetLastError() != cudaSuccess) return MK_ERR_CUDA;
  }
  return MK_OK;
}

}  // namespace bwd

int bwd_take_status() {
  if (!launched(kFamBwd)) return 0;
  int h = 0;
  if (cudaMemcpyFromSymbol(&h, bwd::g_status, sizeof(int)) != cudaSuccess) return MK_ERR_CUDA;
  if (h != 0) {
    const int zero = 0;
    if (cudaMemcpyToSymbol(bwd::g_status, &zero, sizeof(int)) != cudaSuccess) return MK_ERR_CUDA;
  }
  return h;
}

}  // namespace mk

extern "C" {

int64_t mk_attn_bwd_workspace_bytes(int B, int Hq, int S, int varlen) {
  if (B < 1 || Hq < 1 || S < 1) return -1;
  const int64_t rows = varlen ? (int64_t)Hq * S : (int64_t)B * Hq * S;
  return rows * 4;
}

}  // extern "C"

namespace mk {
static int attn_bwd_impl(const void *q, const void *k, const void *v, const void *o,
                         const float *lse, const void *dO, void *dq, void *dk, void *dv, int B,
                         int Hq, int Hkv, int S, int D, int causal, float scale,
                         const int32_t *cu_seqlens, void *workspace, int64_t workspace_bytes,
                         int stages, void *stream) {
  if (stages < 1 || stages > MK_BWD_ALL) return MK_ERR_INVALID_ARG;
  if (!q || !k || !v || !o || !lse || !dO || !dq || !dk || !dv || !workspace)
    return MK_ERR_INVALID_ARG;
  if (B < 1 || Hq < 1 || Hkv < 1 || S < 1 || Hq % Hkv != 0) return MK_ERR_INVALID_ARG;
  if (!std::isfinite(scale)) return MK_ERR_INVALID_ARG;
  if (D != 64 && D != 128) return MK_ERR_UNSUPPORTED;
  if (Hq > 65535) return MK_ERR_UNSUPPORTED;  // the Delta kernel's grid y
  const bool varlen = cu_seqlens != nullptr;
  const int64_t tokens = varlen ? (int64_t)S : (int64_t)B * S;
  if (tokens > INT32_MAX || tokens * Hq > INT32_MAX) return MK_ERR_INVALID_ARG;
  if (workspace_bytes < mk_attn_bwd_workspace_bytes(B, Hq, S, varlen ? 1 : 0))
    return MK_ERR_INVALID_ARG;
  auto misaligned = [](const void *ptr, uintptr_t a) {
    return (reinterpret_cast<uintptr_t>(ptr) & (a - 1)) != 0;
  };
  if (misaligned(q, 16) || misaligned(k, 16) || misaligned(v, 16) || misaligned(o, 16) ||
      misaligned(dO, 16) || misaligned(dq, 16) || misaligned(dk, 16) || misaligned(dv, 16) ||
      misaligned(lse, 4) || misaligned(workspace, 16) || (varlen && misaligned(cu_seqlens, 4)))
    return MK_ERR_ALIGNMENT;
  const int64_t n_tiles = ((int64_t)S + bwd::kTile - 1) / bwd::kTile;
  const int64_t tiles = varlen ? ((int64_t)S + 127LL * B) / bwd::kTile : (int64_t)B * n_tiles;
  if (tiles * Hq > INT32_MAX) return MK_ERR_INVALID_ARG;
  bwd::Params p;
  p.lse = lse;
  p.delta = reinterpret_cast<float *>(workspace);
  p.o = reinterpret_cast<const uint16_t *>(o);
  p.dq = reinterpret_cast<uint16_t *>(dq);
  p.dk = reinterpret_cast<uint16_t *>(dk);
  p.dv = reinterpret_cast<uint16_t *>(dv);
  p.cu_seqlens = cu_seqlens;
  p.B = B;
  p.Hq = Hq;
  p.Hkv = Hkv;
  p.S = S;
  p.G = Hq / Hkv;
  p.causal = causal != 0;
  p.varlen = varlen;
  p.n_tiles = (int)n_tiles;
  p.n_units = 0;
  p.scale = scale;
  p.scale_log2 = scale * 1.4426950408889634f;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (D == 128) return bwd::launch<128>(q, k, v, o, dO, p, tokens, stages, st);
  return bwd::launch<64>(q, k, v, o, dO, p, tokens, stages, st);
}
}  // namespace mk

extern "C" {

int mk_attn_bwd_stages(const void *q, const void *k, const void *v, const void *o,
                       const float *lse, const void *dO, void *dq, void *dk, void *dv, int B,
                       int Hq, int Hkv, int S, int D, int causal, float scale,
                       const int32_t *cu_seqlens, void *workspace, int64_t workspace_bytes,
                       int stages, void *stream) {
  return mk::finish_call(mk::attn_bwd_impl(q, k, v, o, lse, dO, dq, dk, dv, B, Hq, Hkv, S, D,
                                           causal, scale, cu_seqlens, workspace,
                                           workspace_bytes, stages, stream),
                         stream);
}

int mk_attn_bwd(const void *q, const void *k, const void *v, const void *o, const float *lse,
                const void *dO, void *dq, void *dk, void *dv, int B, int Hq, int Hkv, int S,
                int D, int causal, float scale, const int32_t *cu_seqlens, void *workspace,
                int64_t workspace_bytes, void *stream) {
  return mk_attn_bwd_stages(q, k, v, o, lse, dO, dq, dk, dv, B, Hq, Hkv, S, D, causal, scale,
                            cu_seqlens, workspace, workspace_bytes, MK_BWD_DQ | MK_BWD_DKDV,
                            stream);
}

}  // extern "C"
