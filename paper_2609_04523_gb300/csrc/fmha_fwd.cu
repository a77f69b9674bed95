// fmha_fwd.cu -- attention forward pass for GB300 (sm_103a) and its C ABI.
//
// Computes, per sequence b, query head h (key/value head h / (Hq/Hkv)) and
// query row i:  o[i] = softmax(scale * q[i] K^T + causal mask) V  and the
// natural-log row log-sum-exp -- the operation of the paper's Flash Attention
// and GQA Attention kernels (Table 2), under the contract of Section 2.1 and
// Section 3.1 (same inputs and outputs as the reference operation).
//
// Design: persistent CTAs, one per SM.  A work unit is a pair of 128-row query
// tiles (A = rows 256p..256p+127, B = the next 128) of one (sequence, query
// head); both tiles share every K/V block the producer loads.  Roles:
//   warps 0-3   softmax of tile A, thread r owns row r = TMEM lane r
//   warps 4-7   softmax of tile B (same lanes, warp % 4 selects the lane quarter)
//   warp 8      tcgen05 MMA issuer (one thread)
//   warp 9      TMA producer (one thread): maps each of the CTA's units once
//               and publishes it in a small shared-memory ring for the other
//               roles; Q_A, Q_B per unit, then K_j, V_j blocks of 128 keys
//               through an n-stage 128-byte-swizzled ring
//   warps 10-11 idle (they complete the third warpgroup)
// Schedule: units are dealt to the persistent CTAs round by round (snake
// order), heaviest first: fixed length by tile pair, causal varlen by level
// (pair index) from a per-CTA table, which approximates longest-processing-
// time order.  Fixed length and varlen are separate instantiations.
// Registers: the block launches with 168 per thread (384 threads); the third
// warpgroup gives back down to kRegsCtl and the two softmax warpgroups grow to
// kRegsSoftmax, so each SM sub-partition (one warp of each warpgroup) stays
// within its 16K registers: 2 * 208 + 80 = 496 <= 3 * 168.
// TMEM (512 columns): S_A = 0..127, S_B = 128..255, O_A = 256.., O_B = 256+D..
// P_X (bf16) overwrites the first 64 columns of S_X and is the TMEM A operand
// of O_X += P_X V_j; V_j is an MN-major shared-memory B operand.
// MMA issue order per key block j (ping-pong):
//   O_A += P_A(j-1) V_{j-1};  S_A(j) = Q_A K_j^T;  O_B += P_B(j-1) V_{j-1};  S_B(j) = Q_B K_j^T
// so the softmax of one tile runs while the tensor pipe works on the other.
// P_X is published in two halves of 64 keys, each on its own barrier: the
// MMA warp issues P_X V over keys 0..63 while keys 64..127 are exponentiated.
// Because S_X(j) is issued after P_X(j-1) V_{j-1}, every MMA that touches O_X
// has completed when S_X(j) has: the softmax warps rescale O_X in TMEM (lazily,
// only when the row max rises by more than a threshold, 8 in log2 units by
// default) with no extra wait.
// Softmax: base-2 online softmax in fp32 (t = s * scale * log2 e, ex2 on the
// MUFU unit), P rounded to bf16 (RNE); epilogue o = O / l -> bf16,
// lse = ln 2 * (m + log2 l).  Causal tiles visit key blocks 0..qt only and mask
// only the diagonal block; sequence tails are masked by key position.
#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include <atomic>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <mutex>

#include "mk_attn.h"
#include "ptx.cuh"
#include "tma_host.h"

namespace mk {

constexpr int kTile = 128;            // query rows per tile, keys per block
constexpr int kSoftmaxThreads = 128;  // per tile: one thread per query row
constexpr int kMmaWarp = 8;
constexpr int kLoadWarp = 9;
constexpr int kThreads = 384;
constexpr int kLaunchRegs = 168;      // 65536 / 384, rounded down to a multiple of 8
constexpr uint32_t kRegsSoftmax = 208;
constexpr uint32_t kRegsCtl = 80;
static_assert(2 * kRegsSoftmax + kRegsCtl <= 3 * kLaunchRegs, "register split");
constexpr int kBoxCols = 64;          // bf16 elements per 128-byte swizzle row
constexpr int kBoxBytes = kTile * kBoxCols * 2;  // one TMA box: 128 rows x 128 B
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColS = 0;         // S_X at kColS + 128 * X
constexpr uint32_t kColO = 256;       // O_X at kColO + D * X
constexpr int kCuCache = 2048;        // cu_seqlens entries cached in shared memory
constexpr int kMaxLevels = 1024;      // causal varlen: longest-first order up to 1024 tile pairs
                                      // (262144 tokens) per sequence

// MK_SCHED_DYNAMIC: per-launch claim counter and finished-CTA counter, a ring
// of slots so that launches running at once on other streams do not share
// one.  Zero at load; each launch's last CTA puts its slot back to zero.
constexpr int kSchedSlots = 1024;
__device__ unsigned g_sched_next[kSchedSlots];
__device__ unsigned g_sched_done[kSchedSlots];
__device__ int g_status = 0;               // MK_ERR_TIMEOUT once a wait ran out

template <int D>
struct KernelCfg {
  static_assert(D == 64 || D == 128, "head dimension 64 or 128");
  static constexpr int kStages = (D == 128) ? 2 : 4;
  static constexpr int kHalves = D / kBoxCols;      // swizzle boxes per tile
  static constexpr int kTileBytes = kTile * D * 2;  // one Q, K or V tile
  // D = 64: o is staged per warp (32 rows x 64 columns, 4 KB, 128-byte
  // swizzle) and written by TMA stores; 32 KB for the eight softmax warps.
  // At D = 128 there is no room for it, and the rows are stored directly.
  static constexpr bool kStageO = (D == 64);
  static constexpr int kOffQ = 0;                   // Q_A, then Q_B
  static constexpr int kOffK = 2 * kTileBytes;
  static constexpr int kOffV = kOffK + kStages * kTileBytes;
  static constexpr int kOffStage = kOffV + kStages * kTileBytes;
  static constexpr int kOffCu = kOffStage + (kStageO ? 8 * 4096 : 0);
  static constexpr int kOffLvl = kOffCu + kCuCache * 4;  // (kMaxLevels + 2) ints
  static constexpr int kOffCtl = kOffLvl + ((kMaxLevels + 2) * 4 + 15) / 16 * 16;
  static constexpr int kSmemBytes = kOffCtl + 512 + 1024;  // + control block + alignment slack
  static_assert(kSmemBytes <= 232448, "shared memory per block");
};

struct Unit {
  int valid;
  int b, hq, pair;
  int seq_start, len;
};

constexpr int kUnitRing = 4;  // unit descriptors published by the producer warp

struct SharedCtl {
  uint64_t bar_q_full[2], bar_q_empty[2];
  uint64_t bar_kv_full[4], bar_kv_empty[4];  // K/V slots
  uint64_t bar_s_full[2];
  uint64_t bar_p_full[2][2];  // [tile][half]: P_X keys 0..63, then keys 64..127
  uint64_t bar_o_final[2];
  uint64_t bar_mma_drained;
  // The producer maps each of the CTA's units once and publishes it here; the
  // MMA and softmax warps read it.  The producer is at most two units ahead of
  // the slowest reader (it loads a unit's Q only after the MMA warp has issued
  // the previous unit's last S, which needs the softmax's last P of the unit
  // before that), so four entries are never overwritten while still unread.
  uint64_t bar_unit[kUnitRing];
  Unit unit_ring[kUnitRing];  // valid = 0: no more units
  uint32_t tmem_base;
  int abort;
  int lvl_P;   // causal varlen: most tile pairs of any sequence
  int lvl_ok;  // causal varlen: the longest-first level table is valid
};
static_assert(sizeof(SharedCtl) <= 512, "control block");

struct Params {
  uint16_t *o;              // bf16 bits
  float *lse;
  const int32_t *cu_seqlens;
  int B, Hq, Hkv, S;        // S = tokens per sequence, or total tokens T (varlen)
  int group;                // Hq / Hkv
  int causal, varlen;
  int n_pairs;              // fixed length: query-tile pairs per sequence
  int n_units;              // fixed: exact; varlen: upper bound
  float scale_log2;         // scale * log2(e)
  int o_align32;            // o is 32-byte aligned: 256-bit stores in the epilogue
  int stall_first_slot;     // failure-path test: the producer loads nothing
  int schedule;             // MK_SCHED_*: units over the persistent CTAs
  float rescale_log2;       // lazy O rescale threshold (log2 units)
  int sched_slot;           // MK_SCHED_DYNAMIC: this launch's counter slot
};

__device__ __forceinline__ int clamp_tok(int x, int T) { return x < 0 ? 0 : (x > T ? T : x); }

__device__ __forceinline__ int pairs_of_len(int L) { return ((L + kTile - 1) / kTile + 1) / 2; }

// Token range [s0, s1) of varlen sequence b; cu_seqlens entries are clamped
// to [0, T] and a negative length reads as zero.
__device__ __forceinline__ void seq_bounds(const Params &p, const int *cu_smem, int b, int &s0,
                                           int &s1) {
  const int T = p.S;
  s0 = clamp_tok(b < kCuCache ? cu_smem[b] : p.cu_seqlens[b], T);
  s1 = clamp_tok(b + 1 < kCuCache ? cu_smem[b + 1] : p.cu_seqlens[b + 1], T);
  if (s1 < s0) s1 = s0;
}

// Causal varlen schedule table (shared memory), for longest-first order: with
// N(k) = number of sequences with at least k tile pairs and P the most pairs
// of any sequence, lvl[k] = M(k) = N(k) + N(k+1) + ... + N(P) for k = 1..P+1.
// Level k (k = P first, down to 1) holds pair k-1 of every sequence with at
// least k pairs, for every head: Hq * N(k) units, the unit cost growing with k.
struct Sched {
  const int *lvl;
  int P;
  int ok;
};

// Maps unit index u to (sequence, query head, tile pair).  Must be called by
// all 32 lanes of a warp (varlen uses warp ballots); every lane gets the result.
// Only the producer warp maps units; the other roles read its unit ring.
// Fixed length: units are ordered by pair, heaviest first when causal, so that
// the static round-robin over CTAs approximates longest-processing-time order;
// consecutive units share a K/V head (GQA groups are contiguous).  Causal
// varlen with a valid table: levels k = P .. 1 in turn, each in sequence order
// then head order, which again puts the heaviest units first.  Otherwise varlen
// unit u is pair u / Hq of head u % Hq in sequence order.
template <bool VL>
__device__ __forceinline__ Unit map_unit(const Params &p, const int *cu_smem, const Sched &sc,
                                         int u) {
  Unit w;
  if constexpr (!VL) {
    const int per_level = p.B * p.Hq;
    const int level = u / per_level;
    const int rem = u - level * per_level;
    w.valid = u < p.n_units;
    w.hq = rem % p.Hq;
    w.b = rem / p.Hq;
    w.pair = p.causal ? (p.n_pairs - 1 - level) : level;
    w.seq_start = w.b * p.S;
    w.len = p.S;
    return w;
  } else {
  const int lane = lane_id();
  w.valid = 0;
  w.b = w.pair = w.seq_start = w.len = w.hq = 0;
  if (sc.ok) {
    // Level k: the largest k in [1, P] with Hq * M(k) > u (M is non-increasing).
    const int64_t uu = u;
    if (sc.P < 1 || uu >= (int64_t)p.Hq * sc.lvl[1]) return w;
    int lo = 1, hi = sc.P;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if ((int64_t)p.Hq * sc.lvl[mid] > uu) lo = mid; else hi = mid - 1;
    }
    const int k = lo;
    const int64_t rem = uu - (int64_t)p.Hq * sc.lvl[k + 1];
    int i = (int)(rem / p.Hq);  // the i-th sequence (in order) with at least k pairs
    w.hq = (int)(rem - (int64_t)i * p.Hq);
    w.pair = k - 1;
    for (int base = 0; base < p.B; base += 32) {
      const int b = base + lane;
      int s0 = 0, s1 = 0;
      if (b < p.B) seq_bounds(p, cu_smem, b, s0, s1);
      const unsigned m = __ballot_sync(0xffffffffu, b < p.B && pairs_of_len(s1 - s0) >= k);
      const int c = __popc(m);
      if (i < c) {
        unsigned mm = m;
        for (int t = 0; t < i; ++t) mm &= mm - 1;  // drop the i lowest set bits
        const int src = __ffs(mm) - 1;
        w.valid = 1;
        w.b = base + src;
        w.seq_start = __shfl_sync(0xffffffffu, s0, src);
        w.len = __shfl_sync(0xffffffffu, s1 - s0, src);
        break;
      }
      i -= c;
    }
    return w;
  }
  const int rank = u / p.Hq;
  w.hq = u % p.Hq;
  int carry = 0;
  for (int base = 0; base < p.B; base += 32) {
    const int b = base + lane;
    int s0 = 0, s1 = 0, np = 0;
    if (b < p.B) {
      seq_bounds(p, cu_smem, b, s0, s1);
      np = pairs_of_len(s1 - s0);
    }
    int incl = np;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl += y;
    }
    const int excl = incl - np;
    const bool mine = (b < p.B) && rank >= carry + excl && rank < carry + incl;
    const unsigned m = __ballot_sync(0xffffffffu, mine);
    if (m) {
      const int src = __ffs(m) - 1;
      w.valid = 1;
      w.b = base + src;
      w.pair = rank - carry - __shfl_sync(0xffffffffu, excl, src);
      w.seq_start = __shfl_sync(0xffffffffu, s0, src);
      w.len = __shfl_sync(0xffffffffu, s1 - s0, src);
      break;
    }
    carry += __shfl_sync(0xffffffffu, incl, 31);
  }
  return w;
  }
}

// In place, one warp: a[i] = a[i] + a[i+1] + ... + a[n-1] for i in [0, n).
__device__ __forceinline__ void warp_suffix_sum(int *a, int n) {
  const int lane = lane_id();
  const int chunk = (n + 31) / 32;
  const int lo = lane * chunk, hi = min(n, lo + chunk);
  int tot = 0;
  for (int i = hi - 1; i >= lo; --i) {
    tot += a[i];
    a[i] = tot;
  }
  int incl = tot;  // this lane's chunk and those of the lanes above it
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int y = __shfl_down_sync(0xffffffffu, incl, off);
    if (lane + off < 32) incl += y;
  }
  const int above = incl - tot;
  for (int i = lo; i < hi; ++i) a[i] += above;
  __syncwarp();
}

// Key blocks visited by tile X (0 = A, 1 = B) of a unit; 0 if the tile lies
// past the end of the sequence.
__device__ __forceinline__ int tile_blocks(const Params &p, const Unit &w, int X) {
  const int qt = 2 * w.pair + X;
  if (qt * kTile >= w.len) return 0;
  const int n_kb = (w.len + kTile - 1) / kTile;
  return p.causal ? min(qt + 1, n_kb) : n_kb;
}

// Unit processed by this CTA in round k.  Units are numbered heaviest first
// (fixed-length causal).  The default (snake) alternates the direction of the
// rounds over the CTAs (CTA c takes unit kG + c in even rounds and
// kG + G - 1 - c in odd ones), which balances the per-CTA sums of decreasing
// unit costs far better than plain round-robin; blocked gives each CTA a
// contiguous run of units.  A unit index >= n_units means no unit.
__device__ __forceinline__ int unit_of_round(int k, int schedule, int n_units) {
  const int G = gridDim.x, c = blockIdx.x;
  if (schedule == MK_SCHED_BLOCKED) {
    const int per = (n_units + G - 1) / G;
    return k < per ? c * per + k : n_units;
  }
  if (schedule == MK_SCHED_ROUND_ROBIN) return k * G + c;
  return (k & 1) ? (k + 1) * G - 1 - c : k * G + c;
}

// MK_SCHED_DYNAMIC, at CTA exit (one thread, after the CTA's last claim): the
// launch's last CTA puts its counter slot back to zero.  Out of line, so that
// nothing of it is held in registers across the kernel.
__device__ __noinline__ void sched_release(int slot) {
  __threadfence();
  if (atomicAdd(&g_sched_done[slot], 1u) == gridDim.x - 1) {
    atomicExch(&g_sched_next[slot], 0u);
    atomicExch(&g_sched_done[slot], 0u);
  }
}

// Bounded wait that ignores the abort flag: used only at teardown to let
// operations already in flight land before the CTA releases its resources.
__device__ __forceinline__ void drain_wait(uint64_t *bar, uint32_t parity) {
  int local_abort = 0;
  mbar_wait(bar, parity, &local_abort);
}

template <int D, bool VL>
__global__ void __launch_bounds__(kThreads, 1)
    mk_attn_fwd_persistent(const __grid_constant__ CUtensorMap tm_q,
                    const __grid_constant__ CUtensorMap tm_k,
                    const __grid_constant__ CUtensorMap tm_v,
                    const __grid_constant__ CUtensorMap tm_o, const Params p) {
  using C = KernelCfg<D>;
  constexpr int NS = C::kStages;

  extern __shared__ uint8_t smem_raw[];
  // 1024-byte alignment for the 128-byte-swizzle atoms.
  const uint32_t raw_addr = smem_addr(smem_raw);
  uint8_t *smem = smem_raw + ((1024u - (raw_addr & 1023u)) & 1023u);
  SharedCtl *ctl = reinterpret_cast<SharedCtl *>(smem + C::kOffCtl);
  int *cu_smem = reinterpret_cast<int *>(smem + C::kOffCu);
  const uint32_t sQ = smem_addr(smem + C::kOffQ);
  const uint32_t sK = smem_addr(smem + C::kOffK);
  const uint32_t sV = smem_addr(smem + C::kOffV);
  const int warp = threadIdx.x / 32;

  int *lvl = reinterpret_cast<int *>(smem + C::kOffLvl);
  if constexpr (VL) {
    const int n = min(p.B + 1, kCuCache);
    for (int i = threadIdx.x; i < n; i += kThreads) cu_smem[i] = p.cu_seqlens[i];
  }
  if (VL && p.causal) {
    // Longest-first schedule table: a histogram of tile pairs per sequence,
    // then two suffix sums (see Sched).
    for (int i = threadIdx.x; i < kMaxLevels + 2; i += kThreads) lvl[i] = 0;
    if (threadIdx.x == 0) ctl->lvl_P = 0;
    __syncthreads();
    for (int b = threadIdx.x; b < p.B; b += kThreads) {
      int s0, s1;
      seq_bounds(p, cu_smem, b, s0, s1);
      const int np = pairs_of_len(s1 - s0);
      atomicMax(&ctl->lvl_P, np);
      atomicAdd(&lvl[min(np, kMaxLevels + 1)], 1);
    }
    __syncthreads();
    if (warp == 0) {
      const int P = ctl->lvl_P;
      if (P <= kMaxLevels) {
        warp_suffix_sum(lvl, P + 1);  // lvl[k] = N(k)
        warp_suffix_sum(lvl, P + 1);  // lvl[k] = M(k); lvl[P + 1] stays 0
      }
      if (lane_id() == 0) ctl->lvl_ok = P <= kMaxLevels;
    }
  } else if (threadIdx.x == 0) {
    ctl->lvl_ok = 0;
    ctl->lvl_P = 0;
  }
  if (threadIdx.x == 0) {
    for (int x = 0; x < 2; ++x) {
      mbar_init(&ctl->bar_q_full[x], 1);
      mbar_init(&ctl->bar_q_empty[x], 1);
      mbar_init(&ctl->bar_s_full[x], 1);
      mbar_init(&ctl->bar_p_full[x][0], kSoftmaxThreads);
      mbar_init(&ctl->bar_p_full[x][1], kSoftmaxThreads);
      mbar_init(&ctl->bar_o_final[x], 1);
    }
    for (int s = 0; s < NS; ++s) {
      mbar_init(&ctl->bar_kv_full[s], 1);
      mbar_init(&ctl->bar_kv_empty[s], 1);
    }
    mbar_init(&ctl->bar_mma_drained, 1);
    for (int e = 0; e < kUnitRing; ++e) mbar_init(&ctl->bar_unit[e], 1);
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
  const Sched sched = {lvl, ctl->lvl_P, ctl->lvl_ok};

  if (warp >= 8) {
    // Third warpgroup: producer, MMA issuer and two idle warps.  All four
    // warps give registers back at this one instruction.
    setmaxnreg_dec<kRegsCtl>();
    // The producer and MMA warps run their loops and waits with all 32 lanes
    // converged; one lane chosen by elect.sync issues each TMA / tcgen05
    // instruction, so the bookkeeping and descriptors stay warp-uniform.
    //
    // K/V slots: iteration j of a unit (j = 0..n, n = key blocks of the unit)
    // uses slot (global iteration) % NS, which holds K_j (for S(j) = Q K_j^T,
    // j < n) and V_{j-1} (for O += P(j-1) V_{j-1}, j >= 1).  One full and one
    // empty barrier per slot: one wait and one commit per iteration.
    if (warp == kLoadWarp) {
      // ---------------------------------------------------------- producer
      if (elect_one()) {
        tma_prefetch_desc(&tm_q);
        tma_prefetch_desc(&tm_k);
        tma_prefetch_desc(&tm_v);
      }
      const uint64_t pol_q = l2_policy_evict_first();
      const uint64_t pol_kv = l2_policy_evict_last();
      uint32_t q_iter = 0, it = 0, n_pub = 0;
      uint32_t q_issued[2] = {0, 0};  // Q loads issued per tile, for the teardown drain
      auto publish = [&](const Unit &w) {
        const int e = n_pub % kUnitRing;
        if (elect_one()) {
          ctl->unit_ring[e] = w;
          mbar_arrive(&ctl->bar_unit[e]);  // release: the entry is visible to the waiters
        }
        __syncwarp();
        ++n_pub;
      };
      // MK_SCHED_DYNAMIC: the first unit is blockIdx.x; each later one is
      // claimed (lane 0) two key blocks before the current unit's loads end,
      // and the claim's result is read at the next unit, so its latency is
      // hidden.  A unit without a claim point claims at the top of the loop.
      unsigned claim = 0;
      bool claimed = false;
      bool ok = true;
      for (int k = 0; ok; ++k) {
        int u;
        if (p.schedule == MK_SCHED_DYNAMIC) {
          if (k == 0) {
            u = blockIdx.x;
          } else {
            if (!claimed && lane_id() == 0) claim = atomicAdd(&g_sched_next[p.sched_slot], 1u);
            u = (int)gridDim.x + (int)__shfl_sync(0xffffffffu, claim, 0);
            claimed = false;
          }
          if (u >= p.n_units) break;
        } else {
          if (k * (int)gridDim.x >= p.n_units) break;
          u = unit_of_round(k, p.schedule, p.n_units);
          if (u >= p.n_units) continue;
        }
        const Unit w = map_unit<VL>(p, cu_smem, sched, u);
        if (!w.valid) continue;
        publish(w);
        // Failure-path test: the first unit is published but nothing is
        // loaded, so the MMA warp's bounded wait for its Q runs out.
        if (p.stall_first_slot) break;
        const int hkv = w.hq / p.group;
        const int n_blk = max(tile_blocks(p, w, 0), tile_blocks(p, w, 1));
        // Q_A, then K_0, then Q_B: the unit's first S (tile A) needs only the
        // first two, so it starts a tile-load earlier.
        auto load_q = [&](int x) {
          ok = mbar_wait_all(&ctl->bar_q_empty[x], (q_iter & 1) ^ 1, abort);
          if (!ok) return;
          if (elect_one()) {
            mbar_arrive_expect_tx(&ctl->bar_q_full[x], C::kTileBytes);
#pragma unroll
            for (int h = 0; h < C::kHalves; ++h)
              tma_load_3d(smem + C::kOffQ + x * C::kTileBytes + h * kBoxBytes, &tm_q,
                          &ctl->bar_q_full[x], h * kBoxCols, w.hq,
                          w.seq_start + (2 * w.pair + x) * kTile, pol_q);
          }
          __syncwarp();
          ++q_issued[x];
        };
        load_q(0);
        if (!ok) break;
        const int claim_j = n_blk > 2 ? n_blk - 2 : 0;
        for (int j = 0; j <= n_blk; ++j) {
          if (p.schedule == MK_SCHED_DYNAMIC && j == claim_j) {
            if (lane_id() == 0) claim = atomicAdd(&g_sched_next[p.sched_slot], 1u);
            claimed = true;
          }
          const int s = it % NS;
          ok = mbar_wait_all(&ctl->bar_kv_empty[s], ((it / NS) & 1) ^ 1, abort);
          if (!ok) break;
          if (elect_one()) {
            const uint32_t bytes = (j < n_blk ? C::kTileBytes : 0) + (j > 0 ? C::kTileBytes : 0);
            mbar_arrive_expect_tx(&ctl->bar_kv_full[s], bytes);
            if (j < n_blk) {
#pragma unroll
              for (int h = 0; h < C::kHalves; ++h)
                tma_load_3d(smem + C::kOffK + s * C::kTileBytes + h * kBoxBytes, &tm_k,
                            &ctl->bar_kv_full[s], h * kBoxCols, hkv, w.seq_start + j * kTile,
                            pol_kv);
            }
            if (j > 0) {
#pragma unroll
              for (int h = 0; h < C::kHalves; ++h)
                tma_load_3d(smem + C::kOffV + s * C::kTileBytes + h * kBoxBytes, &tm_v,
                            &ctl->bar_kv_full[s], h * kBoxCols, hkv,
                            w.seq_start + (j - 1) * kTile, pol_kv);
            }
          }
          __syncwarp();
          ++it;
          if (j == 0) {
            load_q(1);
            if (!ok) break;
            ++q_iter;
          }
        }
      }
      {
        const Unit none = {};
        publish(none);
      }
      // Teardown: every load issued must land before the CTA exits.  For each
      // slot the last issued phase is waited for (earlier phases precede it).
      for (int x = 0; x < 2; ++x)
        if (q_issued[x] > 0) drain_wait(&ctl->bar_q_full[x], (q_issued[x] - 1) & 1);
      for (uint32_t n = (it > (uint32_t)NS ? it - NS : 0); n < it; ++n)
        drain_wait(&ctl->bar_kv_full[n % NS], (n / NS) & 1);
    } else if (warp == kMmaWarp) {
      // ---------------------------------------------------------- MMA issuer
      constexpr uint32_t idesc_qk = idesc_bf16_f32(kTile, kTile, false, false);
      constexpr uint32_t idesc_pv = idesc_bf16_f32(kTile, D, false, true);
      // Q and K are K-major (head dim contiguous); 16 bf16 = 32 B per MMA step
      // inside a 128-byte swizzle row, 8-row groups 1024 B apart.  V is the
      // MN-major B operand of P V: 8-key groups 1024 B apart (SBO), 64-column
      // chunks of the head dimension one TMA box apart (LBO, unused at D = 64).
      // The descriptor's address field is addr >> 4, so stepping the start
      // address by b bytes adds b >> 4 to the descriptor.
      constexpr uint32_t kVLbo = (D > kBoxCols) ? kBoxBytes : 1024;
      const uint64_t dq0 = sdesc_sw128(sQ, 16, 1024);
      const uint64_t dk0 = sdesc_sw128(sK, 16, 1024);
      const uint64_t dv0 = sdesc_sw128(sV, kVLbo, 1024);
      constexpr uint64_t kTileStep = C::kTileBytes >> 4;
      uint32_t q_iter = 0, it = 0;
      uint32_t p_cnt[2] = {0, 0};
      bool ok = true;

      // S_X = Q_X K^T for the K tile in slot s (elected lane only).
      auto issue_s = [&](int x, int s) {
        const uint64_t a0 = dq0 + x * kTileStep;
        const uint64_t b0 = dk0 + s * kTileStep;
        const uint32_t d_tmem = tmem + kColS + x * 128;
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t off = ((kk >> 2) * kBoxBytes + (kk & 3) * 32) >> 4;
          umma_ss(d_tmem, a0 + off, b0 + off, idesc_qk, kk > 0 ? 1u : 0u);
        }
        umma_commit(&ctl->bar_s_full[x]);
      };
      // O_X (+)= P_X V over keys 64 * half .. 64 * half + 63 of the V tile in
      // slot s (elected lane only).
      auto issue_pv = [&](int x, int s, int half, bool first) {
        const uint64_t b0 = dv0 + s * kTileStep;
        const uint32_t d_tmem = tmem + kColO + x * D;
        const uint32_t a_tmem = tmem + kColS + x * 128;
#pragma unroll
        for (int k4 = 0; k4 < kTile / 32; ++k4) {
          const int kk = half * (kTile / 32) + k4;
          umma_ts(d_tmem, a_tmem + kk * 8, b0 + (uint64_t)(kk * 128), idesc_pv,
                  (!first || kk > 0) ? 1u : 0u);
        }
      };

      for (uint32_t n_read = 0; ok; ++n_read) {
        ok = mbar_wait_all(&ctl->bar_unit[n_read % kUnitRing], (n_read / kUnitRing) & 1, abort);
        if (!ok) break;
        const Unit w = ctl->unit_ring[n_read % kUnitRing];
        if (!w.valid) break;
        const int nx[2] = {tile_blocks(p, w, 0), tile_blocks(p, w, 1)};
        const int n_blk = max(nx[0], nx[1]);
        const int n_min = min(nx[0], nx[1]);
        // Generic iteration j: any mix of P V and S per tile (unit edges).
        auto edge_iteration = [&](int j) {
          const int s = it % NS;
          ok = mbar_wait_all(&ctl->bar_kv_full[s], (it / NS) & 1, abort);
#pragma unroll
          for (int x = 0; x < 2; ++x) {
            if (!ok) break;
            // Iteration 0 waits for Q_X (loaded after K_0 for tile B), also
            // when the tile has no key block: its Q_empty commit below must
            // not release a load still in flight.
            if (j == 0) {
              ok = mbar_wait_all(&ctl->bar_q_full[x], q_iter & 1, abort);
              if (!ok) break;
            }
            const bool do_pv = j > 0 && j - 1 < nx[x];
            const bool do_s = j < nx[x];
            if (do_pv) {
              ok = mbar_wait_all(&ctl->bar_p_full[x][0], p_cnt[x] & 1, abort);
              if (!ok) break;
              tc_fence_after_sync();
              if (elect_one()) issue_pv(x, s, 0, j == 1);
              __syncwarp();
              ok = mbar_wait_all(&ctl->bar_p_full[x][1], p_cnt[x] & 1, abort);
              ++p_cnt[x];
              if (!ok) break;
            }
            tc_fence_after_sync();
            if (elect_one()) {
              if (do_pv) {
                issue_pv(x, s, 1, false);
                if (j == nx[x]) umma_commit(&ctl->bar_o_final[x]);
              }
              if (do_s) issue_s(x, s);
              if (j == nx[x] - 1 || (j == 0 && nx[x] == 0))
                umma_commit(&ctl->bar_q_empty[x]);  // Q_X no longer read
            }
            __syncwarp();
          }
          if (!ok) return;
          if (elect_one()) umma_commit(&ctl->bar_kv_empty[s]);
          __syncwarp();
          ++it;
        };
        // Iteration 0 (S only), then the steady iterations 1 .. n_min - 1 in
        // which both tiles do P V and S (no per-tile conditions), then the
        // iterations in which only the longer tile still works.
        if (ok) edge_iteration(0);
        for (int j = 1; ok && j < n_min; ++j) {
          const int s = it % NS;
          ok = mbar_wait_all(&ctl->bar_kv_full[s], (it / NS) & 1, abort);
#pragma unroll
          for (int x = 0; x < 2; ++x) {
            if (!ok) break;
            // P_X(j-1) arrives in two halves; the first half's MMAs run
            // while the softmax computes the second.
            ok = mbar_wait_all(&ctl->bar_p_full[x][0], p_cnt[x] & 1, abort);
            if (!ok) break;
            tc_fence_after_sync();
            if (elect_one()) issue_pv(x, s, 0, j == 1);
            __syncwarp();
            ok = mbar_wait_all(&ctl->bar_p_full[x][1], p_cnt[x] & 1, abort);
            ++p_cnt[x];
            if (!ok) break;
            tc_fence_after_sync();
            if (elect_one()) {
              issue_pv(x, s, 1, false);
              issue_s(x, s);
            }
            __syncwarp();
          }
          if (!ok) break;
          if (elect_one()) umma_commit(&ctl->bar_kv_empty[s]);
          __syncwarp();
          ++it;
        }
        if (ok && n_min >= 2) {
          // The shorter tile's last S (j = n_min - 1) was issued in the loop above.
          if (elect_one()) {
#pragma unroll
            for (int x = 0; x < 2; ++x)
              if (nx[x] == n_min) umma_commit(&ctl->bar_q_empty[x]);
          }
          __syncwarp();
        }
        for (int j = max(n_min, 1); ok && j <= n_blk; ++j) edge_iteration(j);
        ++q_iter;
      }
      // Teardown: all MMAs issued by this warp complete before TMEM is freed.
      if (elect_one()) umma_commit(&ctl->bar_mma_drained);
      __syncwarp();
      drain_wait(&ctl->bar_mma_drained, 0);
    }
  } else {
    // ------------------------------------------------------------ softmax
    // Both softmax warpgroups take their larger register budget here.
    setmaxnreg_inc<kRegsSoftmax>();
    const int X = warp / 4;                       // tile of this warpgroup
    const int r = threadIdx.x % kSoftmaxThreads;  // row within the tile == TMEM lane
    const uint32_t t_row = tmem + ((uint32_t)((warp % 4) * 32) << 16);
    const uint32_t t_s = t_row + kColS + X * 128;
    const uint32_t t_o = t_row + kColO + X * D;
    // o is written once and not read again by this kernel: its lines go first
    // when L2 needs room, so the K/V blocks other query tiles still read stay.
    const uint64_t pol_o = l2_policy_evict_first();
    const float c2 = p.scale_log2;
    const bool neg_scale = c2 < 0.f;
    const float c2a = fmaxf(fabsf(c2), 1.17549435e-38f);  // |c2|, at least FLT_MIN
    uint32_t s_cnt = 0, o_cnt = 0;
    bool ok = true;

    for (uint32_t n_read = 0; ok; ++n_read) {
      ok = mbar_wait_all(&ctl->bar_unit[n_read % kUnitRing], (n_read / kUnitRing) & 1, abort);
      if (!ok) break;
      const Unit w = ctl->unit_ring[n_read % kUnitRing];
      if (!w.valid) break;
      const int n_blk = tile_blocks(p, w, X);
      if (n_blk == 0) continue;
      const int qt = 2 * w.pair + X;
      const int qpos = qt * kTile + r;
      const bool row_valid = qpos < w.len;
      const int key_limit = p.causal ? min(w.len, qpos + 1) : w.len;  // keys [0, limit)
      float m_run = -INFINITY;  // running row max, base-2 units
      float l_run = 0.f;        // running row sum relative to m_run

      for (int j = 0; j < n_blk; ++j) {
        ok = mbar_wait_all(&ctl->bar_s_full[X], s_cnt & 1, abort);
        ++s_cnt;
        if (!ok) break;
        tc_fence_after_sync();
        const bool needs_mask = (j * kTile + kTile > w.len) || (p.causal && j == qt);
        const int lim = key_limit - j * kTile;
        // s = S_X(j) row in the form the exponential takes: negated when the
        // scale is negative (t = s * c2 = (-s) * |c2|), hidden keys at -inf.
        // With c2a = max(|c2|, FLT_MIN) > 0 a hidden key gives p = 2^-inf = 0
        // and the row max is c2a * max(s).  (For c2 = 0, every visible
        // s * FLT_MIN is at most a denormal, which ex2.approx.ftz reads as 0:
        // p = 1, exactly as for a zero scale.)  The exponential loop below is
        // branch-free: a branch inside it would stop the scheduler from
        // overlapping the MUFU latencies of consecutive keys.
        auto load_scores = [&](float (&s)[kTile]) {
          uint32_t raw[kTile];
          tmem_ld_32x32b_x128(t_s, raw);
          tmem_ld_wait();
          reg_fence_n(raw);
#pragma unroll
          for (int c = 0; c < kTile; ++c) s[c] = __uint_as_float(raw[c]);
          if (neg_scale) {
#pragma unroll
            for (int c = 0; c < kTile; ++c) s[c] = -s[c];
          }
          if (needs_mask) {
#pragma unroll
            for (int c = 0; c < kTile; ++c) s[c] = (c < lim) ? s[c] : -INFINITY;
          }
        };
        float s[kTile];
        load_scores(s);
        float mx0 = fmaxf(s[0], s[1]), mx1 = fmaxf(s[2], s[3]);
        float mx2 = fmaxf(s[4], s[5]), mx3 = fmaxf(s[6], s[7]);
#pragma unroll
        for (int c = 8; c < kTile; c += 8) {
          mx0 = fmax3(mx0, s[c], s[c + 1]);
          mx1 = fmax3(mx1, s[c + 2], s[c + 3]);
          mx2 = fmax3(mx2, s[c + 4], s[c + 5]);
          mx3 = fmax3(mx3, s[c + 6], s[c + 7]);
        }
        mx0 = fmaxf(fmax3(mx0, mx1, mx2), mx3);
        const float m_new = fmaxf(m_run, mx0 * c2a);
        // Lazy rescaling: keep the old reference max unless the new one exceeds
        // it by more than the threshold.  Exact either way, because O and l
        // always share the same reference max.
        const bool rescale = m_new > m_run + p.rescale_log2;
        float alpha = 1.f;
        if (rescale) {
          alpha = ex2_approx(m_run - m_new);  // 0 when m_run = -inf
          l_run *= alpha;
          m_run = m_new;
        }
        if (j > 0 && __any_sync(0xffffffffu, rescale)) {
          // O_X already holds blocks 0..j-1: P_X(j-1) V_{j-1} was issued before
          // S_X(j), and S_X(j) has completed.  The scores are read again
          // afterwards rather than kept live across this (rare) step.
#pragma unroll
          for (int c = 0; c < D / 32; ++c) {
            uint32_t o_raw[32];
            tmem_ld_32x32b_x32(t_o + c * 32, o_raw);
            tmem_ld_wait();
            reg_fence(o_raw);
#pragma unroll
            for (int e = 0; e < 32; ++e)
              o_raw[e] = __float_as_uint(__uint_as_float(o_raw[e]) * alpha);
            tmem_st_32x32b_x32(t_o + c * 32, o_raw);
          }
          tmem_st_wait();
          load_scores(s);
        }
        // p = 2^(s * c2a - m): one FMA and one MUFU ex2 per key.
        const float neg_m = (m_run == -INFINITY) ? 0.f : -m_run;
        float sum0 = 0.f, sum1 = 0.f, sum2 = 0.f, sum3 = 0.f;
        // P_X(j) (bf16, 64 columns) overwrites the first half of S_X(j), in
        // two halves of 64 keys (32 columns), each announced on its own
        // barrier so that the MMA warp starts O_X += P V on keys 0..63 while
        // keys 64..127 are still being exponentiated.
#pragma unroll
        for (int half = 0; half < 2; ++half) {
          uint32_t pk[32];
#pragma unroll
          for (int c = half * 64; c < half * 64 + 64; c += 4) {
            float a0, a1, a2, a3;
            ffma2_bcast(a0, a1, s[c], s[c + 1], c2a, neg_m);
            ffma2_bcast(a2, a3, s[c + 2], s[c + 3], c2a, neg_m);
            const float p0 = ex2_approx(a0), p1 = ex2_approx(a1);
            const float p2 = ex2_approx(a2), p3 = ex2_approx(a3);
            fadd2_acc(sum0, sum1, p0, p1);
            fadd2_acc(sum2, sum3, p2, p3);
            pk[(c % 64) / 2] = pack_bf16x2(p0, p1);
            pk[(c % 64) / 2 + 1] = pack_bf16x2(p2, p3);
          }
          tmem_st_32x32b_x32(t_s + half * 32, pk);
          tmem_st_wait();
          tc_fence_before_sync();
          mbar_arrive(&ctl->bar_p_full[X][half]);
        }
        l_run += (sum0 + sum1) + (sum2 + sum3);
      }
      if (!ok) break;

      // ---------------------------------------------------------- epilogue
      ok = mbar_wait_all(&ctl->bar_o_final[X], o_cnt & 1, abort);
      ++o_cnt;
      if (!ok) break;
      tc_fence_after_sync();
      const float inv_l = 1.f / l_run;
      const int64_t tok = (int64_t)w.seq_start + qpos;
      // Check build: the row lies inside o and lse (tokens x Hq rows).
      const bool row_store =
          row_valid &&
          dbg_in_range(tok, VL ? (int64_t)p.S : (int64_t)p.B * p.S, &g_status) &&
          dbg_in_range(w.hq, p.Hq, &g_status);
      // D = 64, a tile that lies inside its sequence: each warp stages its 32
      // rows in the 128-byte swizzle and stores them with one TMA store, which
      // writes whole lines and keeps the stores off the load/store pipe.  A
      // tile cut by the end of its sequence keeps the per-row stores.
      const int64_t tok0 = (int64_t)w.seq_start + qt * kTile;
      const bool tile_store =
          C::kStageO && qt * kTile + kTile <= w.len &&
          dbg_in_range(tok0 + kTile - 1, VL ? (int64_t)p.S : (int64_t)p.B * p.S, &g_status) &&
          dbg_in_range(w.hq, p.Hq, &g_status);
      if (tile_store) {
        const int wq = warp % 4;
        uint8_t *wbox = smem + C::kOffStage + (X * 4 + wq) * 4096;
        const uint32_t row_a = smem_addr(wbox) + lane_id() * 128;
        uint32_t o_raw[2][32];
        tmem_ld_32x32b_x32(t_o, o_raw[0]);
        tmem_ld_32x32b_x32(t_o + 32, o_raw[1]);
        // The box is free once this warp's previous store has read it.
        if (lane_id() == 0) bulk_wait_group_read_all();
        __syncwarp();
        tmem_ld_wait();
#pragma unroll
        for (int cc = 0; cc < 2; ++cc) {
          reg_fence(o_raw[cc]);
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            // 16-byte chunk j = 4 cc + e of this row goes to position j ^ (row % 8).
            const uint32_t a = row_a + ((((cc * 4 + e) ^ (lane_id() & 7)) & 7) << 4);
            const float *f = reinterpret_cast<const float *>(&o_raw[cc][8 * e]);
            st_shared_v4(a, pack_bf16x2(f[0] * inv_l, f[1] * inv_l),
                         pack_bf16x2(f[2] * inv_l, f[3] * inv_l),
                         pack_bf16x2(f[4] * inv_l, f[5] * inv_l),
                         pack_bf16x2(f[6] * inv_l, f[7] * inv_l));
          }
        }
        fence_proxy_async_shared();
        __syncwarp();
        if (lane_id() == 0) {
          tma_store_3d(&tm_o, wbox, 0, w.hq, (int32_t)tok0 + wq * 32, pol_o);
          bulk_commit_group();
        }
        __syncwarp();
      }
      uint4 *dst = reinterpret_cast<uint4 *>(p.o + (tok * p.Hq + w.hq) * (int64_t)D);
#pragma unroll
      for (int c = 0; c < (tile_store ? 0 : D / 32); ++c) {
        uint32_t o_raw[32];
        tmem_ld_32x32b_x32(t_o + c * 32, o_raw);
        tmem_ld_wait();
        reg_fence(o_raw);
        uint32_t v[16];
#pragma unroll
        for (int e = 0; e < 16; ++e)
          v[e] = pack_bf16x2(__uint_as_float(o_raw[2 * e]) * inv_l,
                             __uint_as_float(o_raw[2 * e + 1]) * inv_l);
        if (row_store) {
          // Each thread writes its own row: 32-byte stores fill whole sectors
          // (half as many store instructions and sector writes as 16-byte ones).
          if (p.o_align32) {
            st_global_v8_hint(dst + c * 4, v[0], v[1], v[2], v[3], v[4], v[5], v[6], v[7], pol_o);
            st_global_v8_hint(dst + c * 4 + 2, v[8], v[9], v[10], v[11], v[12], v[13], v[14], v[15],
                              pol_o);
          } else {
#pragma unroll
            for (int e = 0; e < 4; ++e)
              st_global_v4_hint(dst + c * 4 + e, v[4 * e], v[4 * e + 1], v[4 * e + 2], v[4 * e + 3],
                                pol_o);
          }
        }
      }
      // O_X has been read: the next unit's first P_X V (which overwrites O_X)
      // is issued only after this warpgroup produces that unit's P_X(0).
      tc_fence_before_sync();
      if (row_store) {
        const float lse = (m_run + log2f(l_run)) * 0.69314718055994530942f;
        const int64_t li = VL ? (int64_t)w.hq * p.S + tok
                                    : ((int64_t)w.b * p.Hq + w.hq) * p.S + qpos;
        p.lse[li] = lse;
      }
    }
    if (!ok) *abort = 1;
    // Every TMA store of o this warp issued completes before the CTA releases
    // its shared memory.
    if (C::kStageO && lane_id() == 0) bulk_wait_group_all();
  }

  tc_fence_before_sync();
  __syncthreads();
  if (warp == kMmaWarp) {
    tc_fence_after_sync();
    tmem_dealloc(tmem, kTmemCols);
  }
  if (threadIdx.x == 0 && ctl->abort) {
    atomicExch(&g_status, (int)MK_ERR_TIMEOUT);
  }
  // MK_SCHED_DYNAMIC: every claim of this CTA was made before the barrier
  // above; the launch's last CTA to finish puts the slot back to zero.
  if (p.schedule == MK_SCHED_DYNAMIC && threadIdx.x == 0) sched_release(p.sched_slot);
}

// =================================================================== host

struct DeviceInfo {
  std::once_flag once;
  int sm_count = 0;
  cudaError_t attr_err[4] = {cudaSuccess, cudaSuccess, cudaSuccess, cudaSuccess};
  int regs[4] = {0, 0, 0, 0};  // [D == 128][varlen]
};

static DeviceInfo g_devices[64];

// Sets the shared-memory limit and reads the register count of one kernel
// instantiation (first call on a device only).
template <int D, bool VL>
static void kernel_setup(DeviceInfo &di) {
  const int vi = (D == 128 ? 2 : 0) + (VL ? 1 : 0);
  di.attr_err[vi] = cudaFuncSetAttribute(mk_attn_fwd_persistent<D, VL>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         KernelCfg<D>::kSmemBytes);
  cudaFuncAttributes fa;
  if (cudaFuncGetAttributes(&fa, mk_attn_fwd_persistent<D, VL>) == cudaSuccess) di.regs[vi] = fa.numRegs;
}

template <int D, bool VL>
static int launch(const void *q, const void *k, const void *v, const Params &p, int64_t tokens,
                  cudaStream_t stream) {
  using C = KernelCfg<D>;
  CUtensorMap tq, tk, tv, to;
  if (!encode_tokens_heads_dim(&tq, q, tokens, p.Hq, D, kTile) ||
      !encode_tokens_heads_dim(&to, p.o, tokens, p.Hq, D, 32) ||
      !encode_tokens_heads_dim(&tk, k, tokens, p.Hkv, D, kTile) ||
      !encode_tokens_heads_dim(&tv, v, tokens, p.Hkv, D, kTile))
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
  const int vi = (D == 128 ? 2 : 0) + (VL ? 1 : 0);
  if (di.sm_count <= 0 || di.attr_err[vi] != cudaSuccess) return MK_ERR_CUDA;
  // The warpgroup register split assumes the block launches with exactly
  // kLaunchRegs registers per thread; anything else could leave a
  // setmaxnreg.inc waiting forever, so refuse to launch.
  if (di.regs[vi] != kLaunchRegs) return MK_ERR_CUDA;
  const mk_attn_tuning tune = current_tuning();
  const int ctas = tune.ctas > 0 ? tune.ctas : di.sm_count;
  const int grid = p.n_units < ctas ? p.n_units : ctas;
  mark_launched(kFamFwd);
  mk_attn_fwd_persistent<D, VL><<<grid, kThreads, C::kSmemBytes, stream>>>(tq, tk, tv, to, p);
  return cudaGetLastError() == cudaSuccess ? MK_OK : MK_ERR_CUDA;
}

}  // namespace mk

namespace mk {
int fwd_take_status() {
  if (!launched(kFamFwd)) return 0;
  int h = 0;
  if (cudaMemcpyFromSymbol(&h, g_status, sizeof(int)) != cudaSuccess) return MK_ERR_CUDA;
  if (h != 0) {
    const int zero = 0;
    if (cudaMemcpyToSymbol(g_status, &zero, sizeof(int)) != cudaSuccess) return MK_ERR_CUDA;
  }
  return h;
}

static int attn_fwd_impl(const void *q, const void *k, const void *v, void *o, float *lse, int B,
                         int Hq, int Hkv, int S, int D, int causal, float scale,
                         const int32_t *cu_seqlens, void *stream, int stall_first_slot) {
  if (!q || !k || !v || !o || !lse) return MK_ERR_INVALID_ARG;
  if (B < 1 || Hq < 1 || Hkv < 1 || S < 1) return MK_ERR_INVALID_ARG;
  if (Hq % Hkv != 0) return MK_ERR_INVALID_ARG;
  if (!std::isfinite(scale)) return MK_ERR_INVALID_ARG;
  if (D != 64 && D != 128) return MK_ERR_UNSUPPORTED;
  auto misaligned = [](const void *ptr) { return (reinterpret_cast<uintptr_t>(ptr) & 15u) != 0; };
  if (misaligned(q) || misaligned(k) || misaligned(v) || misaligned(o) || misaligned(lse))
    return MK_ERR_ALIGNMENT;
  if (cu_seqlens && (reinterpret_cast<uintptr_t>(cu_seqlens) & 3u) != 0) return MK_ERR_ALIGNMENT;

  const bool varlen = cu_seqlens != nullptr;
  const int64_t tokens = varlen ? (int64_t)S : (int64_t)B * S;
  if (tokens > INT32_MAX) return MK_ERR_INVALID_ARG;
  // Work units (pairs of 128-row query tiles): fixed length B * Hq *
  // ceil(ceil(S/128)/2); varlen at most Hq * (T + 255 B) / 256, since a
  // sequence of L tokens has ceil(ceil(L/128)/2) <= L/256 + 1 pairs.
  const int64_t n_pairs = (((int64_t)S + kTile - 1) / kTile + 1) / 2;
  const int64_t n_units = varlen ? (int64_t)Hq * (((int64_t)S + 255LL * B) / 256)
                                 : n_pairs * B * Hq;
  if (n_units > INT32_MAX || n_units < 1) return MK_ERR_INVALID_ARG;

  Params p;
  p.o = reinterpret_cast<uint16_t *>(o);
  p.lse = lse;
  p.cu_seqlens = cu_seqlens;
  p.B = B;
  p.Hq = Hq;
  p.Hkv = Hkv;
  p.S = S;
  p.group = Hq / Hkv;
  p.causal = causal != 0;
  p.varlen = varlen;
  p.n_pairs = (int)n_pairs;
  p.n_units = (int)n_units;
  p.scale_log2 = scale * 1.4426950408889634f;
  p.o_align32 = (reinterpret_cast<uintptr_t>(o) & 31u) == 0;
  p.stall_first_slot = stall_first_slot;
  const mk_attn_tuning tune = current_tuning();
  p.schedule = tune.schedule;
  p.rescale_log2 = tune.rescale_log2;
  static std::atomic<uint32_t> sched_epoch{0};
  p.sched_slot = (int)(sched_epoch.fetch_add(1, std::memory_order_relaxed) % kSchedSlots);
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (D == 128)
    return varlen ? launch<128, true>(q, k, v, p, tokens, st) : launch<128, false>(q, k, v, p, tokens, st);
  return varlen ? launch<64, true>(q, k, v, p, tokens, st) : launch<64, false>(q, k, v, p, tokens, st);
}
}  // namespace mk

extern "C" {

int mk_attn_fwd(const void *q, const void *k, const void *v, void *o, float *lse, int B,
                int Hq, int Hkv, int S, int D, int causal, float scale,
                const int32_t *cu_seqlens, void *stream) {
  return mk::finish_call(
      mk::attn_fwd_impl(q, k, v, o, lse, B, Hq, Hkv, S, D, causal, scale, cu_seqlens, stream, 0),
      stream);
}

int mk_attn_fwd_stall_test(const void *q, const void *k, const void *v, void *o, float *lse,
                           int B, int Hq, int Hkv, int S, int D, int causal, float scale,
                           const int32_t *cu_seqlens, void *stream) {
  return mk::finish_call(
      mk::attn_fwd_impl(q, k, v, o, lse, B, Hq, Hkv, S, D, causal, scale, cu_seqlens, stream, 1),
      stream);
}


}  // extern "C"
