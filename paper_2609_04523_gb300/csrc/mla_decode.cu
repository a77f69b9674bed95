// mla_decode.cu -- one decode step of multi-head latent attention (the
// absorbed form) against a paged latent cache, for GB300 (sm_103a), and its C
// ABI.
//
// Every query head attends to one shared latent cache: the cached row c_j
// (576 = 512 latent + 64 rotary components) is the key in full and, through
// its first 512 components, the value -- the paper's MLA Attention row
// (Table 2, Table 3), under the contract of Sections 2.1 and 3.1:
//   o[b,h,:512] = sum_j softmax_j(scale * q[b,h,:] . c_j) c_j[:512]
//   lse[b,h]    = ln sum_j exp(scale * q[b,h,:] . c_j)
// with position j in slot j % page_size of page page_table[b, j / page_size].
//
// All heads share every key, so a block of 64 keys is a pair of dense
// contractions on tcgen05 with the query heads as the MMA's M dimension (up to
// 128 heads, missing heads zero):
//   S  = Q C^T        M = heads, N = 64 keys, K = 576 (nine 64-wide chunks)
//   O += P C[:, :dv]  M = heads, N = 64 value components per MMA, K = 64 keys
// O for 128 heads x 512 components fills TMEM's 512 columns, so two CTAs
// share the work, as a cluster of two: CTA h keeps the value half
// 256 h .. 256 h + 255 of O, loads only the cache chunks it needs for that half
// (chunks 4 h .. 4 h + 3, and CTA 0 also the rotary chunk 8), and computes the
// part of S over those chunks.  The two CTAs exchange their partial scores
// (128 x 64 fp32 per block) through distributed shared memory -- each thread
// sends its row with asynchronous stores that complete on an mbarrier of the
// partner -- and both add them (the sum is the same in both CTAs), so each
// cached byte crosses from L2 into one SM only, and each CTA's value chunks
// are the key chunks it already holds.  S over the four TMEM
// chunks reads Q from TMEM (the TS form, at the tensor rate for N = 64); CTA
// 0's rotary chunk reads Q from shared memory.
//
// TMEM (512 columns): partial S, then P (bf16, first 32 columns), double
// buffered at 0 and 64; the CTA's four Q chunks at 128 (32 columns each);
// O (256 columns) at 256.  Shared memory: CTA 0's Q chunk 8 (16 KB), a ring
// of three block slots (up to five 8 KB chunks each), two 32 KB exchange
// slots written by the partner CTA.
//
// Softmax: base 2, one thread per head row, lazy rescale (O in TMEM is
// rescaled only when the row max rises by more than 8).  KV splits with a
// log-sum-exp merge fill the GPU at small batch, as in the paged decode step.
//
// Roles: warps 0-3 softmax, exchange and epilogue (thread = head row = TMEM
// lane), warp 4 tcgen05 MMA issuer, warp 5 TMA producer.  One CTA per SM.
// Every wait is bounded; a CTA that gives up records a timeout, and its
// partner's waits for it run out in turn, so both reach the final cluster
// barrier.  A CTA's last asynchronous store to its partner is either waited
// for by the partner or followed by a wait of its own that runs out (2 s)
// before it reaches that barrier, so no store lands after the partner left.
#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include <cmath>
#include <cstdint>
#include <mutex>

#include "mk_attn.h"
#include "ptx.cuh"
#include "tma_host.h"

namespace mk {
namespace mla {

constexpr int kDqk = MK_MLA_DQK;          // 576
constexpr int kDv = MK_MLA_DV;            // 512
constexpr int kChunk = 64;                // components per chunk (one 128-byte swizzle row)
constexpr int kDvCta = kDv / 2;           // 256 value components per CTA
constexpr int kChunksV = kDvCta / kChunk; // 4
constexpr int kHeads = 128;               // M: heads per CTA
constexpr int kBlock = 64;                // keys per block (N of S)
constexpr int kChunkBytes = kBlock * kChunk * 2;   // 8 KB: 64 rows x 128 B
constexpr int kQChunkBytes = kHeads * kChunk * 2;  // 16 KB
constexpr int kMaxChunksCta = 5;          // CTA 0: chunks 0-3 and 8; CTA 1: chunks 4-7
constexpr int kSlotBytes = kMaxChunksCta * kChunkBytes;
constexpr int kSlots = 3;
constexpr int kExchBytes = kHeads * kBlock * 4;    // 32 KB: one block's partial scores
constexpr int kOffQ8 = 0;
constexpr int kOffRing = kQChunkBytes;
constexpr int kOffExch = kOffRing + kSlots * kSlotBytes;
constexpr int kOffCtl = kOffExch + 2 * kExchBytes;
constexpr int kSmemBytes = kOffCtl + 256 + 1024;
static_assert(kSmemBytes <= 232448, "shared memory per CTA");
constexpr int kThreads = 192;
constexpr int kMmaWarp = 4, kLoadWarp = 5;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColS = 0;      // S buffer x at kColS + 64 x
constexpr uint32_t kColQ = 128;    // TMEM Q chunk j at kColQ + 32 j (bf16 pairs)
constexpr uint32_t kColO = 256;    // O: 256 columns
constexpr float kRescaleThreshold = 8.0f;

__device__ int g_status = 0;

struct Ctl {
  uint64_t q_full, qt_full;
  uint64_t slot_full[kSlots], slot_empty[kSlots];
  uint64_t s_full[2], p_full[2], pv_done[2];
  uint64_t exch_full[2];   // the partner's partial scores of block n are here (32 KB tx)
  uint64_t exch_empty[2];  // the partner has read this CTA's partial scores
  uint64_t mma_drained;
  uint32_t tmem_base;
  int abort;
};
static_assert(sizeof(Ctl) <= 256, "control block");

struct Params {
  const uint16_t *q;          // bf16 [B, Hq, 576]
  const int32_t *page_table;  // [B, max_pages]
  const int32_t *seq_lens;    // [B]
  uint16_t *o;                // bf16 [B, Hq, 512]
  float *lse;                 // [B, Hq]
  float *part;                // [B, Hq, n_splits, 516]: 512 components, lse, 3 pad; n_splits > 1
  int B, Hq, head_groups;
  int page_size, max_pages, num_pages;
  int n_splits, blocks_per_split;
  float scale_log2;
};

__device__ __forceinline__ void record(int status) { atomicCAS(&g_status, 0, status); }

__device__ __forceinline__ void drain_wait(uint64_t *bar, uint32_t parity) {
  int local_abort = 0;
  mbar_wait(bar, parity, &local_abort);
}

// 2-D tiled TMA load (cache viewed as [tokens, 576]).
__device__ __forceinline__ void tma_load_2d(void *dst, const CUtensorMap *map, uint64_t *bar,
                                            int32_t c0, int32_t c1, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%3, %4}], [%2], %5;" ::"r"(smem_addr(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_addr(bar)), "r"(c0), "r"(c1), "l"(policy)
      : "memory");
}

// ---------------------------------------------------------- cluster helpers

// The shared::cluster address of the partner CTA's copy of a local shared
// memory address.
__device__ __forceinline__ uint32_t peer_addr(uint32_t local, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(local), "r"(rank));
  return r;
}

// All threads of both CTAs of the cluster (release / acquire).
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::
                   : "memory");
}

// Asynchronous store of 16 bytes into the partner CTA's shared memory,
// counted (complete_tx) on the partner's mbarrier `remote_bar`.
__device__ __forceinline__ void st_async_peer_v4(uint32_t addr, uint32_t a, uint32_t b, uint32_t c,
                                                 uint32_t d, uint32_t remote_bar) {
  asm volatile(
      "st.async.shared::cluster.mbarrier::complete_tx::bytes.v4.b32 [%0], {%1, %2, %3, %4}, [%5];" ::"r"(
          addr),
      "r"(a), "r"(b), "r"(c), "r"(d), "r"(remote_bar)
      : "memory");
}

__device__ __forceinline__ void ld_shared_v4(uint32_t addr, uint32_t &a, uint32_t &b, uint32_t &c,
                                             uint32_t &d) {
  asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];"
               : "=r"(a), "=r"(b), "=r"(c), "=r"(d)
               : "r"(addr)
               : "memory");
}

// Relaxed arrival on an mbarrier of the partner CTA.  It follows local reads
// whose values have already been consumed, so nothing remains to order; a
// release arrival here costs about 1,000 clk per block (it waits for this
// thread's outstanding remote stores).
__device__ __forceinline__ void mbar_arrive_peer_relaxed(uint32_t remote_bar) {
  asm volatile("mbarrier.arrive.relaxed.cluster.shared::cluster.b64 _, [%0];" ::"r"(remote_bar)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait_cluster(uint32_t bar, uint32_t parity) {
  uint32_t done;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(done)
      : "r"(bar), "r"(parity)
      : "memory");
  return done != 0;
}

// Bounded wait (as mbar_wait) with acquire at cluster scope: the phase was
// completed by arrivals of the partner CTA, whose writes it publishes.
__device__ __forceinline__ bool mbar_wait_cluster(uint64_t *bar, uint32_t parity,
                                                  volatile int *abort) {
  const uint32_t a = smem_addr(bar);
  if (mbar_try_wait_cluster(a, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  for (uint32_t it = 1;; ++it) {
    if (mbar_try_wait_cluster(a, parity)) return true;
    if ((it & 255u) == 0) {
      if (*abort) return false;
      if (global_timer_ns() - t0 > kWaitLimitNs) {
        *abort = 1;
        return false;
      }
    }
  }
}

__global__ void __launch_bounds__(kThreads, 1)
    mla_decode_kernel(const __grid_constant__ CUtensorMap tm_q,
                      const __grid_constant__ CUtensorMap tm_c, const Params p) {
  // blockIdx.x = 2 (b * head_groups + hg) + half: the two CTAs of a cluster
  // (cluster rank = half) share (b, hg, split).  blockIdx.y = split.
  const int split = blockIdx.y, half = blockIdx.x & 1;
  const uint32_t peer = (uint32_t)(half ^ 1);
  const int b = (blockIdx.x >> 1) / p.head_groups, hg = (blockIdx.x >> 1) % p.head_groups;
  const int PS = p.page_size;
  int L = p.seq_lens[b];
  if (L < 0 || L > p.max_pages * PS) {
    if (threadIdx.x == 0) record(MK_ERR_INVALID_ARG);
    L = L < 0 ? 0 : p.max_pages * PS;
  }
  const int nblk_seq = (L + kBlock - 1) / kBlock;
  const int first = split * p.blocks_per_split;
  const int nb = max(0, min(first + p.blocks_per_split, nblk_seq) - first);
  // Splits past the end of the sequence do nothing (the merge skips them);
  // split 0 always runs, so an empty sequence still gets o = 0, lse = -inf.
  // Both CTAs of a cluster take the same branch.
  if (split > 0 && nb == 0) return;
  // Chunks this CTA holds per block, in slot order: CTA 0 chunks 0-3 and the
  // rotary chunk 8, CTA 1 chunks 4-7.  Positions 0-3 are the CTA's value
  // chunks, whose Q chunks live in TMEM.
  const int n_chunks = half == 0 ? 5 : 4;
  auto chunk_of = [&](int j) { return half == 0 ? (j < 4 ? j : 8) : 4 + j; };

  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw_addr = smem_addr(smem_raw);
  uint8_t *smem = smem_raw + ((1024u - (raw_addr & 1023u)) & 1023u);
  Ctl *ctl = reinterpret_cast<Ctl *>(smem + kOffCtl);
  const int warp = threadIdx.x / 32;

  if (threadIdx.x == 0) {
    mbar_init(&ctl->q_full, 1);
    mbar_init(&ctl->qt_full, kHeads);
    for (int s = 0; s < kSlots; ++s) {
      mbar_init(&ctl->slot_full[s], 1);
      mbar_init(&ctl->slot_empty[s], 1);
    }
    for (int x = 0; x < 2; ++x) {
      mbar_init(&ctl->s_full[x], 1);
      mbar_init(&ctl->p_full[x], kHeads);
      mbar_init(&ctl->pv_done[x], 1);
      mbar_init(&ctl->exch_full[x], 1);
      mbar_init(&ctl->exch_empty[x], kHeads);
    }
    mbar_init(&ctl->mma_drained, 1);
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
  // The partner's barriers are initialised before any arrival on them.
  cluster_sync();
  const uint32_t tmem = ctl->tmem_base;
  volatile int *abort = &ctl->abort;

  if (warp == kLoadWarp) {
    // ------------------------------------------------------------ producer
    bool ok = true;
    if (nb > 0) {
      if (elect_one()) {
        tma_prefetch_desc(&tm_c);
        if (half == 0) {
          tma_prefetch_desc(&tm_q);
          mbar_arrive_expect_tx(&ctl->q_full, kQChunkBytes);
          tma_load_3d(smem + kOffQ8, &tm_q, &ctl->q_full, 8 * kChunk, hg * kHeads, b,
                      l2_policy_evict_last());
        }
      }
      __syncwarp();
    }
    // Each cached chunk is read by one CTA, once.
    const uint64_t pol_c = l2_policy_evict_first();
    // A block is 64 / PS pages (PS <= 64) or half a page (PS = 128): one TMA
    // load of min(PS, 64) rows per page piece and chunk.
    const int rows_per_load = PS < kBlock ? PS : kBlock;
    const int loads_per_block = kBlock / rows_per_load;  // 1..4
    const int n_pages_seq = (L + PS - 1) / PS;
    const int lane = lane_id();
    // Physical page of piece `lane` of block n (lanes < loads_per_block), one
    // global load per lane per block, loaded one block ahead.  Pages past the
    // sequence end take the block's first page instead (finite rows, masked
    // out), so every slot moves the same number of bytes.
    auto block_pages = [&](int n) {
      int page = 0;
      if (n < nb && lane < loads_per_block) {
        const int page0 = (int)((int64_t)(first + n) * kBlock / PS);
        const int lp = page0 + lane < n_pages_seq ? page0 + lane : page0;
        page = p.page_table[(int64_t)b * p.max_pages + lp];
        if (page < 0 || page >= p.num_pages) {
          record(MK_ERR_INVALID_ARG);
          page = 0;
        }
      }
      return page;
    };
    int pages_cur = block_pages(0);
    for (int n = 0; ok && n < nb; ++n) {
      const int pages_next = block_pages(n + 1);
      const int s = n % kSlots;
      ok = mbar_wait_all(&ctl->slot_empty[s], ((n / kSlots) & 1) ^ 1, abort);
      if (!ok) break;
      int pg[kBlock / 16];
#pragma unroll
      for (int i = 0; i < kBlock / 16; ++i) pg[i] = __shfl_sync(0xffffffffu, pages_cur, i);
      const int row0 = PS > kBlock ? (int)(((int64_t)(first + n) * kBlock) % PS) : 0;
      if (elect_one()) {
        mbar_arrive_expect_tx(&ctl->slot_full[s], n_chunks * kChunkBytes);
        uint8_t *dst = smem + kOffRing + s * kSlotBytes;
        for (int j = 0; j < n_chunks; ++j)
#pragma unroll
          for (int i = 0; i < kBlock / 16; ++i)
            if (i < loads_per_block)
              tma_load_2d(dst + j * kChunkBytes + i * rows_per_load * 128, &tm_c,
                          &ctl->slot_full[s], chunk_of(j) * kChunk, pg[i] * PS + row0, pol_c);
      }
      __syncwarp();
      pages_cur = pages_next;
    }
    // Teardown: the loads issued land before the CTA exits.
    if (nb > 0 && half == 0) drain_wait(&ctl->q_full, 0);
    for (int n = max(0, nb - kSlots); n < nb; ++n)
      drain_wait(&ctl->slot_full[n % kSlots], (n / kSlots) & 1);
  } else if (warp == kMmaWarp) {
    // ---------------------------------------------------------- MMA issuer
    constexpr uint32_t idesc_s = idesc_bf16_f32(kHeads, kBlock, false, false);
    constexpr uint32_t idesc_pv = idesc_bf16_f32(kHeads, kChunk, false, true);
    const uint32_t sQ8 = smem_addr(smem + kOffQ8);
    const uint32_t sRing = smem_addr(smem + kOffRing);
    bool ok = true;
    // Partial S(n) = sum over this CTA's chunks of Q_c C_c^T, into S buffer n % 2.
    auto issue_s = [&](int n) {
      const int s = n % kSlots, x = n & 1;
      ok = mbar_wait_all(&ctl->slot_full[s], (n / kSlots) & 1, abort);
      tc_fence_after_sync();
      if (!ok) return;
      if (elect_one()) {
        const uint32_t slot = sRing + s * kSlotBytes;
        const uint32_t d = tmem + kColS + x * kBlock;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          // A = Q chunk from TMEM: 16 components = 8 columns per MMA.
          const uint64_t b0 = sdesc_sw128(slot + j * kChunkBytes, 16, 1024);
#pragma unroll
          for (int kk = 0; kk < kChunk / 16; ++kk)
            umma_ts(d, tmem + kColQ + j * 32 + kk * 8, b0 + kk * 2, idesc_s,
                    (j > 0 || kk > 0) ? 1u : 0u);
        }
        if (half == 0) {
          const uint64_t a0 = sdesc_sw128(sQ8, 16, 1024);
          const uint64_t b0 = sdesc_sw128(slot + 4 * kChunkBytes, 16, 1024);
#pragma unroll
          for (int kk = 0; kk < kChunk / 16; ++kk) umma_ss(d, a0 + kk * 2, b0 + kk * 2, idesc_s, 1u);
        }
        umma_commit(&ctl->s_full[x]);
      }
      __syncwarp();
    };
    // O (+)= P(n) C_n[:, value chunks]: P is bf16 in the first 32 columns of
    // S buffer n % 2 (the TMEM A operand); each value chunk (positions 0-3 of
    // the slot) an MN-major B operand of 64 keys x 64 components.
    auto issue_pv = [&](int n) {
      const int s = n % kSlots, x = n & 1;
      if (elect_one()) {
        const uint32_t slot = sRing + s * kSlotBytes;
#pragma unroll
        for (int j = 0; j < kChunksV; ++j) {
          const uint64_t b0 = sdesc_sw128(slot + j * kChunkBytes, 1024, 1024);
#pragma unroll
          for (int kk = 0; kk < kBlock / 16; ++kk)
            umma_ts(tmem + kColO + j * kChunk, tmem + kColS + x * kBlock + kk * 8,
                    b0 + (uint64_t)(kk * 128), idesc_pv, (n > 0 || kk > 0) ? 1u : 0u);
        }
        umma_commit(&ctl->pv_done[x]);
        umma_commit(&ctl->slot_empty[s]);
      }
      __syncwarp();
    };
    if (nb > 0) {
      if (half == 0) ok = mbar_wait_all(&ctl->q_full, 0, abort);
      if (ok) ok = mbar_wait_all(&ctl->qt_full, 0, abort);
      tc_fence_after_sync();
      if (ok) issue_s(0);
      for (int n = 0; ok && n < nb; ++n) {
        // S(n+1) into the other buffer: its P(n-1) was read by PV(n-1),
        // issued before this.
        if (n + 1 < nb) issue_s(n + 1);
        if (!ok) break;
        ok = mbar_wait_all(&ctl->p_full[n & 1], (n >> 1) & 1, abort);
        if (!ok) break;
        tc_fence_after_sync();
        issue_pv(n);
      }
    }
    if (elect_one()) umma_commit(&ctl->mma_drained);
    __syncwarp();
    drain_wait(&ctl->mma_drained, 0);
  } else {
    // ------------------------------------------------------------ softmax
    const int row = threadIdx.x;  // head within the group = TMEM lane
    const uint32_t t_row = tmem + ((uint32_t)((warp & 3) * 32) << 16);
    const float c2 = p.scale_log2;
    float m_run = -INFINITY, l_run = 0.f;
    bool ok = true;
    if (nb > 0) {
      // This CTA's four TMEM Q chunks of this head row as bf16 pairs
      // (component k of chunk position j in the low (k even) or high half of
      // column kColQ + 32 j + k / 2).  Heads past Hq are zero.
      const int hq = hg * kHeads + row;
      const uint4 *qrow = reinterpret_cast<const uint4 *>(p.q + ((int64_t)b * p.Hq + hq) * kDqk +
                                                          chunk_of(0) * kChunk);
#pragma unroll 1
      for (int j = 0; j < 4; ++j) {
        uint32_t w[32];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const uint4 u = hq < p.Hq ? __ldg(qrow + j * 8 + e) : make_uint4(0u, 0u, 0u, 0u);
          w[4 * e] = u.x;
          w[4 * e + 1] = u.y;
          w[4 * e + 2] = u.z;
          w[4 * e + 3] = u.w;
        }
        tmem_st_32x32b_x32(t_row + kColQ + j * 32, w);
      }
      tmem_st_wait();
      tc_fence_before_sync();
      mbar_arrive(&ctl->qt_full);
    }
    // Exchange slots, laid out [warp][16-byte chunk i of the row][lane]: the
    // 32 lanes of a warp write (to the partner) and read (locally) 512
    // contiguous bytes per instruction.
    const uint32_t exch_own = smem_addr(smem + kOffExch) + warp * 8192 + lane_id() * 16;
    const uint32_t exch_peer = peer_addr(exch_own, peer);
    const uint32_t peer_full0 = peer_addr(smem_addr(&ctl->exch_full[0]), peer);
    const uint32_t peer_full1 = peer_addr(smem_addr(&ctl->exch_full[1]), peer);
    const uint32_t peer_empty0 = peer_addr(smem_addr(&ctl->exch_empty[0]), peer);
    const uint32_t peer_empty1 = peer_addr(smem_addr(&ctl->exch_empty[1]), peer);
    for (int n = 0; ok && n < nb; ++n) {
      const int x = n & 1;
      ok = mbar_wait_all(&ctl->s_full[x], (n >> 1) & 1, abort);
      if (!ok) break;
      tc_fence_after_sync();
      uint32_t raw[kBlock / 32][32];
#pragma unroll
      for (int c = 0; c < kBlock / 32; ++c)
        tmem_ld_32x32b_x32(t_row + kColS + x * kBlock + c * 32, raw[c]);
      tmem_ld_wait();
#pragma unroll
      for (int c = 0; c < kBlock / 32; ++c) reg_fence(raw[c]);
      // Send this CTA's partial scores to the partner's slot x once the
      // partner has read what was there (block n - 2).
      ok = mbar_wait_cluster(&ctl->exch_empty[x], ((n >> 1) & 1) ^ 1, abort);
      if (!ok) break;
      // This CTA's slot x for block n expects the partner's 32 KB.
      if (threadIdx.x == 0) mbar_arrive_expect_tx(&ctl->exch_full[x], kExchBytes);
#pragma unroll
      for (int i = 0; i < kBlock / 4; ++i) {
        const uint32_t *w = &raw[i / 8][(i % 8) * 4];
        st_async_peer_v4(exch_peer + x * kExchBytes + i * 512, w[0], w[1], w[2], w[3],
                         x ? peer_full1 : peer_full0);
      }
      // The partner's partial scores of block n, added to this CTA's.
      ok = mbar_wait_cluster(&ctl->exch_full[x], (n >> 1) & 1, abort);
      if (!ok) break;
      float s[kBlock];
#pragma unroll
      for (int i = 0; i < kBlock / 4; ++i) {
        uint32_t a0, a1, a2, a3;
        ld_shared_v4(exch_own + x * kExchBytes + i * 512, a0, a1, a2, a3);
        const uint32_t *w = &raw[i / 8][(i % 8) * 4];
        s[4 * i] = (__uint_as_float(w[0]) + __uint_as_float(a0)) * c2;
        s[4 * i + 1] = (__uint_as_float(w[1]) + __uint_as_float(a1)) * c2;
        s[4 * i + 2] = (__uint_as_float(w[2]) + __uint_as_float(a2)) * c2;
        s[4 * i + 3] = (__uint_as_float(w[3]) + __uint_as_float(a3)) * c2;
      }
      mbar_arrive_peer_relaxed(x ? peer_empty1 : peer_empty0);
      const int key0 = (first + n) * kBlock;
      if (key0 + kBlock > L) {
#pragma unroll
        for (int c = 0; c < kBlock; ++c) s[c] = key0 + c < L ? s[c] : -INFINITY;
      }
      float mx0 = fmaxf(s[0], s[1]), mx1 = fmaxf(s[2], s[3]);
      float mx2 = fmaxf(s[4], s[5]), mx3 = fmaxf(s[6], s[7]);
#pragma unroll
      for (int c = 8; c < kBlock; c += 8) {
        mx0 = fmax3(mx0, s[c], s[c + 1]);
        mx1 = fmax3(mx1, s[c + 2], s[c + 3]);
        mx2 = fmax3(mx2, s[c + 4], s[c + 5]);
        mx3 = fmax3(mx3, s[c + 6], s[c + 7]);
      }
      const float m_new = fmaxf(m_run, fmaxf(fmax3(mx0, mx1, mx2), mx3));
      if (m_new > m_run + kRescaleThreshold) {
        const float alpha = ex2_approx(m_run - m_new);  // 0 when m_run = -inf
        l_run *= alpha;
        m_run = m_new;
        if (n > 0) {
          // O holds blocks 0..n-1 once PV(n-1) is done (PV(n-2) is, since
          // S(n) was issued after it).
          ok = mbar_wait_all(&ctl->pv_done[(n - 1) & 1], ((n - 1) >> 1) & 1, abort);
          if (!ok) break;
          tc_fence_after_sync();
#pragma unroll 1
          for (int c = 0; c < kDvCta / 32; ++c) {
            uint32_t o_raw[32];
            tmem_ld_32x32b_x32(t_row + kColO + c * 32, o_raw);
            tmem_ld_wait();
            reg_fence(o_raw);
#pragma unroll
            for (int e = 0; e < 32; ++e) o_raw[e] = __float_as_uint(__uint_as_float(o_raw[e]) * alpha);
            tmem_st_32x32b_x32(t_row + kColO + c * 32, o_raw);
          }
          tmem_st_wait();
        }
      }
      const float neg_m = m_run == -INFINITY ? 0.f : -m_run;
      float sum0 = 0.f, sum1 = 0.f, sum2 = 0.f, sum3 = 0.f;
      uint32_t pk[kBlock / 2];
#pragma unroll
      for (int c = 0; c < kBlock; c += 4) {
        const float p0 = ex2_approx(s[c] + neg_m), p1 = ex2_approx(s[c + 1] + neg_m);
        const float p2 = ex2_approx(s[c + 2] + neg_m), p3 = ex2_approx(s[c + 3] + neg_m);
        fadd2_acc(sum0, sum1, p0, p1);
        fadd2_acc(sum2, sum3, p2, p3);
        pk[c / 2] = pack_bf16x2(p0, p1);
        pk[c / 2 + 1] = pack_bf16x2(p2, p3);
      }
      l_run += (sum0 + sum1) + (sum2 + sum3);
      tmem_st_32x32b_x32(t_row + kColS + x * kBlock, pk);
      tmem_st_wait();
      tc_fence_before_sync();
      mbar_arrive(&ctl->p_full[x]);
    }
    // ------------------------------------------------------------ epilogue
    if (ok && nb > 0) {
      // PV(nb-1) and PV(nb-2) done: each pv_done buffer has no later phase.
      ok = mbar_wait_all(&ctl->pv_done[(nb - 1) & 1], ((nb - 1) >> 1) & 1, abort);
      if (ok && nb > 1) ok = mbar_wait_all(&ctl->pv_done[(nb - 2) & 1], ((nb - 2) >> 1) & 1, abort);
      tc_fence_after_sync();
    }
    const int h = hg * kHeads + row;
    if (ok) {
      const int64_t bh = (int64_t)b * p.Hq + h;
      // Check build: the (sequence, head) row and the split lie inside the
      // outputs and the partials.
      const bool valid = h < p.Hq && dbg_in_range(bh, (int64_t)p.B * p.Hq, &g_status) &&
                         dbg_in_range(split, p.n_splits, &g_status);
      const float inv_l = l_run > 0.f ? 1.f / l_run : 0.f;
      const float lse = l_run > 0.f ? (m_run + log2f(l_run)) * 0.69314718055994530942f : -INFINITY;
#pragma unroll 1
      for (int c = 0; c < kDvCta / 32; ++c) {
        float v[32];
        if (nb > 0) {
          uint32_t o_raw[32];
          tmem_ld_32x32b_x32(t_row + kColO + c * 32, o_raw);
          tmem_ld_wait();
          reg_fence(o_raw);
#pragma unroll
          for (int e = 0; e < 32; ++e) v[e] = __uint_as_float(o_raw[e]) * inv_l;
        } else {
#pragma unroll
          for (int e = 0; e < 32; ++e) v[e] = 0.f;
        }
        if (!valid) continue;
        const int d0 = half * kDvCta + c * 32;
        if (p.n_splits == 1) {
          uint4 *dst = reinterpret_cast<uint4 *>(p.o + bh * kDv + d0);
#pragma unroll
          for (int e = 0; e < 4; ++e)
            dst[e] = make_uint4(pack_bf16x2(v[8 * e], v[8 * e + 1]), pack_bf16x2(v[8 * e + 2], v[8 * e + 3]),
                                pack_bf16x2(v[8 * e + 4], v[8 * e + 5]), pack_bf16x2(v[8 * e + 6], v[8 * e + 7]));
        } else {
          float4 *dst = reinterpret_cast<float4 *>(p.part + (bh * p.n_splits + split) * (kDv + 4) + d0);
#pragma unroll
          for (int e = 0; e < 8; ++e) dst[e] = make_float4(v[4 * e], v[4 * e + 1], v[4 * e + 2], v[4 * e + 3]);
        }
      }
      if (valid && half == 0) {
        if (p.n_splits == 1)
          p.lse[bh] = lse;
        else
          p.part[(bh * p.n_splits + split) * (kDv + 4) + kDv] = lse;
      }
    }
    if (!ok) *abort = 1;
  }

  tc_fence_before_sync();
  __syncthreads();
  // Neither CTA leaves while the other may still write into its shared
  // memory or arrive on its barriers.
  cluster_sync();
  if (warp == kMmaWarp) {
    tc_fence_after_sync();
    tmem_dealloc(tmem, kTmemCols);
  }
  if (threadIdx.x == 0 && ctl->abort) record(MK_ERR_TIMEOUT);
}

// Combines the splits of each (b, h) by their log-sum-exps (as the paged
// decode step's merge), one warp per (b, h): each split's partial is
// o_s = (sum over its keys of exp(s_j) c_j) / exp(lse_s), stored with lse_s
// at component 512 of a 516-float row.
__global__ void __launch_bounds__(128) mla_merge_kernel(const Params p) {
  // Launched as a programmatic dependent of the latent decode kernel: nothing
  // is read before that kernel's partials are complete and visible.
  griddep_wait();
  constexpr int NDL = kDv / 32;
  const int row = blockIdx.x * 4 + threadIdx.x / 32;  // b * Hq + h
  if (row >= p.B * p.Hq) return;
  const int lane = lane_id();
  const float *pr = p.part + (int64_t)row * p.n_splits * (kDv + 4);
  int L = p.seq_lens[row / p.Hq];
  L = L < 0 ? 0 : (L > p.max_pages * p.page_size ? p.max_pages * p.page_size : L);
  const int nblk = (L + kBlock - 1) / kBlock;
  const int n_valid = max(1, min(p.n_splits, (nblk + p.blocks_per_split - 1) / p.blocks_per_split));
  float mx = -INFINITY;
  for (int s = 0; s < n_valid; ++s) mx = fmaxf(mx, pr[s * (kDv + 4) + kDv]);
  float acc[NDL];
#pragma unroll
  for (int e = 0; e < NDL; ++e) acc[e] = 0.f;
  float wsum = 0.f;
  if (mx > -INFINITY) {
    for (int s = 0; s < n_valid; ++s) {
      const float w = exp2f((pr[s * (kDv + 4) + kDv] - mx) * 1.4426950408889634f);
      wsum += w;
      const float4 *src = reinterpret_cast<const float4 *>(pr + s * (kDv + 4) + lane * NDL);
#pragma unroll
      for (int e = 0; e < NDL / 4; ++e) {
        const float4 f = src[e];
        acc[4 * e] = fmaf(w, f.x, acc[4 * e]);
        acc[4 * e + 1] = fmaf(w, f.y, acc[4 * e + 1]);
        acc[4 * e + 2] = fmaf(w, f.z, acc[4 * e + 2]);
        acc[4 * e + 3] = fmaf(w, f.w, acc[4 * e + 3]);
      }
    }
  }
  const float inv = wsum > 0.f ? 1.f / wsum : 0.f;
  uint4 *orow = reinterpret_cast<uint4 *>(p.o + (int64_t)row * kDv + lane * NDL);
#pragma unroll
  for (int e = 0; e < NDL / 8; ++e)
    orow[e] = make_uint4(pack_bf16x2(acc[8 * e] * inv, acc[8 * e + 1] * inv),
                         pack_bf16x2(acc[8 * e + 2] * inv, acc[8 * e + 3] * inv),
                         pack_bf16x2(acc[8 * e + 4] * inv, acc[8 * e + 5] * inv),
                         pack_bf16x2(acc[8 * e + 6] * inv, acc[8 * e + 7] * inv));
  if (lane == 0) p.lse[row] = wsum > 0.f ? mx + logf(wsum) : -INFINITY;
}

// ------------------------------------------------------------------- host

struct DeviceInfo {
  std::once_flag once;
  int sm_count = 0;
  cudaError_t attr = cudaSuccess;
};
static DeviceInfo g_devices[64];

static int sm_count_and_setup() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  DeviceInfo &di = g_devices[dev];
  std::call_once(di.once, [&] {
    if (cudaDeviceGetAttribute(&di.sm_count, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      di.sm_count = 0;
    di.attr = cudaFuncSetAttribute(mla_decode_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                   kSmemBytes);
  });
  return di.attr == cudaSuccess ? di.sm_count : 0;
}

// KV splits of whole 64-key blocks: about mla_split_ctas_per_sm (process-wide
// tuning) CTAs per SM over B x head groups x 2 value halves.  One CTA fills
// an SM, so this is the number of waves: more, shorter splits even out
// unequal sequence lengths, at the cost of a Q load and a merge row each.
static void plan(int B, int head_groups, int max_blocks, int sms, int &n_splits, int &bps) {
  const int64_t units = (int64_t)B * head_groups * 2;
  int64_t want = ((int64_t)current_tuning().mla_split_ctas_per_sm * sms + units - 1) / units;
  want = want < 1 ? 1 : (want > max_blocks ? max_blocks : want);
  bps = (int)((max_blocks + want - 1) / want);
  n_splits = (max_blocks + bps - 1) / bps;
}

static bool encode(CUtensorMap *map, const void *base, int rank, const cuuint64_t *dims,
                   const cuuint64_t *strides, const cuuint32_t *box) {
  auto enc = tensor_map_encoder();
  if (!enc) return false;
  const cuuint32_t estr[3] = {1, 1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, rank, const_cast<void *>(base), dims, strides,
             box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace mla

int mla_take_status() {
  if (!launched(kFamMla)) return 0;
  int h = 0;
  if (cudaMemcpyFromSymbol(&h, mla::g_status, sizeof(int)) != cudaSuccess) return MK_ERR_CUDA;
  if (h != 0) {
    const int zero = 0;
    if (cudaMemcpyToSymbol(mla::g_status, &zero, sizeof(int)) != cudaSuccess) return MK_ERR_CUDA;
  }
  return h;
}

}  // namespace mk

extern "C" {

int64_t mk_attn_mla_decode_workspace_bytes(int B, int Hq, int page_size, int max_pages) {
  if (B < 1 || Hq < 1 || page_size < 1 || max_pages < 1) return -1;
  const int sms = mk::mla::sm_count_and_setup();
  if (sms <= 0) return -1;
  const int64_t max_keys = (int64_t)max_pages * page_size;
  const int max_blocks = (int)((max_keys + mk::mla::kBlock - 1) / mk::mla::kBlock);
  const int head_groups = (Hq + mk::mla::kHeads - 1) / mk::mla::kHeads;
  int n_splits = 1, bps = max_blocks;
  mk::mla::plan(B, head_groups, max_blocks, sms, n_splits, bps);
  if (n_splits == 1) return 0;
  return (int64_t)B * Hq * n_splits * (mk::mla::kDv + 4) * 4;
}

}  // extern "C"

namespace mk {
static int mla_decode_impl(const void *q, const void *cache, const int32_t *page_table,
                           const int32_t *seq_lens, void *o, float *lse, int B, int Hq,
                           int page_size, int max_pages, int num_pages, float scale,
                           void *workspace, int64_t workspace_bytes, void *stream) {
  if (!q || !cache || !page_table || !seq_lens || !o || !lse) return MK_ERR_INVALID_ARG;
  if (B < 1 || Hq < 1 || max_pages < 1 || num_pages < 1) return MK_ERR_INVALID_ARG;
  if (!std::isfinite(scale)) return MK_ERR_INVALID_ARG;
  if (page_size != 16 && page_size != 32 && page_size != 64 && page_size != 128)
    return MK_ERR_UNSUPPORTED;
  if ((int64_t)num_pages * page_size > INT32_MAX || (int64_t)max_pages * page_size > INT32_MAX)
    return MK_ERR_INVALID_ARG;
  const int head_groups = (Hq + mla::kHeads - 1) / mla::kHeads;
  if ((int64_t)B * head_groups > (1 << 29)) return MK_ERR_UNSUPPORTED;  // grid x
  auto misaligned = [](const void *ptr, uintptr_t a) {
    return (reinterpret_cast<uintptr_t>(ptr) & (a - 1)) != 0;
  };
  if (misaligned(q, 16) || misaligned(cache, 16) || misaligned(o, 16) || misaligned(lse, 4) ||
      misaligned(page_table, 4) || misaligned(seq_lens, 4))
    return MK_ERR_ALIGNMENT;
  const int sms = mla::sm_count_and_setup();
  if (sms <= 0) return MK_ERR_CUDA;
  const int64_t max_keys = (int64_t)max_pages * page_size;
  const int max_blocks = (int)((max_keys + mla::kBlock - 1) / mla::kBlock);
  mla::Params p;
  p.q = reinterpret_cast<const uint16_t *>(q);
  p.page_table = page_table;
  p.seq_lens = seq_lens;
  p.o = reinterpret_cast<uint16_t *>(o);
  p.lse = lse;
  p.B = B;
  p.Hq = Hq;
  p.head_groups = head_groups;
  p.page_size = page_size;
  p.max_pages = max_pages;
  p.num_pages = num_pages;
  p.scale_log2 = scale * 1.4426950408889634f;
  mla::plan(B, head_groups, max_blocks, sms, p.n_splits, p.blocks_per_split);
  p.part = nullptr;
  if (p.n_splits > 1) {
    const int64_t need = (int64_t)B * Hq * p.n_splits * (mla::kDv + 4) * 4;
    if (!workspace || workspace_bytes < need) return MK_ERR_INVALID_ARG;
    if (misaligned(workspace, 16)) return MK_ERR_ALIGNMENT;
    p.part = reinterpret_cast<float *>(workspace);
  }
  CUtensorMap tq, tc;
  const cuuint64_t qdims[3] = {(cuuint64_t)mla::kDqk, (cuuint64_t)Hq, (cuuint64_t)B};
  const cuuint64_t qstr[2] = {(cuuint64_t)mla::kDqk * 2, (cuuint64_t)Hq * mla::kDqk * 2};
  const cuuint32_t qbox[3] = {(cuuint32_t)mla::kChunk, (cuuint32_t)mla::kHeads, 1};
  const cuuint64_t cdims[2] = {(cuuint64_t)mla::kDqk, (cuuint64_t)num_pages * page_size};
  const cuuint64_t cstr[1] = {(cuuint64_t)mla::kDqk * 2};
  const cuuint32_t cbox[2] = {(cuuint32_t)mla::kChunk,
                             (cuuint32_t)(page_size < mla::kBlock ? page_size : mla::kBlock)};
  if (!mla::encode(&tq, q, 3, qdims, qstr, qbox) || !mla::encode(&tc, cache, 2, cdims, cstr, cbox))
    return MK_ERR_CUDA;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const dim3 grid(2 * B * head_groups, p.n_splits, 1);
  mark_launched(kFamMla);
  {
    // Clusters of two CTAs along x: the two value halves of one (b, hg, split).
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.gridDim = grid;
    cfg.blockDim = dim3(mla::kThreads);
    cfg.dynamicSmemBytes = mla::kSmemBytes;
    cfg.stream = st;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (cudaLaunchKernelEx(&cfg, mla::mla_decode_kernel, tq, tc, p) != cudaSuccess) return MK_ERR_CUDA;
  }
  if (p.n_splits > 1) {
    // Scheduled while the decode grid drains; it waits for the partials itself.
    DependentLaunch dl(dim3((B * Hq + 3) / 4), dim3(128), 0, st);
    if (cudaLaunchKernelEx(&dl.cfg, mla::mla_merge_kernel, p) != cudaSuccess) return MK_ERR_CUDA;
  }
  return MK_OK;
}
}  // namespace mk

extern "C" {

int mk_attn_mla_decode_paged(const void *q, const void *cache, const int32_t *page_table,
                             const int32_t *seq_lens, void *o, float *lse, int B, int Hq,
                             int page_size, int max_pages, int num_pages, float scale,
                             void *workspace, int64_t workspace_bytes, void *stream) {
  return mk::finish_call(mk::mla_decode_impl(q, cache, page_table, seq_lens, o, lse, B, Hq,
                                             page_size, max_pages, num_pages, scale, workspace,
                                             workspace_bytes, stream),
                         stream);
}

}  // extern "C"

