// fmha_fwd.cu -- attention forward pass for GB300 (sm_103a) and its C ABI.
//
// Computes, per sequence b, query head h (key/value head h / (Hq/Hkv)) and
// query row i:  o[i] = softmax(scale * q[i] K^T + causal mask) V  and the
// natural-log row log-sum-exp -- the operation of the paper's Flash Attention
// and GQA Attention kernels (Table 2), under the contract of Section 2.1 and
// Section 3.1 (same inputs and outputs as the reference operation).
//
// Design (one CTA = one 128-row query tile of one (sequence, query head)):
//   warp 5 (one thread)  TMA producer: the Q tile once, then K_j and V_j blocks of
//                        128 keys through an n-stage shared-memory ring
//                        (128-byte swizzle, mbarrier transaction counts).
//   warp 4 (one thread)  tcgen05 MMA issuer: S_j = Q K_j^T into one of two TMEM
//                        S buffers (fp32), and O += P_j V_j with P_j read from
//                        TMEM (bf16, written over S_j) and V_j as an MN-major
//                        shared-memory operand.
//   warps 0-3            softmax: thread r owns query row r, i.e. TMEM lane r.
//                        Online softmax in base 2 (t = s * scale * log2 e),
//                        lazy O rescaling (only when the row max rises by more
//                        than kRescaleThreshold), P rounded to bf16 (RNE) into
//                        TMEM; then the epilogue O / l -> bf16 and
//                        lse = ln 2 * (m + log2 l).
// Causal tiles visit key blocks 0..qt only (block skipping) and mask only the
// diagonal block; the ragged tail of a sequence is masked by key position.
// TMEM: S0 = columns 0..127, S1 = 128..255, O = 256..256+D.
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

namespace mk {

constexpr int kTile = 128;            // query rows per tile, keys per block
constexpr int kSoftmaxThreads = 128;  // warps 0..3, one thread per query row
constexpr int kMmaWarp = 4;
constexpr int kLoadWarp = 5;
constexpr int kThreads = 192;
constexpr int kBoxCols = 64;          // bf16 elements per 128-byte swizzle row
constexpr int kBoxBytes = kTile * kBoxCols * 2;  // one TMA box: 128 rows x 128 B
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColS = 0;         // S buffer sb at kColS + 128 * sb
constexpr uint32_t kColO = 256;
constexpr float kRescaleThreshold = 8.0f;  // log2 units: rescale O when m rises by > 2^8

__device__ int g_status = 0;              // MK_ERR_TIMEOUT once a wait ran out
__device__ unsigned int g_abort_epoch = 0; // launch epoch that timed out

template <int D>
struct KernelCfg {
  static_assert(D == 64 || D == 128, "head dimension 64 or 128");
  static constexpr int kStages = (D == 128) ? 2 : 4;
  static constexpr int kHalves = D / kBoxCols;        // swizzle boxes per tile
  static constexpr int kTileBytes = kTile * D * 2;    // one Q, K or V tile
  static constexpr int kOffQ = 0;
  static constexpr int kOffK = kOffQ + kTileBytes;
  static constexpr int kOffV = kOffK + kStages * kTileBytes;
  static constexpr int kOffBar = kOffV + kStages * kTileBytes;
  static constexpr int kSmemBytes = kOffBar + 256 + 1024;  // + barriers + alignment slack
};

struct SharedCtl {
  uint64_t bar_q;
  uint64_t bar_k_full[4], bar_k_empty[4];
  uint64_t bar_v_full[4], bar_v_empty[4];
  uint64_t bar_s_full[2], bar_p_full[2];
  uint64_t bar_o_done;       // one phase per P_j V_j
  uint64_t bar_o_final;      // the last P_j V_j of the tile
  uint64_t bar_mma_drained;
  uint32_t tmem_base;
  int abort;
  int tile_valid, tile_b, tile_qt, tile_seq_start, tile_len;
};
static_assert(sizeof(SharedCtl) <= 256, "control block");

struct Params {
  uint16_t *o;             // bf16 bits
  float *lse;
  const int32_t *cu_seqlens;
  int B, Hq, Hkv, S;       // S = tokens per sequence, or total tokens T (varlen)
  int group;               // Hq / Hkv
  int causal, varlen;
  int n_qtiles;            // fixed: ceil(S/128) ; varlen: bound on tiles per head
  float scale_log2;        // scale * log2(e)
  unsigned int epoch;
};

__device__ __forceinline__ int clamp_tok(int x, int T) { return x < 0 ? 0 : (x > T ? T : x); }

// Maps this CTA to (sequence, query tile, head).  Fixed length: causal tiles
// are ordered longest first (largest qt first) so that the hardware's in-order
// CTA dispatch approximates longest-processing-time scheduling.  Varlen: warp 0
// scans cu_seqlens (clamped to [0, T], negative lengths read as 0) and finds the
// sequence holding tile `rank` of this head.
__device__ __forceinline__ void map_tile(const Params &p, SharedCtl *ctl, int &hq) {
  const int idx = blockIdx.x;
  if (!p.varlen) {
    const int per_level = p.B * p.Hq;
    const int level = idx / per_level;
    const int rem = idx - level * per_level;
    hq = rem % p.Hq;
    if (threadIdx.x == 0) {
      const int b = rem / p.Hq;
      ctl->tile_valid = 1;
      ctl->tile_b = b;
      ctl->tile_qt = p.causal ? (p.n_qtiles - 1 - level) : level;
      ctl->tile_seq_start = b * p.S;
      ctl->tile_len = p.S;
    }
    return;
  }
  hq = idx % p.Hq;
  if (threadIdx.x < 32) {
    const int rank = idx / p.Hq;
    const int lane = threadIdx.x;
    const int T = p.S;
    int carry = 0;
    int found = 0, f_b = 0, f_qt = 0, f_s0 = 0, f_len = 0;
    for (int base = 0; base < p.B && !found; base += 32) {
      const int b = base + lane;
      int s0 = 0, s1 = 0, nt = 0;
      if (b < p.B) {
        s0 = clamp_tok(p.cu_seqlens[b], T);
        s1 = clamp_tok(p.cu_seqlens[b + 1], T);
        if (s1 < s0) s1 = s0;
        nt = (s1 - s0 + kTile - 1) / kTile;
      }
      int incl = nt;
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, off);
        if (lane >= off) incl += y;
      }
      const int excl = incl - nt;
      const bool mine = (b < p.B) && rank >= carry + excl && rank < carry + incl;
      const unsigned m = __ballot_sync(0xffffffffu, mine);
      if (m) {
        const int src = __ffs(m) - 1;
        f_b = base + src;
        f_qt = rank - carry - __shfl_sync(0xffffffffu, excl, src);
        f_s0 = __shfl_sync(0xffffffffu, s0, src);
        f_len = __shfl_sync(0xffffffffu, s1 - s0, src);
        found = 1;
      }
      carry += __shfl_sync(0xffffffffu, incl, 31);
    }
    if (lane == 0) {
      ctl->tile_valid = found;
      ctl->tile_b = f_b;
      ctl->tile_qt = f_qt;
      ctl->tile_seq_start = f_s0;
      ctl->tile_len = f_len;
    }
  }
}

// Bounded wait that ignores the abort flag: used only at teardown to let
// operations already in flight land before the CTA releases its resources.
__device__ __forceinline__ void drain_wait(uint64_t *bar, uint32_t parity) {
  int local_abort = 0;
  mbar_wait(bar, parity, &local_abort);
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    fmha_fwd_kernel(const __grid_constant__ CUtensorMap tm_q,
                    const __grid_constant__ CUtensorMap tm_k,
                    const __grid_constant__ CUtensorMap tm_v, const Params p) {
  using C = KernelCfg<D>;
  constexpr int NS = C::kStages;

  if (*reinterpret_cast<volatile unsigned int *>(&g_abort_epoch) == p.epoch) return;

  extern __shared__ uint8_t smem_raw[];
  // 1024-byte alignment for the 128-byte-swizzle atoms.
  const uint32_t raw_addr = smem_addr(smem_raw);
  uint8_t *smem = smem_raw + ((1024u - (raw_addr & 1023u)) & 1023u);
  SharedCtl *ctl = reinterpret_cast<SharedCtl *>(smem + C::kOffBar);
  const uint32_t sQ = smem_addr(smem + C::kOffQ);
  const uint32_t sK = smem_addr(smem + C::kOffK);
  const uint32_t sV = smem_addr(smem + C::kOffV);

  const int warp = threadIdx.x / 32;
  int hq = 0;
  map_tile(p, ctl, hq);

  if (threadIdx.x == 0) {
    mbar_init(&ctl->bar_q, 1);
    for (int s = 0; s < NS; ++s) {
      mbar_init(&ctl->bar_k_full[s], 1);
      mbar_init(&ctl->bar_k_empty[s], 1);
      mbar_init(&ctl->bar_v_full[s], 1);
      mbar_init(&ctl->bar_v_empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&ctl->bar_s_full[b], 1);
      mbar_init(&ctl->bar_p_full[b], kSoftmaxThreads);
    }
    mbar_init(&ctl->bar_o_done, 1);
    mbar_init(&ctl->bar_o_final, 1);
    mbar_init(&ctl->bar_mma_drained, 1);
    ctl->abort = 0;
    fence_mbar_init();
  }
  __syncthreads();
  if (!ctl->tile_valid) return;  // uniform: varlen CTAs beyond the last tile

  if (warp == kMmaWarp) {
    tmem_alloc(&ctl->tmem_base, kTmemCols);
    tmem_relinquish_alloc_permit();
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem = ctl->tmem_base;

  const int qt = ctl->tile_qt;
  const int seq_start = ctl->tile_seq_start;
  const int L = ctl->tile_len;
  const int hkv = hq / p.group;
  const int n_kblocks_seq = (L + kTile - 1) / kTile;
  const int nblk = p.causal ? min(qt + 1, n_kblocks_seq) : n_kblocks_seq;
  volatile int *abort = &ctl->abort;

  if (warp == kLoadWarp) {
    // ------------------------------------------------------------ producer
    if (lane_id() == 0) {
      tma_prefetch_desc(&tm_q);
      tma_prefetch_desc(&tm_k);
      tma_prefetch_desc(&tm_v);
      const uint64_t pol_q = l2_policy_evict_first();
      const uint64_t pol_kv = l2_policy_evict_last();
      mbar_arrive_expect_tx(&ctl->bar_q, C::kTileBytes);
      for (int h = 0; h < C::kHalves; ++h)
        tma_load_3d(smem + C::kOffQ + h * kBoxBytes, &tm_q, &ctl->bar_q, h * kBoxCols, hq,
                    seq_start + qt * kTile, pol_q);
      int issued = 0;
      for (int j = 0; j < nblk; ++j) {
        const int s = j % NS;
        const uint32_t ph = (j / NS) & 1;
        if (!mbar_wait(&ctl->bar_k_empty[s], ph ^ 1, abort)) break;
        mbar_arrive_expect_tx(&ctl->bar_k_full[s], C::kTileBytes);
        for (int h = 0; h < C::kHalves; ++h)
          tma_load_3d(smem + C::kOffK + s * C::kTileBytes + h * kBoxBytes, &tm_k,
                      &ctl->bar_k_full[s], h * kBoxCols, hkv, seq_start + j * kTile, pol_kv);
        if (!mbar_wait(&ctl->bar_v_empty[s], ph ^ 1, abort)) {
          issued = j * 2 + 1;
          break;
        }
        mbar_arrive_expect_tx(&ctl->bar_v_full[s], C::kTileBytes);
        for (int h = 0; h < C::kHalves; ++h)
          tma_load_3d(smem + C::kOffV + s * C::kTileBytes + h * kBoxBytes, &tm_v,
                      &ctl->bar_v_full[s], h * kBoxCols, hkv, seq_start + j * kTile, pol_kv);
        issued = j * 2 + 2;
      }
      // Teardown: every load issued must land before the CTA exits.
      drain_wait(&ctl->bar_q, 0);
      for (int n = (issued > 2 * NS ? issued - 2 * NS : 0); n < issued; ++n) {
        const int j = n / 2, s = j % NS;
        const uint32_t ph = (j / NS) & 1;
        drain_wait((n & 1) ? &ctl->bar_v_full[s] : &ctl->bar_k_full[s], ph);
      }
    }
  } else if (warp == kMmaWarp) {
    // ------------------------------------------------------------ MMA issuer
    if (lane_id() == 0) {
      constexpr uint32_t idesc_qk = idesc_bf16_f32(kTile, kTile, false, false);
      constexpr uint32_t idesc_pv = idesc_bf16_f32(kTile, D, false, true);
      bool ok = mbar_wait(&ctl->bar_q, 0, abort);
      auto issue_pv = [&](int i) -> bool {
        const int sb = i & 1, s = i % NS;
        const uint32_t ph = (i / NS) & 1;
        if (!mbar_wait(&ctl->bar_p_full[sb], (i >> 1) & 1, abort)) return false;
        if (!mbar_wait(&ctl->bar_v_full[s], ph, abort)) return false;
        tc_fence_after_sync();
        const uint32_t v_base = sV + s * C::kTileBytes;
#pragma unroll
        for (int kk = 0; kk < kTile / 16; ++kk) {
          // V as the B operand of P V: N = head dim (contiguous, MN-major),
          // K = keys.  8-key groups are 1024 B apart (SBO); 64-column chunks
          // of the head dimension are one TMA box (16 KB) apart (LBO).  With
          // D = 64 there is one chunk and the LBO field is not used.
          constexpr uint32_t kVLbo = (D > kBoxCols) ? kBoxBytes : 1024;
          const uint64_t bdesc = sdesc_sw128(v_base + kk * 16 * 128, kVLbo, 1024);
          umma_ts(tmem + kColO, tmem + kColS + sb * 128 + kk * 8, bdesc, idesc_pv,
                  (i > 0 || kk > 0) ? 1u : 0u);
        }
        umma_commit(&ctl->bar_v_empty[s]);
        umma_commit(&ctl->bar_o_done);
        if (i == nblk - 1) umma_commit(&ctl->bar_o_final);
        return true;
      };
      for (int j = 0; ok && j < nblk; ++j) {
        const int s = j % NS, sb = j & 1;
        const uint32_t ph = (j / NS) & 1;
        if (!mbar_wait(&ctl->bar_k_full[s], ph, abort)) {
          ok = false;
          break;
        }
        tc_fence_after_sync();
        const uint32_t k_base = sK + s * C::kTileBytes;
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          // Q and K are K-major (head dim contiguous); 16 bf16 = 32 B per MMA
          // step inside a 128-byte swizzle row; 8-row groups 1024 B apart.
          const uint32_t off = (kk / 4) * kBoxBytes + (kk % 4) * 32;
          const uint64_t adesc = sdesc_sw128(sQ + off, 16, 1024);
          const uint64_t bdesc = sdesc_sw128(k_base + off, 16, 1024);
          umma_ss(tmem + kColS + sb * 128, adesc, bdesc, idesc_qk, kk > 0 ? 1u : 0u);
        }
        umma_commit(&ctl->bar_s_full[sb]);
        umma_commit(&ctl->bar_k_empty[s]);
        if (j > 0 && !issue_pv(j - 1)) ok = false;
      }
      if (ok) issue_pv(nblk - 1);
      // Teardown: all MMAs issued by this thread complete before TMEM is freed.
      umma_commit(&ctl->bar_mma_drained);
      drain_wait(&ctl->bar_mma_drained, 0);
    }
  } else {
    // ------------------------------------------------------------ softmax
    const int r = threadIdx.x;  // query row within the tile == TMEM lane
    const uint32_t t_row = tmem + ((uint32_t)(warp * 32) << 16);
    const int qpos = qt * kTile + r;
    const bool row_valid = qpos < L;
    const int key_limit = p.causal ? min(L, qpos + 1) : L;  // keys [0, key_limit) visible
    const float c2 = p.scale_log2;
    float m_run = -INFINITY;  // running row max, base-2 units
    float l_run = 0.f;        // running row sum relative to m_run
    bool ok = true;

    for (int j = 0; j < nblk; ++j) {
      const int sb = j & 1;
      ok = mbar_wait(&ctl->bar_s_full[sb], (j >> 1) & 1, abort);
      if (!__all_sync(0xffffffffu, ok)) {
        ok = false;
        *abort = 1;
        break;
      }
      tc_fence_after_sync();
      float t[kTile];
      {
        uint32_t raw[4][32];
#pragma unroll
        for (int c = 0; c < 4; ++c) tmem_ld_32x32b_x32(t_row + kColS + sb * 128 + c * 32, raw[c]);
        tmem_ld_wait();
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          reg_fence(raw[c]);
#pragma unroll
          for (int e = 0; e < 32; ++e) t[c * 32 + e] = __uint_as_float(raw[c][e]) * c2;
        }
      }
      const bool needs_mask = (j * kTile + kTile > L) || (p.causal && j == qt);
      if (needs_mask) {
        const int lim = key_limit - j * kTile;
#pragma unroll
        for (int c = 0; c < kTile; ++c) t[c] = (c < lim) ? t[c] : -INFINITY;
      }
      float mx0 = t[0], mx1 = t[1], mx2 = t[2], mx3 = t[3];
#pragma unroll
      for (int c = 4; c < kTile; c += 4) {
        mx0 = fmaxf(mx0, t[c]);
        mx1 = fmaxf(mx1, t[c + 1]);
        mx2 = fmaxf(mx2, t[c + 2]);
        mx3 = fmaxf(mx3, t[c + 3]);
      }
      const float m_blk = fmaxf(fmaxf(mx0, mx1), fmaxf(mx2, mx3));
      const float m_new = fmaxf(m_run, m_blk);
      // Lazy rescaling: keep the old reference max unless the new one exceeds
      // it by more than the threshold.  Exact either way, because O and l
      // always share the same reference max.
      const bool rescale = m_new > m_run + kRescaleThreshold;
      float alpha = 1.f;
      if (rescale) {
        alpha = ex2_approx(m_run - m_new);  // 0 when m_run = -inf
        l_run *= alpha;
        m_run = m_new;
      }
      if (j > 0 && __any_sync(0xffffffffu, rescale)) {
        // O holds blocks 0..j-1 only once P_{j-1} V_{j-1} has completed.
        ok = mbar_wait(&ctl->bar_o_done, (j - 1) & 1, abort);
        if (!__all_sync(0xffffffffu, ok)) {
          ok = false;
          *abort = 1;
          break;
        }
        tc_fence_after_sync();
#pragma unroll
        for (int c = 0; c < D / 32; ++c) {
          uint32_t o_raw[32];
          tmem_ld_32x32b_x32(t_row + kColO + c * 32, o_raw);
          tmem_ld_wait();
          reg_fence(o_raw);
#pragma unroll
          for (int e = 0; e < 32; ++e)
            o_raw[e] = __float_as_uint(__uint_as_float(o_raw[e]) * alpha);
          tmem_st_32x32b_x32(t_row + kColO + c * 32, o_raw);
        }
        tmem_st_wait();
      }
      const float m_use = (m_run == -INFINITY) ? 0.f : m_run;
      float sum0 = 0.f, sum1 = 0.f, sum2 = 0.f, sum3 = 0.f;
      uint32_t pk[2][32];
#pragma unroll
      for (int c = 0; c < kTile; c += 4) {
        const float p0 = ex2_approx(t[c] - m_use);
        const float p1 = ex2_approx(t[c + 1] - m_use);
        const float p2 = ex2_approx(t[c + 2] - m_use);
        const float p3 = ex2_approx(t[c + 3] - m_use);
        sum0 += p0;
        sum1 += p1;
        sum2 += p2;
        sum3 += p3;
        pk[c / 64][(c % 64) / 2] = pack_bf16x2(p0, p1);
        pk[c / 64][(c % 64) / 2 + 1] = pack_bf16x2(p2, p3);
      }
      l_run += (sum0 + sum1) + (sum2 + sum3);
      // P_j (bf16, 64 columns) overwrites the first half of S_j.
      tmem_st_32x32b_x32(t_row + kColS + sb * 128, pk[0]);
      tmem_st_32x32b_x32(t_row + kColS + sb * 128 + 32, pk[1]);
      tmem_st_wait();
      tc_fence_before_sync();
      mbar_arrive(&ctl->bar_p_full[sb]);
    }

    // ------------------------------------------------------------ epilogue
    if (ok) {
      // A barrier of its own: bar_o_done may still be two phases short here.
      ok = mbar_wait(&ctl->bar_o_final, 0, abort);
      ok = __all_sync(0xffffffffu, ok);
    }
    if (ok) {
      tc_fence_after_sync();
      const float inv_l = 1.f / l_run;
      const int64_t tok = (int64_t)seq_start + qpos;
      uint4 *dst = reinterpret_cast<uint4 *>(p.o + (tok * p.Hq + hq) * (int64_t)D);
#pragma unroll
      for (int c = 0; c < D / 32; ++c) {
        uint32_t o_raw[32];
        tmem_ld_32x32b_x32(t_row + kColO + c * 32, o_raw);
        tmem_ld_wait();
        reg_fence(o_raw);
        uint32_t w[16];
#pragma unroll
        for (int e = 0; e < 16; ++e)
          w[e] = pack_bf16x2(__uint_as_float(o_raw[2 * e]) * inv_l,
                             __uint_as_float(o_raw[2 * e + 1]) * inv_l);
        if (row_valid) {
#pragma unroll
          for (int e = 0; e < 4; ++e)
            dst[c * 4 + e] = make_uint4(w[4 * e], w[4 * e + 1], w[4 * e + 2], w[4 * e + 3]);
        }
      }
      if (row_valid) {
        const float lse = (m_run + log2f(l_run)) * 0.69314718055994530942f;
        const int64_t li = p.varlen ? (int64_t)hq * p.S + tok
                                    : ((int64_t)ctl->tile_b * p.Hq + hq) * p.S + qpos;
        p.lse[li] = lse;
      }
    } else {
      *abort = 1;
    }
  }

  tc_fence_before_sync();
  __syncthreads();
  if (warp == kMmaWarp) {
    tc_fence_after_sync();
    tmem_dealloc(tmem, kTmemCols);
  }
  if (threadIdx.x == 0 && ctl->abort) {
    atomicExch(&g_status, (int)MK_ERR_TIMEOUT);
    atomicExch(&g_abort_epoch, p.epoch);
  }
}

// =================================================================== host

static PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void *ptr = nullptr;
    cudaDriverEntryPointQueryResult q = cudaDriverEntryPointSymbolNotFound;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000,
                                         cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  });
  return fn;
}

// [tokens, heads, D] bf16, boxes of 128 tokens x 1 head x 64 elements, 128-byte swizzle.
static bool encode_tokens_heads_dim(CUtensorMap *map, const void *base, uint64_t tokens,
                                    uint64_t heads, uint64_t D) {
  auto enc = tensor_map_encoder();
  if (!enc) return false;
  const cuuint64_t dims[3] = {D, heads, tokens};
  const cuuint64_t strides[2] = {D * 2, heads * D * 2};
  const cuuint32_t box[3] = {(cuuint32_t)kBoxCols, 1, (cuuint32_t)kTile};
  const cuuint32_t estr[3] = {1, 1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(base), dims, strides,
             box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

static std::atomic<unsigned int> g_epoch_counter{0};

static unsigned int next_epoch() {
  unsigned int e;
  do {
    e = g_epoch_counter.fetch_add(1) + 1;
  } while (e == 0);
  return e;
}

template <int D>
static int launch(const void *q, const void *k, const void *v, const Params &p, int64_t tokens,
                  int64_t grid, cudaStream_t stream) {
  using C = KernelCfg<D>;
  CUtensorMap tq, tk, tv;
  if (!encode_tokens_heads_dim(&tq, q, tokens, p.Hq, D) ||
      !encode_tokens_heads_dim(&tk, k, tokens, p.Hkv, D) ||
      !encode_tokens_heads_dim(&tv, v, tokens, p.Hkv, D))
    return MK_ERR_CUDA;
  static std::once_flag attr_once[64];
  static cudaError_t attr_err[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return MK_ERR_CUDA;
  std::call_once(attr_once[dev], [&] {
    attr_err[dev] = cudaFuncSetAttribute(fmha_fwd_kernel<D>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         C::kSmemBytes);
  });
  if (attr_err[dev] != cudaSuccess) return MK_ERR_CUDA;
  fmha_fwd_kernel<D><<<(unsigned)grid, kThreads, C::kSmemBytes, stream>>>(tq, tk, tv, p);
  return cudaGetLastError() == cudaSuccess ? MK_OK : MK_ERR_CUDA;
}

}  // namespace mk

extern "C" {

int mk_attn_fwd(const void *q, const void *k, const void *v, void *o, float *lse, int B,
                int Hq, int Hkv, int S, int D, int causal, float scale,
                const int32_t *cu_seqlens, void *stream) {
  using namespace mk;
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
  // Work tiles: fixed length B * Hq * ceil(S/128); varlen at most
  // Hq * (T + 127 B) / 128 (each sequence wastes under one tile).
  const int64_t n_qtiles = varlen ? ((int64_t)S + 127LL * B) / kTile : ((int64_t)S + kTile - 1) / kTile;
  const int64_t grid = varlen ? n_qtiles * Hq : n_qtiles * B * Hq;
  if (grid > INT32_MAX || (int64_t)Hq * tokens > INT32_MAX * 64LL) return MK_ERR_INVALID_ARG;

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
  p.n_qtiles = (int)n_qtiles;
  p.scale_log2 = scale * 1.4426950408889634f;
  p.epoch = next_epoch();
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  return D == 128 ? launch<128>(q, k, v, p, tokens, grid, st)
                  : launch<64>(q, k, v, p, tokens, grid, st);
}

const char *mk_attn_error_string(int status) {
  switch (status) {
    case MK_OK: return "success";
    case MK_ERR_INVALID_ARG: return "invalid argument";
    case MK_ERR_UNSUPPORTED: return "unsupported head dimension (64 or 128)";
    case MK_ERR_ALIGNMENT: return "pointer not 16-byte aligned";
    case MK_ERR_CUDA: return "CUDA call failed";
    case MK_ERR_TIMEOUT: return "kernel wait timed out";
    default: return "unknown status";
  }
}

int mk_attn_check_status(void *stream) {
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (cudaStreamSynchronize(st) != cudaSuccess) return MK_ERR_CUDA;
  int h = 0;
  if (cudaMemcpyFromSymbol(&h, mk::g_status, sizeof(int)) != cudaSuccess) return MK_ERR_CUDA;
  if (h != 0) {
    const int zero = 0;
    if (cudaMemcpyToSymbol(mk::g_status, &zero, sizeof(int)) != cudaSuccess) return MK_ERR_CUDA;
    return h;
  }
  return MK_OK;
}

int mk_attn_version(void) { return 100; }

}  // extern "C"
