// decode.cu -- one decode step of attention against a paged K/V cache, for
// GB300 (sm_103a), and its C ABI.
//
// Computes, for each sequence b and query head h (key/value head
// g = h / (Hq/Hkv)), the attention of the newest query q[b,h,:] over the
// L_b = seq_lens[b] cached positions of that sequence, which live in pages of
// page_size positions: position j is slot j % page_size of physical page
// page_table[b, j / page_size] of k_cache / v_cache [num_pages, page_size,
// Hkv, D].  Output o[b,h,:] (bf16) and the natural-log row log-sum-exp
// lse[b,h] -- the Paged Attention row of the paper's Table 2, under the same
// contract as the forward pass (same inputs and outputs as the reference
// operation, Sections 2.1 and 3.1).
//
// The work is HBM-bound (each cached key and value is read once, for
// 4 * G * D flops per key with G = Hq / Hkv heads sharing it), so it runs on
// the CUDA cores, and the design is about keeping the HBM busy:
//   * split-KV: CTA (split, g, b) takes a contiguous run of the sequence's
//     pages, so that short batches still fill the GPU; its partial result
//     (o / l and lse over its keys) goes to a caller-provided fp32 workspace,
//     and a merge kernel combines the splits by their log-sum-exps.  With a
//     single split the decode kernel writes o and lse itself.
//   * a producer warp streams K and V pages with TMA into a shared-memory
//     ring of about 64 KB (2 to 8 pages); the page is the box (page_size
//     tokens x 1 head x 64 elements, 128-byte swizzle), so a page-table
//     gather costs nothing;
//   * four compute warps split each page's keys and each handles all the
//     query heads of the CTA (up to 8), so every key and value row is read
//     from shared memory and converted once.  Sixteen lanes share a key (D/16
//     dimensions each), two keys per instruction.  The per-head partial dot
//     products are summed over the 16 lanes by a transposed reduction (each
//     exchange step halves the values a lane holds), which leaves every lane
//     with the full score of one head: MH heads cost MH - 1 + log2(16 / MH)
//     shuffles instead of 4 MH, and one exp2 per lane covers them all.  The
//     probabilities are then broadcast by shuffles for o += p v, which runs
//     on packed fp32x2 FMAs.  Online base-2 softmax with a lazy rescale: a
//     head's reference max moves only when a score exceeds it by more than 8
//     (exact either way).  At the end the warps' states are merged through
//     shared memory (aliasing the drained page ring).
#include <cuda.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>
#include <mutex>

#include "mk_attn.h"
#include "ptx.cuh"
#include "tma_host.h"

namespace mk {
namespace dec {

constexpr int kWarps = 4;                    // compute warps
constexpr int kThreads = 32 * (kWarps + 1);  // + one producer warp
constexpr int kMaxStages = 8;
// Split planning (defaults of mk_attn_tuning): aim for about 24 CTAs per SM,
// and no split shorter than 2 pages.

__device__ int g_status = 0;  // MK_ERR_TIMEOUT or MK_ERR_INVALID_ARG from a decode launch

struct Params {
  const uint16_t *q;          // bf16 [B, Hq, D]
  const int32_t *page_table;  // [B, max_pages]
  const int32_t *seq_lens;    // [B]
  uint16_t *o;                // bf16 [B, Hq, D]
  float *lse;                 // [B, Hq]
  float *part;                // [B, Hq, n_splits, D + 1]; unused with one split
  int B, Hq, Hkv, G;
  int HG, head_groups;        // query heads per CTA (the last CTA of a group may have fewer),
                              // CTAs per key/value head: head_groups = ceil(G / HG)
  int page_size, max_pages, num_pages;
  int n_splits, pages_per_split;
  float scale_log2;           // scale * log2(e)
};

struct Ctl {
  uint64_t full[kMaxStages], empty[kMaxStages];
  int abort;
};

__device__ __forceinline__ void record(int status) { atomicCAS(&g_status, 0, status); }

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

template <int D>
struct Cfg {
  static_assert(D == 64 || D == 128, "head dimension 64 or 128");
  static constexpr int kDimsPerLane = D / 16;  // 16 lanes per key: 4 or 8
  static constexpr int kBoxes = D / 64;        // 128-byte swizzle rows per token
};

constexpr int kMaxHeads = 8;              // query heads per CTA
constexpr float kRescaleThreshold = 8.0f;  // log2 units

// This lane's D/16 elements of token r of a page tile (kBoxes boxes of
// page_size rows x 128 B, each 1024-B group of 8 rows stored with its 16-byte
// chunks permuted: chunk c of row r at position c ^ (r % 8)).  Lanes
// 16*grp + sl read row r of their half-warp; sl selects the dimensions.
template <int D>
__device__ __forceinline__ void load_row(const uint8_t *tile, int r, int page_size, int sl,
                                         float (&x)[Cfg<D>::kDimsPerLane]) {
  if constexpr (D == 128) {  // 8 elements = one 16-byte chunk: chunk sl % 8 of box sl / 8
    const uint8_t *a = tile + (sl >> 3) * page_size * 128 + r * 128 + (((sl & 7) ^ (r & 7)) << 4);
    const uint4 w = *reinterpret_cast<const uint4 *>(a);
    x[0] = bf16_lo(w.x); x[1] = bf16_hi(w.x); x[2] = bf16_lo(w.y); x[3] = bf16_hi(w.y);
    x[4] = bf16_lo(w.z); x[5] = bf16_hi(w.z); x[6] = bf16_lo(w.w); x[7] = bf16_hi(w.w);
  } else {  // 4 elements = half a chunk: chunk sl / 2, half sl % 2
    const uint8_t *a = tile + r * 128 + (((sl >> 1) ^ (r & 7)) << 4) + (sl & 1) * 8;
    const uint2 w = *reinterpret_cast<const uint2 *>(a);
    x[0] = bf16_lo(w.x); x[1] = bf16_hi(w.x); x[2] = bf16_lo(w.y); x[3] = bf16_hi(w.y);
  }
}

// Transposed sum over the 16 lanes of each half-warp of MH per-head values.
// Exchange step k (lane distance 8 >> k) halves the n = MH >> k values a
// lane holds while n > 1 -- the lane keeps the upper half if its bit is set,
// else the lower half, and adds the other lane's copy of the kept half --
// and is a plain butterfly step once n = 1.  The result on lane sl is the
// full sum for head head_of_lane<MH>(sl).
template <int MH>
__device__ __forceinline__ int head_of_lane(int sl) {
  int h = 0;
#pragma unroll
  for (int k = 0; k < 4; ++k)
    if ((MH >> k) > 1 && (sl & (8 >> k))) h += (MH >> k) / 2;
  return h;
}

// The lowest lane of a half-warp that ends up with head h's sum.
template <int MH>
__host__ __device__ constexpr int lane_of_head(int h) {
  int sl = 0;
  for (int k = 0; k < 4; ++k)
    if ((MH >> k) > 1 && h >= (MH >> k) / 2) {
      sl |= 8 >> k;
      h -= (MH >> k) / 2;
    }
  return sl;
}

template <int MH>
__device__ __forceinline__ float transpose_sum16(const float (&a)[MH], int sl) {
  float v[MH];
#pragma unroll
  for (int j = 0; j < MH; ++j) v[j] = a[j];
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    constexpr int kMH = MH;
    const int off = 8 >> k;
    const int n = kMH >> k;
    if (n > 1) {
      const bool up = (sl & off) != 0;
#pragma unroll
      for (int j = 0; j < n / 2; ++j) {
        const float keep = up ? v[j + n / 2] : v[j];
        const float send = up ? v[j] : v[j + n / 2];
        v[j] = keep + __shfl_xor_sync(0xffffffffu, send, off);
      }
    } else {
      v[0] += __shfl_xor_sync(0xffffffffu, v[0], off);
    }
  }
  return v[0];
}

// Score of key r of a page tile for head head_of_lane<MH>(sl) (the dot
// product with the pre-scaled query, summed over the half-warp).
template <int D, int MH>
__device__ __forceinline__ float score(const uint8_t *kt, int r, int page_size, int sl,
                                       const float2 (&q2)[MH][Cfg<D>::kDimsPerLane / 2]) {
  constexpr int NDL = Cfg<D>::kDimsPerLane;
  float kx[NDL];
  load_row<D>(kt, r, page_size, sl, kx);
  float part[MH];
#pragma unroll
  for (int h = 0; h < MH; ++h) {
    float2 t = __fmul2_rn(q2[h][0], make_float2(kx[0], kx[1]));
#pragma unroll
    for (int e = 1; e < NDL / 2; ++e) t = __ffma2_rn(q2[h][e], make_float2(kx[2 * e], kx[2 * e + 1]), t);
    part[h] = t.x + t.y;
  }
  return transpose_sum16<MH>(part, sl);
}

// Pages in flight per CTA: about 64 KB of K and V whatever the page size
// (2 to kMaxStages pages), so that small pages keep as many bytes in flight.
__host__ __device__ constexpr int ring_stages(int D, int page_size) {
  return 65536 / (4 * page_size * D) < 2
             ? 2
             : (65536 / (4 * page_size * D) > kMaxStages ? kMaxStages : 65536 / (4 * page_size * D));
}

// Bytes of the page ring, which the merge area reuses: the larger of the two.
__host__ __device__ constexpr int area_bytes(int D, int page_size, int MH) {
  return ring_stages(D, page_size) * 4 * page_size * D > kWarps * MH * (D + 2) * 4
             ? ring_stages(D, page_size) * 4 * page_size * D
             : (kWarps * MH * (D + 2) * 4 + 7) / 8 * 8;
}

// MH: query heads a CTA can hold in registers (1, 2, 4 or kMaxHeads); the
// CTA handles nh <= MH of them.
template <int D, int MH>
__global__ void __launch_bounds__(kThreads, MH > 4 ? 2 : 3)
    decode_kernel(const __grid_constant__ CUtensorMap tm_k, const __grid_constant__ CUtensorMap tm_v,
                  const Params p) {
  static_assert(MH >= 1 && MH <= kMaxHeads, "heads per CTA");
  using C = Cfg<D>;
  constexpr int NDL = C::kDimsPerLane;
  const int split = blockIdx.x, b = blockIdx.z;
  const int g = blockIdx.y / p.head_groups;  // key/value head
  const int hg0 = (blockIdx.y % p.head_groups) * p.HG;
  const int h0 = g * p.G + hg0;              // first query head of the CTA
  const int nh = min(p.HG, p.G - hg0);       // its query heads
  const int PS = p.page_size;
  const int tile_bytes = PS * D * 2;  // one page of K (or V) for one head
  const int NS = ring_stages(D, PS);

  // Pages [first, first + n_pg) of the sequence belong to this split.
  int L = p.seq_lens[b];
  if (L < 0 || L > p.max_pages * PS) {
    if (threadIdx.x == 0) record(MK_ERR_INVALID_ARG);
    L = L < 0 ? 0 : p.max_pages * PS;
  }
  const int n_pages_b = (L + PS - 1) / PS;
  const int first = split * p.pages_per_split;
  const int n_pg = max(0, min(first + p.pages_per_split, n_pages_b) - first);
  // Splits past the end of the sequence have nothing to do (the merge does
  // not read them); split 0 always runs, so an empty sequence still gets its
  // o = 0, lse = -inf.
  if (split > 0 && n_pg == 0) return;

  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw_addr = smem_addr(smem_raw);
  uint8_t *smem = smem_raw + ((1024u - (raw_addr & 1023u)) & 1023u);
  // [stages][K, V tiles], reused after the last page as the merge area
  // [warp][head][D + 2] floats | control
  float *mrg = reinterpret_cast<float *>(smem);
  Ctl *ctl = reinterpret_cast<Ctl *>(smem + area_bytes(D, PS, MH));
  const int warp = threadIdx.x / 32;

  if (threadIdx.x == 0) {
    for (int s = 0; s < NS; ++s) {
      mbar_init(&ctl->full[s], 1);
      mbar_init(&ctl->empty[s], kWarps);
    }
    ctl->abort = 0;
    fence_mbar_init();
  }
  __syncthreads();
  volatile int *abort = &ctl->abort;

  if (warp == kWarps) {
    // ------------------------------------------------------------ producer
    const uint64_t pol = l2_policy_evict_first();  // the cache is streamed once
    bool ok = true;
    int s = 0;
    uint32_t phase = 0;  // of page i: (i / NS) & 1
    for (int i = 0; ok && i < n_pg; ++i) {
      ok = mbar_wait_all(&ctl->empty[s], phase ^ 1, abort);
      if (!ok) break;
      if (elect_one()) {
        int page = p.page_table[(int64_t)b * p.max_pages + first + i];
        if (page < 0 || page >= p.num_pages) {
          record(MK_ERR_INVALID_ARG);
          page = 0;  // keep the pipeline going; the result is undefined
        }
        mbar_arrive_expect_tx(&ctl->full[s], 2 * tile_bytes);
        uint8_t *kt = smem + s * 2 * tile_bytes;
#pragma unroll
        for (int h = 0; h < C::kBoxes; ++h) {
          tma_load_3d(kt + h * PS * 128, &tm_k, &ctl->full[s], h * 64, g, page * PS, pol);
          tma_load_3d(kt + tile_bytes + h * PS * 128, &tm_v, &ctl->full[s], h * 64, g, page * PS,
                      pol);
        }
      }
      __syncwarp();
      if (++s == NS) s = 0, phase ^= 1;
    }
    // Teardown: the loads issued land before the CTA exits.
    for (int i = max(0, n_pg - NS); i < n_pg; ++i) {
      int local_abort = 0;
      mbar_wait(&ctl->full[i % NS], (i / NS) & 1, &local_abort);
    }
  } else {
    // ------------------------------------------------------------- compute
    // Half-warp grp (lanes 16*grp .. 16*grp+15) takes key 2*pr + grp of each
    // key pair pr = warp, warp + kWarps, ... of a page; lane sl = lane % 16
    // owns dimensions NDL*sl .. NDL*sl + NDL - 1 of every head, and after
    // each reduction the score of head hl of its half's key.  Query heads
    // nh .. MH-1 have q = 0 and are never written.
    const int lane = lane_id(), grp = lane >> 4, sl = lane & 15;
    const int hl = head_of_lane<MH>(sl);
    float2 q2[MH][NDL / 2], acc[MH][NDL / 2];
#pragma unroll
    for (int h = 0; h < MH; ++h) {
      const uint16_t *qr = p.q + ((int64_t)b * p.Hq + h0 + min(h, nh - 1)) * D + sl * NDL;
#pragma unroll
      for (int e = 0; e < NDL / 2; ++e) {
        const float f = h < nh ? p.scale_log2 : 0.f;
        q2[h][e] = make_float2(__uint_as_float((uint32_t)qr[2 * e] << 16) * f,
                               __uint_as_float((uint32_t)qr[2 * e + 1] << 16) * f);
        acc[h][e] = make_float2(0.f, 0.f);
      }
    }
    // Running max (log2 units) of head hl, the same on every lane that owns
    // hl, and its sum of exp2(s - ml) over this half-warp's keys.
    float ml = -INFINITY, ll = 0.f;
    bool ok = true;
    int s = 0;
    uint32_t phase = 0;
    for (int i = 0; ok && i < n_pg; ++i) {
      ok = mbar_wait_all(&ctl->full[s], phase, abort);
      if (!ok) break;
      const uint8_t *kt = smem + s * 2 * tile_bytes;
      const uint8_t *vt = kt + tile_bytes;
      const int key0 = (first + i) * PS;  // position of the page's first slot
      // Two independent key pairs per step (pr and pr + kWarps; page_size / 2
      // is a multiple of 2 * kWarps), one rescale vote for both.
      for (int pr = warp; 2 * pr < PS; pr += 2 * kWarps) {
        const int r0 = 2 * pr + grp, r1 = r0 + 2 * kWarps;
        const bool valid0 = key0 + r0 < L, valid1 = key0 + r1 < L;
        float sc0 = score<D, MH>(kt, r0, PS, sl, q2);
        float sc1 = score<D, MH>(kt, r1, PS, sl, q2);
        sc0 = valid0 ? sc0 : -INFINITY;
        sc1 = valid1 ? sc1 : -INFINITY;
        const float s01 = fmaxf(sc0, sc1);
        const float smax = fmaxf(s01, __shfl_xor_sync(0xffffffffu, s01, 16));  // all four keys
        const bool need = smax > ml + kRescaleThreshold;
        if (__any_sync(0xffffffffu, need)) {  // rare after the first keys
          const float m_new = need ? smax : ml;
          const float alpha = ml == -INFINITY ? 0.f : ex2_approx(ml - m_new);
          ll *= alpha;
          ml = m_new;
#pragma unroll
          for (int h = 0; h < MH; ++h) {
            const float a = __shfl_sync(0xffffffffu, alpha, lane_of_head<MH>(h));
#pragma unroll
            for (int e = 0; e < NDL / 2; ++e) acc[h][e] = __fmul2_rn(acc[h][e], make_float2(a, a));
          }
        }
        const float pl0 = valid0 ? ex2_approx(sc0 - ml) : 0.f;
        const float pl1 = valid1 ? ex2_approx(sc1 - ml) : 0.f;
        ll += pl0 + pl1;
        float vx0[NDL], vx1[NDL];
        load_row<D>(vt, r0, PS, sl, vx0);
        load_row<D>(vt, r1, PS, sl, vx1);
#pragma unroll
        for (int h = 0; h < MH; ++h) {
          const float ph0 = __shfl_sync(0xffffffffu, pl0, (lane & 16) | lane_of_head<MH>(h));
          const float ph1 = __shfl_sync(0xffffffffu, pl1, (lane & 16) | lane_of_head<MH>(h));
#pragma unroll
          for (int e = 0; e < NDL / 2; ++e) {
            acc[h][e] = __ffma2_rn(make_float2(ph0, ph0), make_float2(vx0[2 * e], vx0[2 * e + 1]),
                                   acc[h][e]);
            acc[h][e] = __ffma2_rn(make_float2(ph1, ph1), make_float2(vx1[2 * e], vx1[2 * e + 1]),
                                   acc[h][e]);
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&ctl->empty[s]);
      if (++s == NS) s = 0, phase ^= 1;
    }
    if (!ok) *abort = 1;
    // The two half-warps share ml: add their sums.  mrg[warp][h] =
    // (m, l, acc[0..D)) once every compute warp is past the page ring.
    ll += __shfl_xor_sync(0xffffffffu, ll, 16);
#pragma unroll
    for (int h = 0; h < MH; ++h)
#pragma unroll
      for (int e = 0; e < NDL / 2; ++e) {
        acc[h][e].x += __shfl_xor_sync(0xffffffffu, acc[h][e].x, 16);
        acc[h][e].y += __shfl_xor_sync(0xffffffffu, acc[h][e].y, 16);
      }
    named_barrier_sync(1, 32 * kWarps);
    if (grp == 0) {
#pragma unroll
      for (int h = 0; h < MH; ++h) {
        if (h < nh) {
          float *st = mrg + (warp * MH + h) * (D + 2) + 2 + sl * NDL;
#pragma unroll
          for (int e = 0; e < NDL / 2; ++e) st[2 * e] = acc[h][e].x, st[2 * e + 1] = acc[h][e].y;
        }
      }
      if (hl < nh && sl == lane_of_head<MH>(hl)) {
        float *st = mrg + (warp * MH + hl) * (D + 2);
        st[0] = ml;
        st[1] = ll;
      }
    }
    named_barrier_sync(1, 32 * kWarps);
    // Warp w finishes heads w, w + kWarps: merge the four warps' states by
    // their maxima, then o = acc / l and lse = ln 2 * (M + log2 l); no key at
    // all gives o = 0 and lse = -inf.
    for (int h = warp; h < nh; h += kWarps) {
      float M = -INFINITY;
#pragma unroll
      for (int w = 0; w < kWarps; ++w) M = fmaxf(M, mrg[(w * MH + h) * (D + 2)]);
      float lt = 0.f, o2[D / 32];
#pragma unroll
      for (int e = 0; e < D / 32; ++e) o2[e] = 0.f;
      if (M > -INFINITY) {
#pragma unroll
        for (int w = 0; w < kWarps; ++w) {
          const float *st = mrg + (w * MH + h) * (D + 2);
          const float f = st[0] == -INFINITY ? 0.f : ex2_approx(st[0] - M);
          lt = fmaf(f, st[1], lt);
#pragma unroll
          for (int e = 0; e < D / 32; ++e) o2[e] = fmaf(f, st[2 + lane * (D / 32) + e], o2[e]);
        }
      }
      const float inv_l = lt > 0.f ? 1.f / lt : 0.f;
      const float lse = lt > 0.f ? (M + log2f(lt)) * 0.69314718055994530942f : -INFINITY;
      const int hq = h0 + h;
      // Check build: the (sequence, head) row and the split lie inside the
      // outputs and the partials.
      if (!dbg_in_range((int64_t)b * p.Hq + hq, (int64_t)p.B * p.Hq, &g_status) ||
          !dbg_in_range(split, p.n_splits, &g_status))
        continue;
      if (p.n_splits == 1) {
        uint16_t *orow = p.o + ((int64_t)b * p.Hq + hq) * D + lane * (D / 32);
#pragma unroll
        for (int e = 0; e < D / 32; e += 2)
          *reinterpret_cast<uint32_t *>(orow + e) = pack_bf16x2(o2[e] * inv_l, o2[e + 1] * inv_l);
        if (lane == 0) p.lse[(int64_t)b * p.Hq + hq] = lse;
      } else {
        float *pr = p.part + (((int64_t)b * p.Hq + hq) * p.n_splits + split) * (D + 1);
#pragma unroll
        for (int e = 0; e < D / 32; ++e) pr[lane * (D / 32) + e] = o2[e] * inv_l;
        if (lane == 0) pr[D] = lse;
      }
    }
  }
  __syncthreads();
  if (threadIdx.x == 0 && ctl->abort) record(MK_ERR_TIMEOUT);
}

// Combines the splits of each (b, h): with lse_s the split log-sum-exps and
// o_s = (sum over the split's keys of exp(s_j) v_j) / exp(lse_s),
//   o = sum_s exp(lse_s) o_s / sum_s exp(lse_s),  lse = ln sum_s exp(lse_s),
// evaluated relative to the largest lse_s.  One warp per (b, h).
template <int D>
__global__ void __launch_bounds__(128) merge_kernel(const Params p) {
  // Launched as a programmatic dependent of the decode kernel: nothing is read
  // before that kernel's partials are complete and visible.
  griddep_wait();
  constexpr int NDL = D / 32;
  const int row = blockIdx.x * 4 + threadIdx.x / 32;  // b * Hq + h
  if (row >= p.B * p.Hq) return;
  const int lane = lane_id();
  const float *pr = p.part + (int64_t)row * p.n_splits * (D + 1);
  // The splits that hold pages of this sequence (the decode kernel skips the
  // others); split 0 always exists.
  int L = p.seq_lens[row / p.Hq];
  L = L < 0 ? 0 : (L > p.max_pages * p.page_size ? p.max_pages * p.page_size : L);
  const int n_pages = (L + p.page_size - 1) / p.page_size;
  const int n_valid = max(1, min(p.n_splits, (n_pages + p.pages_per_split - 1) / p.pages_per_split));
  // The split lse values, one per lane, then a warp max: the loads are issued
  // together rather than one after another.
  float mx = -INFINITY;
  for (int s0 = 0; s0 < n_valid; s0 += 32) {
    const int s = s0 + lane;
    mx = fmaxf(mx, s < n_valid ? pr[s * (D + 1) + D] : -INFINITY);
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
  float acc[NDL];
#pragma unroll
  for (int e = 0; e < NDL; ++e) acc[e] = 0.f;
  float wsum = 0.f;
  if (mx > -INFINITY) {
    // Groups of kGroup splits: every load of a group is issued before the
    // first use; the sums run in split order.
    constexpr int kGroup = 8;
    for (int s0 = 0; s0 < n_valid; s0 += kGroup) {
      float lv[kGroup], v[kGroup][NDL];
#pragma unroll
      for (int t = 0; t < kGroup; ++t) {
        const bool in = s0 + t < n_valid;
        const float *ps = pr + (int64_t)(s0 + t) * (D + 1);
        lv[t] = in ? ps[D] : -INFINITY;
#pragma unroll
        for (int e = 0; e < NDL; ++e) v[t][e] = in ? ps[lane * NDL + e] : 0.f;
      }
#pragma unroll
      for (int t = 0; t < kGroup; ++t) {
        if (s0 + t < n_valid) {
          const float w = exp2f((lv[t] - mx) * 1.4426950408889634f);
          wsum += w;
#pragma unroll
          for (int e = 0; e < NDL; ++e) acc[e] = fmaf(w, v[t][e], acc[e]);
        }
      }
    }
  }
  const float inv = wsum > 0.f ? 1.f / wsum : 0.f;
  uint16_t *orow = p.o + (int64_t)row * D + lane * NDL;
#pragma unroll
  for (int e = 0; e < NDL; e += 2)
    *reinterpret_cast<uint32_t *>(orow + e) = pack_bf16x2(acc[e] * inv, acc[e + 1] * inv);
  if (lane == 0) p.lse[row] = wsum > 0.f ? mx + logf(wsum) : -INFINITY;
}

// ------------------------------------------------------------------- host

struct DeviceInfo {
  std::once_flag once;
  int sm_count = 0;
};
static DeviceInfo g_devices[64];

static int sm_count() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  DeviceInfo &di = g_devices[dev];
  std::call_once(di.once, [&] {
    if (cudaDeviceGetAttribute(&di.sm_count, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      di.sm_count = 0;
  });
  return di.sm_count;
}

// Query heads per CTA: the G heads of a key/value head in ceil(G / kMaxHeads)
// nearly equal groups.
static void head_split(int G, int &HG, int &head_groups) {
  head_groups = (G + kMaxHeads - 1) / kMaxHeads;
  HG = (G + head_groups - 1) / head_groups;
}

// Splits per (b, g, head group): pages_per_split pages each, so that there
// are about split_ctas_per_sm CTAs per SM (several waves of them, so that
// sequences of different lengths even out), but no split shorter than
// split_min_pages pages and no more splits than the longest possible
// sequence has pages (both from the process-wide tuning).
static void plan_splits(int B, int Hkv, int head_groups, int max_pages, int sms, int &n_splits,
                        int &pps) {
  const mk_attn_tuning tune = current_tuning();
  const int64_t units = (int64_t)B * Hkv * head_groups;
  int64_t want = ((int64_t)tune.split_ctas_per_sm * sms + units - 1) / units;
  want = want < 1 ? 1 : (want > max_pages ? max_pages : want);
  pps = (int)((max_pages + want - 1) / want);
  const int min_pages = tune.split_min_pages;
  if (pps < min_pages) pps = min_pages < max_pages ? min_pages : max_pages;
  n_splits = (max_pages + pps - 1) / pps;
}

static size_t smem_bytes(int D, int page_size, int MH) {
  return (size_t)area_bytes(D, page_size, MH) + sizeof(Ctl) + 1024;
}

template <int D, int MH>
static int launch(const CUtensorMap &tk, const CUtensorMap &tv, const Params &p, cudaStream_t st) {
  const size_t sm = smem_bytes(D, p.page_size, MH);
  if (cudaFuncSetAttribute(decode_kernel<D, MH>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)sm) != cudaSuccess)
    return MK_ERR_CUDA;
  const dim3 grid(p.n_splits, p.Hkv * p.head_groups, p.B);
  mark_launched(kFamDecode);
  decode_kernel<D, MH><<<grid, kThreads, sm, st>>>(tk, tv, p);
  if (cudaGetLastError() != cudaSuccess) return MK_ERR_CUDA;
  if (p.n_splits > 1) {
    // Scheduled while the decode grid drains; it waits for the partials itself.
    DependentLaunch dl(dim3((p.B * p.Hq + 3) / 4), dim3(128), 0, st);
    if (cudaLaunchKernelEx(&dl.cfg, merge_kernel<D>, p) != cudaSuccess) return MK_ERR_CUDA;
  }
  return MK_OK;
}

// Scratch of mk_attn_decode_paged_noalloc: the split partials of every call
// on this device, for callers that cannot allocate device memory.  Host code
// sees only a stand-in for it; its device address is looked up once per
// device (with that device current) and then passed to the kernels like a
// caller's workspace.
constexpr int64_t kStaticScratchBytes = MK_ATTN_DECODE_STATIC_SCRATCH_BYTES;
static __device__ __align__(256) float g_static_scratch[kStaticScratchBytes / sizeof(float)];

struct StaticScratch {
  std::mutex mu;
  void *addr[64] = {};
};
static StaticScratch g_scratch;

// Device address of g_static_scratch on the current device, or nullptr if
// the lookup fails (then retried on the next call).
static void *static_scratch_address() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
  std::lock_guard<std::mutex> lock(g_scratch.mu);
  if (!g_scratch.addr[dev]) {
    void *ptr = nullptr;
    if (cudaGetSymbolAddress(&ptr, g_static_scratch) != cudaSuccess || !ptr) {
      cudaGetLastError();  // not sticky: leave no error behind for the caller
      return nullptr;
    }
    g_scratch.addr[dev] = ptr;
  }
  return g_scratch.addr[dev];
}

// The checks of mk_attn_decode_paged that need neither the device nor the
// workspace: pointers, sizes, head dimension, page size, grid limits and
// alignment.  No CUDA call; shared by both decode entry points so that they
// reject the same arguments with the same status.
static int check_host_args(const void *q, const void *k_cache, const void *v_cache,
                           const int32_t *page_table, const int32_t *seq_lens, const void *o,
                           const float *lse, int B, int Hq, int Hkv, int D, int page_size,
                           int max_pages, int num_pages, float scale) {
  if (!q || !k_cache || !v_cache || !page_table || !seq_lens || !o || !lse)
    return MK_ERR_INVALID_ARG;
  if (B < 1 || Hq < 1 || Hkv < 1 || Hq % Hkv != 0 || max_pages < 1 || num_pages < 1)
    return MK_ERR_INVALID_ARG;
  if (!std::isfinite(scale)) return MK_ERR_INVALID_ARG;
  if (D != 64 && D != 128) return MK_ERR_UNSUPPORTED;
  if (page_size != 16 && page_size != 32 && page_size != 64 && page_size != 128)
    return MK_ERR_UNSUPPORTED;
  int HG = 1, head_groups = 1;
  head_split(Hq / Hkv, HG, head_groups);
  if (B > 65535 || (int64_t)Hkv * head_groups > 65535) return MK_ERR_UNSUPPORTED;  // grid z / y
  if ((int64_t)num_pages * page_size > INT32_MAX || (int64_t)max_pages * page_size > INT32_MAX)
    return MK_ERR_INVALID_ARG;
  auto misaligned = [](const void *ptr, uintptr_t a) {
    return (reinterpret_cast<uintptr_t>(ptr) & (a - 1)) != 0;
  };
  if (misaligned(q, 16) || misaligned(k_cache, 16) || misaligned(v_cache, 16) ||
      misaligned(o, 16) || misaligned(lse, 4) || misaligned(page_table, 4) ||
      misaligned(seq_lens, 4))
    return MK_ERR_ALIGNMENT;
  return MK_OK;
}

}  // namespace dec

int decode_take_status() {
  if (!launched(kFamDecode)) return 0;
  int h = 0;
  if (cudaMemcpyFromSymbol(&h, dec::g_status, sizeof(int)) != cudaSuccess) return MK_ERR_CUDA;
  if (h != 0) {
    const int zero = 0;
    if (cudaMemcpyToSymbol(dec::g_status, &zero, sizeof(int)) != cudaSuccess) return MK_ERR_CUDA;
  }
  return h;
}

}  // namespace mk

extern "C" {

int64_t mk_attn_decode_workspace_bytes(int B, int Hq, int Hkv, int D, int page_size,
                                       int max_pages) {
  if (B < 1 || Hq < 1 || Hkv < 1 || Hq % Hkv || (D != 64 && D != 128) || page_size < 1 ||
      max_pages < 1)
    return -1;
  const int sms = mk::dec::sm_count();
  if (sms <= 0) return -1;
  int HG = 1, head_groups = 1, n_splits = 1, pps = max_pages;
  mk::dec::head_split(Hq / Hkv, HG, head_groups);
  mk::dec::plan_splits(B, Hkv, head_groups, max_pages, sms, n_splits, pps);
  if (n_splits == 1) return 0;
  return (int64_t)B * Hq * n_splits * (D + 1) * 4;
}

}  // extern "C"

namespace mk {
static int decode_paged_impl(const void *q, const void *k_cache, const void *v_cache,
                             const int32_t *page_table, const int32_t *seq_lens, void *o,
                             float *lse, int B, int Hq, int Hkv, int D, int page_size,
                             int max_pages, int num_pages, float scale, void *workspace,
                             int64_t workspace_bytes, void *stream) {
  const int chk = dec::check_host_args(q, k_cache, v_cache, page_table, seq_lens, o, lse, B, Hq,
                                       Hkv, D, page_size, max_pages, num_pages, scale);
  if (chk != MK_OK) return chk;
  auto misaligned = [](const void *ptr, uintptr_t a) { return (reinterpret_cast<uintptr_t>(ptr) & (a - 1)) != 0; };
  const int G = Hq / Hkv;
  int HG = 1, head_groups = 1;
  dec::head_split(G, HG, head_groups);
  const int sms = dec::sm_count();
  if (sms <= 0) return MK_ERR_CUDA;
  dec::Params p;
  p.q = reinterpret_cast<const uint16_t *>(q);
  p.page_table = page_table;
  p.seq_lens = seq_lens;
  p.o = reinterpret_cast<uint16_t *>(o);
  p.lse = lse;
  p.B = B;
  p.Hq = Hq;
  p.Hkv = Hkv;
  p.G = G;
  p.HG = HG;
  p.head_groups = head_groups;
  p.page_size = page_size;
  p.max_pages = max_pages;
  p.num_pages = num_pages;
  p.scale_log2 = scale * 1.4426950408889634f;
  dec::plan_splits(B, Hkv, head_groups, max_pages, sms, p.n_splits, p.pages_per_split);
  p.part = nullptr;
  if (p.n_splits > 1) {
    const int64_t need = (int64_t)B * Hq * p.n_splits * (D + 1) * 4;
    if (!workspace || workspace_bytes < need) return MK_ERR_INVALID_ARG;
    if (misaligned(workspace, 16)) return MK_ERR_ALIGNMENT;
    p.part = reinterpret_cast<float *>(workspace);
  }
  CUtensorMap tk, tv;
  const uint64_t tokens = (uint64_t)num_pages * page_size;
  if (!encode_tokens_heads_dim(&tk, k_cache, tokens, Hkv, D, page_size) ||
      !encode_tokens_heads_dim(&tv, v_cache, tokens, Hkv, D, page_size))
    return MK_ERR_CUDA;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (D == 128) {
    if (HG == 1) return dec::launch<128, 1>(tk, tv, p, st);
    if (HG == 2) return dec::launch<128, 2>(tk, tv, p, st);
    if (HG <= 4) return dec::launch<128, 4>(tk, tv, p, st);
    return dec::launch<128, dec::kMaxHeads>(tk, tv, p, st);
  }
  if (HG == 1) return dec::launch<64, 1>(tk, tv, p, st);
  if (HG == 2) return dec::launch<64, 2>(tk, tv, p, st);
  if (HG <= 4) return dec::launch<64, 4>(tk, tv, p, st);
  return dec::launch<64, dec::kMaxHeads>(tk, tv, p, st);
}
}  // namespace mk

extern "C" {

int mk_attn_decode_paged(const void *q, const void *k_cache, const void *v_cache,
                         const int32_t *page_table, const int32_t *seq_lens, void *o, float *lse,
                         int B, int Hq, int Hkv, int D, int page_size, int max_pages,
                         int num_pages, float scale, void *workspace, int64_t workspace_bytes,
                         void *stream) {
  return mk::finish_call(mk::decode_paged_impl(q, k_cache, v_cache, page_table, seq_lens, o, lse,
                                               B, Hq, Hkv, D, page_size, max_pages, num_pages,
                                               scale, workspace, workspace_bytes, stream),
                         stream);
}


int mk_attn_decode_paged_noalloc(const void *q, const void *k_cache, const void *v_cache,
                                 const int32_t *page_table, const int32_t *seq_lens, void *o,
                                 float *lse, int B, int Hq, int Hkv, int D, int page_size,
                                 int max_pages, int num_pages, float scale, void *stream) {
  // Host checks first (no CUDA call), then the scratch size, then the
  // once-per-device address lookup; so an invalid call returns the status
  // mk_attn_decode_paged gives it and touches nothing on the device.
  const int chk = mk::dec::check_host_args(q, k_cache, v_cache, page_table, seq_lens, o, lse, B,
                                           Hq, Hkv, D, page_size, max_pages, num_pages, scale);
  if (chk != MK_OK) return chk;
  const int64_t need = mk_attn_decode_workspace_bytes(B, Hq, Hkv, D, page_size, max_pages);
  if (need < 0) return MK_ERR_CUDA;  // valid sizes: only the device query can fail
  if (need > mk::dec::kStaticScratchBytes) return MK_ERR_SCRATCH_LIMIT;
  // The lookup happens on the first valid call per device, whether or not
  // these sizes need scratch, so that it never happens later during a stream
  // capture.
  void *scratch = mk::dec::static_scratch_address();
  if (!scratch) return MK_ERR_CUDA;
  return mk::finish_call(
      mk::decode_paged_impl(q, k_cache, v_cache, page_table, seq_lens, o, lse, B, Hq, Hkv, D,
                            page_size, max_pages, num_pages, scale, scratch,
                            mk::dec::kStaticScratchBytes, stream),
      stream);
}

}  // extern "C"
