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
//   * a producer warp streams K and V pages into a two-stage shared-memory
//     ring with TMA (the page is the box: page_size tokens x 1 head x 64
//     elements, 128-byte swizzle), so a page-table gather costs nothing;
//   * four compute warps; a warp owns whole query heads of the group, each
//     lane D/32 dimensions of them.  Per chunk of 32 (or 16) keys a lane forms
//     partial dot products for every key, and a transposing butterfly leaves
//     lane l with the full score of key l; an online base-2 softmax
//     (exp2 on the MUFU unit) then weights the values, which each lane
//     accumulates for its dimensions.
#include <cuda.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>

#include "mk_attn.h"
#include "ptx.cuh"
#include "tma_host.h"

namespace mk {
namespace dec {

constexpr int kWarps = 4;                    // compute warps
constexpr int kThreads = 32 * (kWarps + 1);  // + one producer warp
constexpr int kStages = 2;
constexpr int kMaxSplitsPerSm = 2;           // target CTAs: this many per SM

__device__ int g_status = 0;  // MK_ERR_TIMEOUT or MK_ERR_INVALID_ARG from a decode launch

struct Params {
  const uint16_t *q;          // bf16 [B, Hq, D]
  const int32_t *page_table;  // [B, max_pages]
  const int32_t *seq_lens;    // [B]
  uint16_t *o;                // bf16 [B, Hq, D]
  float *lse;                 // [B, Hq]
  float *part;                // [B, Hq, n_splits, D + 1]; unused with one split
  int B, Hq, Hkv, G;
  int page_size, max_pages, num_pages;
  int n_splits, pages_per_split;
  float scale_log2;           // scale * log2(e)
};

struct Ctl {
  uint64_t full[kStages], empty[kStages];
  int abort;
};

__device__ __forceinline__ void record(int status) { atomicCAS(&g_status, 0, status); }

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

// Lane l holds v[0..CH) (partial sums of CH keys over its dimensions); on
// return v[0] of lane l is the sum over all 32 lanes for key l % CH.  Each
// halving stage keeps the half of the keys selected by one lane bit (high bit
// first) and adds the partner lane's copy of it.
template <int CH>
__device__ __forceinline__ float transpose_reduce(float (&v)[CH]) {
  const int lane = lane_id();
  if constexpr (CH == 16) {
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] += __shfl_xor_sync(0xffffffffu, v[i], 16);
  }
#pragma unroll
  for (int half = CH / 2; half >= 1; half >>= 1) {
    const bool upper = (lane & half) != 0;
#pragma unroll
    for (int i = 0; i < half; ++i) {
      const float send = upper ? v[i] : v[i + half];
      const float keep = upper ? v[i + half] : v[i];
      v[i] = keep + __shfl_xor_sync(0xffffffffu, send, half);
    }
  }
  return v[0];
}

template <int D>
struct Cfg {
  static_assert(D == 64 || D == 128, "head dimension 64 or 128");
  static constexpr int kDimsPerLane = D / 32;  // 2 or 4
  static constexpr int kBoxes = D / 64;        // 128-byte swizzle rows per token
};

// Byte offset, within one K or V page tile, of this lane's D/32 elements of
// token r: the tile is kBoxes boxes of page_size rows x 128 B, each 1024-B
// group of 8 rows stored with its 16-byte chunks permuted (chunk c of row r at
// position c ^ (r % 8)).
template <int D>
__device__ __forceinline__ uint32_t lane_offset(int r, int page_size) {
  const int lane = lane_id();
  if constexpr (D == 128) {
    const int box = lane >> 4, chunk = (lane & 15) >> 1, sub = (lane & 1) * 8;
    return box * page_size * 128 + r * 128 + ((chunk ^ (r & 7)) << 4) + sub;
  } else {
    const int chunk = lane >> 2, sub = (lane & 3) * 4;
    return r * 128 + ((chunk ^ (r & 7)) << 4) + sub;
  }
}

template <int D>
__device__ __forceinline__ void load_lane(const uint8_t *tile, int r, int page_size,
                                          float (&x)[Cfg<D>::kDimsPerLane]) {
  const uint8_t *a = tile + lane_offset<D>(r, page_size);
  if constexpr (D == 128) {
    const uint2 w = *reinterpret_cast<const uint2 *>(a);
    x[0] = bf16_lo(w.x); x[1] = bf16_hi(w.x); x[2] = bf16_lo(w.y); x[3] = bf16_hi(w.y);
  } else {
    const uint32_t w = *reinterpret_cast<const uint32_t *>(a);
    x[0] = bf16_lo(w); x[1] = bf16_hi(w);
  }
}

// Heads per compute warp at most (G <= kWarps * kMaxHeadsPerWarp).
constexpr int kMaxHeadsPerWarp = 4;

template <int D, int CH>
__global__ void __launch_bounds__(kThreads)
    decode_kernel(const __grid_constant__ CUtensorMap tm_k, const __grid_constant__ CUtensorMap tm_v,
                  const Params p) {
  using C = Cfg<D>;
  constexpr int NDL = C::kDimsPerLane;
  const int split = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
  const int PS = p.page_size;
  const int tile_bytes = PS * D * 2;  // one page of K (or V) for one head
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw_addr = smem_addr(smem_raw);
  uint8_t *smem = smem_raw + ((1024u - (raw_addr & 1023u)) & 1023u);
  Ctl *ctl = reinterpret_cast<Ctl *>(smem + kStages * 2 * tile_bytes);
  const int warp = threadIdx.x / 32;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&ctl->full[s], 1);
      mbar_init(&ctl->empty[s], kWarps);
    }
    ctl->abort = 0;
    fence_mbar_init();
  }
  __syncthreads();
  volatile int *abort = &ctl->abort;

  // Pages [first, first + n_pg) of the sequence belong to this split.
  int L = p.seq_lens[b];
  if (L < 0 || L > p.max_pages * PS) {
    if (threadIdx.x == 0) record(MK_ERR_INVALID_ARG);
    L = L < 0 ? 0 : p.max_pages * PS;
  }
  const int n_pages_b = (L + PS - 1) / PS;
  const int first = split * p.pages_per_split;
  const int n_pg = max(0, min(first + p.pages_per_split, n_pages_b) - first);

  if (warp == kWarps) {
    // ------------------------------------------------------------ producer
    const uint64_t pol = l2_policy_evict_first();  // the cache is streamed once
    bool ok = true;
    for (int i = 0; ok && i < n_pg; ++i) {
      const int s = i % kStages;
      ok = mbar_wait_all(&ctl->empty[s], ((i / kStages) & 1) ^ 1, abort);
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
    }
    // Teardown: the loads issued land before the CTA exits.
    for (int i = max(0, n_pg - kStages); i < n_pg; ++i) {
      int local_abort = 0;
      mbar_wait(&ctl->full[i % kStages], (i / kStages) & 1, &local_abort);
    }
  } else {
    // ------------------------------------------------------------- compute
    // This warp's heads: hq = g * G + warp + kWarps * t.
    const int lane = lane_id();
    int n_heads = 0;
    float q[kMaxHeadsPerWarp][NDL], acc[kMaxHeadsPerWarp][NDL];
    float m[kMaxHeadsPerWarp], l[kMaxHeadsPerWarp];
#pragma unroll
    for (int t = 0; t < kMaxHeadsPerWarp; ++t) {
      const int gi = warp + kWarps * t;
      m[t] = -INFINITY;
      l[t] = 0.f;
#pragma unroll
      for (int e = 0; e < NDL; ++e) acc[t][e] = 0.f, q[t][e] = 0.f;
      if (gi < p.G) {
        n_heads = t + 1;
        const uint16_t *qr = p.q + ((int64_t)b * p.Hq + g * p.G + gi) * D + lane * NDL;
#pragma unroll
        for (int e = 0; e < NDL; ++e)
          q[t][e] = __uint_as_float((uint32_t)qr[e] << 16) * p.scale_log2;
      }
    }
    bool ok = true;
    for (int i = 0; ok && i < n_pg; ++i) {
      const int s = i % kStages;
      ok = mbar_wait_all(&ctl->full[s], (i / kStages) & 1, abort);
      if (!ok) break;
      const uint8_t *kt = smem + s * 2 * tile_bytes;
      const uint8_t *vt = kt + tile_bytes;
      const int key0 = (first + i) * PS;  // position of the page's first slot
#pragma unroll
      for (int t = 0; t < kMaxHeadsPerWarp; ++t) {
        if (t < n_heads) {
        for (int c0 = 0; c0 < PS; c0 += CH) {
          // Partial scores of keys c0 .. c0+CH-1 over this lane's dimensions.
          float sc[CH];
#pragma unroll
          for (int k = 0; k < CH; ++k) {
            float kx[NDL];
            load_lane<D>(kt, c0 + k, PS, kx);
            float a = 0.f;
#pragma unroll
            for (int e = 0; e < NDL; ++e) a = fmaf(q[t][e], kx[e], a);
            sc[k] = a;
          }
          float sk = transpose_reduce<CH>(sc);  // lane's key: c0 + lane % CH
          const bool valid = key0 + c0 + (lane % CH) < L;
          sk = valid ? sk : -INFINITY;
          float cmax = sk;
#pragma unroll
          for (int off = 16; off >= 1; off >>= 1) cmax = fmaxf(cmax, __shfl_xor_sync(0xffffffffu, cmax, off));
          const float m_new = fmaxf(m[t], cmax);
          // (m_new = -inf only if no key has been visible yet: nothing to scale.)
          const float alpha = m_new == -INFINITY ? 1.f : ex2_approx(m[t] - m_new);
          const float pk = valid ? ex2_approx(sk - m_new) : 0.f;
          float psum = lane < CH ? pk : 0.f;
#pragma unroll
          for (int off = 16; off >= 1; off >>= 1) psum += __shfl_xor_sync(0xffffffffu, psum, off);
          l[t] = l[t] * alpha + psum;
          m[t] = m_new;
#pragma unroll
          for (int e = 0; e < NDL; ++e) acc[t][e] *= alpha;
#pragma unroll
          for (int k = 0; k < CH; ++k) {
            const float pj = __shfl_sync(0xffffffffu, pk, k);
            float vx[NDL];
            load_lane<D>(vt, c0 + k, PS, vx);
#pragma unroll
            for (int e = 0; e < NDL; ++e) acc[t][e] = fmaf(pj, vx[e], acc[t][e]);
          }
        }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&ctl->empty[s]);
    }
    if (!ok) *abort = 1;
    // Results: o = acc / l, lse = ln 2 * (m + log2 l); l = 0 (no key) gives
    // o = 0 and lse = -inf.
#pragma unroll
    for (int t = 0; t < kMaxHeadsPerWarp; ++t) {
      if (t >= n_heads) continue;
      const int hq = g * p.G + warp + kWarps * t;
      const float inv_l = l[t] > 0.f ? 1.f / l[t] : 0.f;
      const float lse = l[t] > 0.f ? (m[t] + log2f(l[t])) * 0.69314718055994530942f : -INFINITY;
      if (p.n_splits == 1) {
        uint16_t *orow = p.o + ((int64_t)b * p.Hq + hq) * D + lane * NDL;
#pragma unroll
        for (int e = 0; e < NDL; e += 2) {
          const uint32_t w = pack_bf16x2(acc[t][e] * inv_l, acc[t][e + 1] * inv_l);
          *reinterpret_cast<uint32_t *>(orow + e) = w;
        }
        if (lane == 0) p.lse[(int64_t)b * p.Hq + hq] = lse;
      } else {
        float *pr = p.part + (((int64_t)b * p.Hq + hq) * p.n_splits + split) * (D + 1);
#pragma unroll
        for (int e = 0; e < NDL; ++e) pr[lane * NDL + e] = acc[t][e] * inv_l;
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
  constexpr int NDL = Cfg<D>::kDimsPerLane;
  const int row = blockIdx.x * 4 + threadIdx.x / 32;  // b * Hq + h
  if (row >= p.B * p.Hq) return;
  const int lane = lane_id();
  const float *pr = p.part + (int64_t)row * p.n_splits * (D + 1);
  float mx = -INFINITY;
  for (int s = 0; s < p.n_splits; ++s) mx = fmaxf(mx, pr[s * (D + 1) + D]);
  float acc[NDL];
#pragma unroll
  for (int e = 0; e < NDL; ++e) acc[e] = 0.f;
  float wsum = 0.f;
  if (mx > -INFINITY) {
    for (int s = 0; s < p.n_splits; ++s) {
      const float w = exp2f((pr[s * (D + 1) + D] - mx) * 1.4426950408889634f);
      wsum += w;
#pragma unroll
      for (int e = 0; e < NDL; ++e) acc[e] = fmaf(w, pr[s * (D + 1) + lane * NDL + e], acc[e]);
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

// Splits per (b, g): enough CTAs for kMaxSplitsPerSm per SM, never more than
// the pages of the longest possible sequence.
static void plan_splits(int B, int Hkv, int max_pages, int sms, int &n_splits, int &pps) {
  const int64_t units = (int64_t)B * Hkv;
  int want = (int)((kMaxSplitsPerSm * (int64_t)sms + units - 1) / units);
  want = want < 1 ? 1 : (want > max_pages ? max_pages : want);
  pps = (max_pages + want - 1) / want;
  n_splits = (max_pages + pps - 1) / pps;
}

static size_t smem_bytes(int D, int page_size) {
  return (size_t)kStages * 2 * page_size * D * 2 + sizeof(Ctl) + 1024;
}

template <int D, int CH>
static int launch(const CUtensorMap &tk, const CUtensorMap &tv, const Params &p, cudaStream_t st) {
  const size_t sm = smem_bytes(D, p.page_size);
  if (cudaFuncSetAttribute(decode_kernel<D, CH>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)sm) != cudaSuccess)
    return MK_ERR_CUDA;
  const dim3 grid(p.n_splits, p.Hkv, p.B);
  decode_kernel<D, CH><<<grid, kThreads, sm, st>>>(tk, tv, p);
  if (cudaGetLastError() != cudaSuccess) return MK_ERR_CUDA;
  if (p.n_splits > 1) {
    merge_kernel<D><<<(p.B * p.Hq + 3) / 4, 128, 0, st>>>(p);
    if (cudaGetLastError() != cudaSuccess) return MK_ERR_CUDA;
  }
  return MK_OK;
}

}  // namespace dec

int decode_take_status() {
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
  int n_splits = 1, pps = max_pages;
  mk::dec::plan_splits(B, Hkv, max_pages, sms, n_splits, pps);
  if (n_splits == 1) return 0;
  return (int64_t)B * Hq * n_splits * (D + 1) * 4;
}

int mk_attn_decode_paged(const void *q, const void *k_cache, const void *v_cache,
                         const int32_t *page_table, const int32_t *seq_lens, void *o, float *lse,
                         int B, int Hq, int Hkv, int D, int page_size, int max_pages,
                         int num_pages, float scale, void *workspace, int64_t workspace_bytes,
                         void *stream) {
  using namespace mk;
  if (!q || !k_cache || !v_cache || !page_table || !seq_lens || !o || !lse)
    return MK_ERR_INVALID_ARG;
  if (B < 1 || Hq < 1 || Hkv < 1 || Hq % Hkv != 0 || max_pages < 1 || num_pages < 1)
    return MK_ERR_INVALID_ARG;
  if (B > 65535 || Hkv > 65535) return MK_ERR_UNSUPPORTED;  // grid y / z
  if (!std::isfinite(scale)) return MK_ERR_INVALID_ARG;
  if (D != 64 && D != 128) return MK_ERR_UNSUPPORTED;
  if (page_size != 16 && page_size != 32 && page_size != 64 && page_size != 128)
    return MK_ERR_UNSUPPORTED;
  const int G = Hq / Hkv;
  if (G > dec::kWarps * dec::kMaxHeadsPerWarp) return MK_ERR_UNSUPPORTED;
  if ((int64_t)num_pages * page_size > INT32_MAX || (int64_t)max_pages * page_size > INT32_MAX)
    return MK_ERR_INVALID_ARG;
  auto misaligned = [](const void *ptr, uintptr_t a) { return (reinterpret_cast<uintptr_t>(ptr) & (a - 1)) != 0; };
  if (misaligned(q, 16) || misaligned(k_cache, 16) || misaligned(v_cache, 16) || misaligned(o, 16) ||
      misaligned(lse, 4) || misaligned(page_table, 4) || misaligned(seq_lens, 4))
    return MK_ERR_ALIGNMENT;
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
  p.page_size = page_size;
  p.max_pages = max_pages;
  p.num_pages = num_pages;
  p.scale_log2 = scale * 1.4426950408889634f;
  dec::plan_splits(B, Hkv, max_pages, sms, p.n_splits, p.pages_per_split);
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
  if (D == 128)
    return page_size == 16 ? dec::launch<128, 16>(tk, tv, p, st) : dec::launch<128, 32>(tk, tv, p, st);
  return page_size == 16 ? dec::launch<64, 16>(tk, tv, p, st) : dec::launch<64, 32>(tk, tv, p, st);
}

}  // extern "C"
