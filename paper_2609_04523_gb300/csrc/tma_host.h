// tma_host.h -- host-side TMA tensor-map encoding shared by the kernels.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include <cstdint>
#include <mutex>

#include "mk_attn.h"

namespace mk {

// cuTensorMapEncodeTiled through the runtime's driver entry point (no -lcuda).
inline PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
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

// [tokens, heads, D] bf16, boxes of box_tokens tokens x 1 head x 64 elements
// (one 128-byte swizzle row per token), 128-byte swizzle.
inline bool encode_tokens_heads_dim(CUtensorMap *map, const void *base, uint64_t tokens,
                                    uint64_t heads, uint64_t D, uint32_t box_tokens) {
  auto enc = tensor_map_encoder();
  if (!enc) return false;
  const cuuint64_t dims[3] = {D, heads, tokens};
  const cuuint64_t strides[2] = {D * 2, heads * D * 2};
  const cuuint32_t box[3] = {64, 1, box_tokens};
  const cuuint32_t estr[3] = {1, 1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(base), dims, strides,
             box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Launch configuration of a kernel that follows another kernel of the same
// call on `stream` and reads its results: with programmatic stream
// serialization it may be scheduled while the first kernel drains, and it calls
// griddep_wait() before reading anything.  Use as a local: cfg.attrs points
// into the object.
struct DependentLaunch {
  cudaLaunchConfig_t cfg;
  cudaLaunchAttribute attr[1];
  DependentLaunch(dim3 grid, dim3 block, size_t smem, cudaStream_t stream) {
    cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
  }
  DependentLaunch(const DependentLaunch &) = delete;
  DependentLaunch &operator=(const DependentLaunch &) = delete;
};

// The process-wide launch tuning (mk_attn_set_tuning), defaults applied.
mk_attn_tuning current_tuning();

// Read and clear the device status word of each kernel family (each defined
// with its kernels).  A family that has enqueued no kernel on the current
// device reads as 0 without touching the device, so that a status check never
// loads the code and device arrays of a family the caller has not used.
int fwd_take_status();
int bwd_take_status();
int decode_take_status();
int mla_take_status();

enum Family { kFamFwd = 0, kFamBwd = 1, kFamDecode = 2, kFamMla = 3 };
// Records that `family` enqueues kernels on the current device (called by
// each launcher before its first launch), and whether it has.
void mark_launched(Family family);
bool launched(Family family);

// Check mode: with MK_ATTN_DEBUG set to a nonzero value in the environment
// (read once, at the first call), every entry point that enqueued work
// synchronises its stream and returns what mk_attn_check_status reports
// instead of MK_OK.  Without it, returns `status` unchanged.
int finish_call(int status, void *stream);

}  // namespace mk
