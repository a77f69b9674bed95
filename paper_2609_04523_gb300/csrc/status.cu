// status.cu -- the library-wide entry points of the C ABI: status strings,
// the device status check that covers every kernel family, and the version.
#include <cuda_runtime.h>

#include "mk_attn.h"
#include "tma_host.h"

extern "C" {

const char *mk_attn_error_string(int status) {
  switch (status) {
    case MK_OK: return "success";
    case MK_ERR_INVALID_ARG: return "invalid argument";
    case MK_ERR_UNSUPPORTED: return "unsupported head dimension (64 or 128)";
    case MK_ERR_ALIGNMENT: return "pointer not 16-byte aligned";
    case MK_ERR_CUDA: return "CUDA call failed";
    case MK_ERR_TIMEOUT: return "kernel wait timed out";
    case MK_ERR_SCRATCH_LIMIT: return "sizes need more scratch than the static decode array holds";
    default: return "unknown status";
  }
}

// Synchronises the stream, then reads and clears the status words of the
// forward, backward and decode kernels; the forward's is reported first.
int mk_attn_check_status(void *stream) {
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (cudaStreamSynchronize(st) != cudaSuccess) return MK_ERR_CUDA;
  const int hf = mk::fwd_take_status();
  const int hb = mk::bwd_take_status();
  const int hd = mk::decode_take_status();
  return hf != 0 ? hf : (hb != 0 ? hb : hd);
}

int mk_attn_version(void) { return 400; }

}  // extern "C"
