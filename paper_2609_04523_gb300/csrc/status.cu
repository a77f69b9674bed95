// status.cu -- the library-wide entry points of the C ABI: status strings,
// the device status check that covers every kernel family, and the version.
#include <cuda_runtime.h>

#include <atomic>
#include <cstdlib>
#include <cstring>
#include <mutex>

#include "mk_attn.h"
#include "tma_host.h"

namespace mk {
namespace {
constexpr mk_attn_tuning kDefaultTuning = {0, MK_SCHED_SNAKE, 8.0f, 24, 2, 3};
std::mutex g_tuning_mu;
mk_attn_tuning g_tuning = kDefaultTuning;
}  // namespace

mk_attn_tuning current_tuning() {
  std::lock_guard<std::mutex> lock(g_tuning_mu);
  return g_tuning;
}

namespace {
constexpr int kMaxDevices = 64;
std::atomic<unsigned> g_launched[kMaxDevices];  // bit f: family f enqueued on device
}  // namespace

void mark_launched(Family family) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return;
  g_launched[dev].fetch_or(1u << family, std::memory_order_relaxed);
}

bool launched(Family family) {
  int dev = 0;
  // Unknown device: report "launched" so that the status word is read.
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return true;
  return (g_launched[dev].load(std::memory_order_relaxed) >> family) & 1u;
}

int finish_call(int status, void *stream) {
  static const bool debug = [] {
    const char *e = std::getenv("MK_ATTN_DEBUG");
    return e != nullptr && e[0] != '\0' && std::strcmp(e, "0") != 0;
  }();
  if (status != MK_OK || !debug) return status;
  return mk_attn_check_status(stream);
}
}  // namespace mk

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
    case MK_ERR_BOUNDS: return "a store index check of the check build failed";
    default: return "unknown status";
  }
}

// Synchronises the stream, then reads and clears the status words of the
// forward, backward, decode and latent decode kernels; the first nonzero one
// in that order is reported.
int mk_attn_check_status(void *stream) {
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (cudaStreamSynchronize(st) != cudaSuccess) return MK_ERR_CUDA;
  const int hf = mk::fwd_take_status();
  const int hb = mk::bwd_take_status();
  const int hd = mk::decode_take_status();
  const int hm = mk::mla_take_status();
  return hf != 0 ? hf : (hb != 0 ? hb : (hd != 0 ? hd : hm));
}

int mk_attn_set_tuning(const mk_attn_tuning *t) {
  mk_attn_tuning v = mk::kDefaultTuning;
  if (t) {
    if (t->ctas < 0 || t->ctas > 65535) return MK_ERR_INVALID_ARG;
    if (t->schedule < MK_SCHED_SNAKE || t->schedule > MK_SCHED_DYNAMIC) return MK_ERR_INVALID_ARG;
    if (!(t->rescale_log2 >= 0.0f && t->rescale_log2 <= 16.0f)) return MK_ERR_INVALID_ARG;
    if (t->split_ctas_per_sm < 1 || t->split_ctas_per_sm > 64) return MK_ERR_INVALID_ARG;
    if (t->split_min_pages < 1 || t->split_min_pages > 4096) return MK_ERR_INVALID_ARG;
    if (t->mla_split_ctas_per_sm < 1 || t->mla_split_ctas_per_sm > 64) return MK_ERR_INVALID_ARG;
    v = *t;
  }
  std::lock_guard<std::mutex> lock(mk::g_tuning_mu);
  mk::g_tuning = v;
  return MK_OK;
}

int mk_attn_get_tuning(mk_attn_tuning *t) {
  if (!t) return MK_ERR_INVALID_ARG;
  *t = mk::current_tuning();
  return MK_OK;
}

int mk_attn_version(void) { return 500; }

}  // extern "C"
