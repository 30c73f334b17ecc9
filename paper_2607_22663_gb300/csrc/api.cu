// Status strings, version, the last CUDA error and the device error word query of libmbe.
#include <atomic>
#include <cstdio>
#include "common.cuh"

namespace mbe {
namespace {
thread_local char g_last_error[256] = "no CUDA error recorded";
std::atomic<uint64_t> g_wait_limit_ns{MBE_DEFAULT_WAIT_LIMIT_NS};
}
uint64_t wait_limit_ns() { return g_wait_limit_ns.load(std::memory_order_relaxed); }
void record_cuda_error(cudaError_t e, const char* where) {
  snprintf(g_last_error, sizeof(g_last_error), "%s: %s (%s)", where, cudaGetErrorName(e), cudaGetErrorString(e));
}
}  // namespace mbe

extern "C" const char* mbe_last_error_string(void) { return mbe::g_last_error; }

extern "C" mbe_status mbe_get_device_error(cudaStream_t stream, uint32_t* flags_or_null) {
  if (cudaStreamSynchronize(stream) != cudaSuccess) return MBE_ERR_CUDA;
  uint32_t bits = 0;
  const uint32_t parts[7] = {mbe::edit_decide_take_error(), mbe::kv_write_take_error(), mbe::attention_take_error(),
                             mbe::denoise_take_error(),     mbe::refresh_take_error(),  mbe::lm_head_take_error(),
                             mbe::train_take_error()};
  for (uint32_t v : parts) {
    if (v == 0xFFFFFFFFu) return MBE_ERR_CUDA;
    bits |= v;
  }
  if (flags_or_null) *flags_or_null = bits;
  if (bits == 0) return MBE_OK;
  return (bits & MBE_DEVERR_TIMEOUT) ? MBE_ERR_TIMEOUT : MBE_ERR_DEVICE_CHECK;
}

extern "C" const char* mbe_status_string(mbe_status status) {
  switch (status) {
    case MBE_OK: return "ok";
    case MBE_ERR_INVALID_ARG: return "invalid argument";
    case MBE_ERR_UNSUPPORTED: return "unsupported configuration";
    case MBE_ERR_CUDA: return "CUDA error";
    case MBE_ERR_TIMEOUT: return "device wait timed out";
    case MBE_ERR_WORKSPACE: return "workspace missing or too small";
    case MBE_ERR_DEVICE_CHECK: return "device-side argument check failed";
  }
  return "unknown status";
}

extern "C" int32_t mbe_version(void) { return 100; }

extern "C" uint64_t mbe_set_wait_limit_ns(uint64_t limit_ns) {
  return mbe::g_wait_limit_ns.exchange(limit_ns, std::memory_order_relaxed);
}
