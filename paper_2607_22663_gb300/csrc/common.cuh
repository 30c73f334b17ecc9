// Internal helpers shared by the translation units of libmbe.
#pragma once
#include <cstdint>
#include <cuda_runtime.h>
#include "mbe.h"

namespace mbe {

// Each translation unit owns one device error word (no relocatable device
// code is needed); mbe_get_device_error() reads and clears all of them.
#define MBE_DEFINE_ERROR_WORD(accessor)                                                     \
  static __device__ unsigned int g_error_word;                                              \
  uint32_t accessor() {                                                                     \
    unsigned int v = 0, z = 0;                                                              \
    if (cudaMemcpyFromSymbol(&v, g_error_word, sizeof(v)) != cudaSuccess) return 0xFFFFFFFFu; \
    cudaMemcpyToSymbol(g_error_word, &z, sizeof(z));                                        \
    return v;                                                                               \
  }

uint32_t edit_decide_take_error();
uint32_t kv_write_take_error();
uint32_t attention_take_error();
uint32_t denoise_take_error();
uint32_t refresh_take_error();
uint32_t lm_head_take_error();
uint32_t train_take_error();

// Wall-clock limit (ns) of the ordinary mbarrier waits of kernels launched
// from now on (mbe_set_wait_limit_ns; 1 s by default).
uint64_t wait_limit_ns();

inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Remembers (per host thread) the last CUDA failure seen by the library.
void record_cuda_error(cudaError_t e, const char* where);

inline mbe_status launch_status(const char* where = "kernel launch") {
  cudaError_t e = cudaGetLastError();
  if (e == cudaSuccess) return MBE_OK;
  record_cuda_error(e, where);
  return MBE_ERR_CUDA;
}

}  // namespace mbe
