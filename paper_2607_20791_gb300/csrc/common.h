// Host-side helpers shared by the library's translation units.
#pragma once

#include <cuda_runtime.h>

#include <cstdarg>
#include <cstdint>
#include <cstdio>

#include "rgd.h"

namespace rgd {

// Sets the calling thread's error string and returns `code`.
int set_error(int code, const char* fmt, ...);
void clear_error();

inline int cuda_error(cudaError_t e, const char* what) {
  return set_error(RGD_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Opts a kernel into `bytes` of dynamic shared memory once per process.
template <typename Kernel>
int ensure_smem(Kernel k, int bytes, bool* done) {
  if (*done) return RGD_OK;
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e != cudaSuccess) return cuda_error(e, "cudaFuncSetAttribute");
  *done = true;
  return RGD_OK;
}

// Argument checks of rgd_sample_head_gated (shared with rgd_decode_step, which
// checks them before launching its first kernel).
int check_gated_head(const char* fn, int32_t rows, int32_t vocab, int32_t dtype, const void* logits,
                     const float* temperature, const float* min_p, const uint64_t* seed, const int32_t* token_out,
                     const rgd_trie* trie, int32_t rows_per_group, int32_t max_len, const rgd_gate_state* state);

}  // namespace rgd

#define RGD_CHECK_ARG(cond, ...)                                        \
  do {                                                                  \
    if (!(cond)) return ::rgd::set_error(RGD_ERR_INVALID_ARG, __VA_ARGS__); \
  } while (0)
