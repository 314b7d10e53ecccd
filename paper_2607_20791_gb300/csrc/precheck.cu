// Residual-stream precheck (App. A): a logistic readout of each prompt's
// last-token activation decides, once per prompt, whether the greedy probe can
// be skipped.  z = w . h + b, p = sigmoid(z); p <= theta skips the probe: the
// group's gate state takes the non-refusal outcome before any probe token and
// its probe row is masked, so only its sample rows decode.
//
// One block per group: each thread reads a strided share of the group's d
// activations (consecutive threads, consecutive elements: coalesced), keeps an
// fp32 partial dot product, and the block reduces them (warp shuffles, then
// shared memory).  The readout is d + 1 parameters, so the kernel is a
// launch-latency-bound GEMV.
#include <cuda_bf16.h>

#include <cmath>

#include "common.h"

namespace rgd {
namespace {

constexpr int kPrecheckThreads = 256;

template <typename T>
__device__ __forceinline__ float load_act(const T* p, int64_t i);
template <>
__device__ __forceinline__ float load_act<float>(const float* p, int64_t i) {
  return __ldg(p + i);
}
template <>
__device__ __forceinline__ float load_act<uint16_t>(const uint16_t* p, int64_t i) {
  return __uint_as_float((uint32_t)__ldg(p + i) << 16);  // bf16 widened exactly
}

template <typename T>
__global__ void __launch_bounds__(kPrecheckThreads)
    precheck_kernel(int32_t d, const T* __restrict__ h, const float* __restrict__ w, float bias, float theta,
                    int32_t rows_per_group, float* prob_out, rgd_gate_state* state, uint8_t* row_active) {
  __shared__ float part[kPrecheckThreads / 32];
  const int g = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const T* hg = h + (int64_t)g * d;
  float acc = 0.f;
  // (unrolled so that a thread's loads are all in flight together; the sums
  // stay in index order)
#pragma unroll 16
  for (int i = tid; i < d; i += kPrecheckThreads) acc = fmaf(__ldg(w + i), load_act<T>(hg, i), acc);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  if (lane == 0) part[warp] = acc;
  __syncthreads();
  if (tid != 0) return;
  float z = bias;
  for (int k = 0; k < kPrecheckThreads / 32; ++k) z += part[k];
  const float p = 1.f / (1.f + expf(-z));
  if (prob_out) prob_out[g] = p;
  if (!(p <= theta)) return;
  rgd_gate_state s = state[g];
  if (s.decision != RGD_PENDING || s.steps != 0 || s.done) return;  // the probe has already begun
  s.decision = RGD_NON_REFUSAL;
  s.done = 1;
  s.decisive_step = -1;
  state[g] = s;
  if (row_active) row_active[(int64_t)g * rows_per_group] = 0;
}

}  // namespace
}  // namespace rgd

using namespace rgd;

extern "C" int rgd_residual_precheck(int32_t groups, int32_t d, int32_t dtype, const void* h, const float* w,
                                     float bias, float theta, int32_t rows_per_group, float* prob_out,
                                     rgd_gate_state* state, uint8_t* row_active, int32_t* dev_status,
                                     rgd_stream_t stream) {
  clear_error();
  (void)dev_status;  // nothing on the device can go wrong for valid arguments
  RGD_CHECK_ARG(groups >= 0 && d >= 1 && rows_per_group >= 1, "rgd_residual_precheck: bad groups/d/rows_per_group");
  RGD_CHECK_ARG(dtype == RGD_F32 || dtype == RGD_BF16, "rgd_residual_precheck: dtype must be RGD_F32 or RGD_BF16");
  RGD_CHECK_ARG(theta >= 0.f && theta <= 1.f, "rgd_residual_precheck: theta must be in [0, 1]");
  RGD_CHECK_ARG(std::isfinite(bias), "rgd_residual_precheck: bias must be finite");
  if (groups == 0) return RGD_OK;
  RGD_CHECK_ARG(h != nullptr && w != nullptr && state != nullptr, "rgd_residual_precheck: h/w/state NULL");
  cudaStream_t st = (cudaStream_t)stream;
  if (dtype == RGD_F32)
    precheck_kernel<float><<<groups, kPrecheckThreads, 0, st>>>(d, static_cast<const float*>(h), w, bias, theta,
                                                                 rows_per_group, prob_out, state, row_active);
  else
    precheck_kernel<uint16_t><<<groups, kPrecheckThreads, 0, st>>>(d, static_cast<const uint16_t*>(h), w, bias,
                                                                    theta, rows_per_group, prob_out, state, row_active);
  cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? RGD_OK : cuda_error(e, "residual_precheck launch");
}
