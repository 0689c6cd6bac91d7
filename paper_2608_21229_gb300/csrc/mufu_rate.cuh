// mufu_rate.cuh -- measures the exponential rate of the GPU's special-function
// unit (ex2.approx.f32), the secondary limit of the softmax: one exponential
// per visible (query, key) pair of one head against 4 d tensor FLOPs.
//
// One CTA per SM (the dynamic shared memory it asks for leaves room for no
// second one), 8 warps, each thread running kEx2Chains independent chains of
// x <- 2^x - 1.5 (the add keeps the values bounded: the chain settles at
// x = -1).  Each CTA times its loop with clock64 between two __syncthreads and
// writes the cycles; the host divides the CTA's exponentials by them.
#pragma once

#include <cstdint>

#include "ptx.cuh"

namespace rc {

constexpr int kEx2Threads = 256;
constexpr int kEx2Chains = 8;
constexpr int kEx2Iters = 2048;
constexpr int kEx2MaxBlocks = 1024;
constexpr int kEx2Smem = 120 * 1024;

__device__ long long g_ex2_cycles[kEx2MaxBlocks];
__device__ float g_ex2_sink;

__global__ void __launch_bounds__(kEx2Threads, 1) ex2_rate_kernel(float x0) {
  float x[kEx2Chains];
#pragma unroll
  for (int i = 0; i < kEx2Chains; ++i) x[i] = x0 - 0.01f * static_cast<float>(i) - 1e-5f * static_cast<float>(threadIdx.x);
  __syncthreads();
  const long long t0 = clock64();
#pragma unroll 4
  for (int it = 0; it < kEx2Iters; ++it) {
#pragma unroll
    for (int i = 0; i < kEx2Chains; ++i) x[i] = ex2_approx(x[i]) - 1.5f;
  }
  __syncthreads();
  const long long t1 = clock64();
  if (threadIdx.x == 0 && blockIdx.x < kEx2MaxBlocks) g_ex2_cycles[blockIdx.x] = t1 - t0;
  float s = 0.f;
#pragma unroll
  for (int i = 0; i < kEx2Chains; ++i) s += x[i];
  if (s == 12345.0f) g_ex2_sink = s;  // keeps the chains alive; never true (each x is near -1)
}

}  // namespace rc
