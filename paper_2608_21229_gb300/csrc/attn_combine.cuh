// attn_combine.cuh -- merge the parts of split items.
//
// When the items of a launch do not divide evenly over the GPU's CTA pairs,
// the last items are split by key range into parts that run on otherwise idle
// pairs.  Each part p of an item leaves, for every query row, its own
// normalised output O_p = (sum_j p_j v_j) / l_p and L_p = m_p + log l_p over
// its keys.  Over all keys of the item the softmax normaliser is
// l = sum_p exp(L_p), so the item's output is
//   O = sum_p exp(L_p - L) O_p   with   L = log sum_p exp(L_p),
// computed here with L_max subtracted first: one warp per query row, D / 32
// head-dim columns per lane.
#pragma once
#include <cuda_bf16.h>

#include "common.cuh"
#include "ptx.cuh"

namespace rc {

constexpr int kMaxParts = 8;

// grid = (ceil(rows / 8), jobs), 256 threads: one warp per query row, all
// parts' loads issued before any is used.
template <int D>
__global__ void __launch_bounds__(256) combine_parts_kernel(const CombineJob* __restrict__ jobs,
                                                            const float* __restrict__ part_o,
                                                            const float* __restrict__ part_lse, int rows_per_part,
                                                            __nv_bfloat16* __restrict__ out, float* __restrict__ lse,
                                                            int64_t row_stride, int num_heads) {
  static_assert(D == 128 || D == 64, "four or two columns per lane");
  constexpr int kC = D / 32;
  grid_dependency_wait();  // the attention kernel's parts are complete
  if (threadIdx.x == 0) grid_launch_dependents();
  const CombineJob job = jobs[blockIdx.y];
  const int r = blockIdx.x * (blockDim.x / 32) + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (r >= job.q_rows) return;
  const int np = min(job.nparts, kMaxParts);
  float L[kMaxParts];
  float v[kMaxParts][kC];
#pragma unroll
  for (int p = 0; p < kMaxParts; ++p) {
    if (p < np) {
      const int64_t row = static_cast<int64_t>(job.part0 + p) * rows_per_part + r;
      L[p] = part_lse[row];
      if constexpr (kC == 4) {
        const float4 x = reinterpret_cast<const float4*>(part_o + row * D)[lane];
        v[p][0] = x.x, v[p][1] = x.y, v[p][2] = x.z, v[p][3] = x.w;
      } else {
        const float2 x = reinterpret_cast<const float2*>(part_o + row * D)[lane];
        v[p][0] = x.x, v[p][1] = x.y;
      }
    } else {
      L[p] = -INFINITY;
#pragma unroll
      for (int c = 0; c < kC; ++c) v[p][c] = 0.f;
    }
  }
  float lmax = L[0];
#pragma unroll
  for (int p = 1; p < kMaxParts; ++p) lmax = fmaxf(lmax, L[p]);
  float acc[kC];
#pragma unroll
  for (int c = 0; c < kC; ++c) acc[c] = 0.f;
  float wsum = 0.f;
#pragma unroll
  for (int p = 0; p < kMaxParts; ++p) {
    const float w = p < np ? expf(L[p] - lmax) : 0.f;
    wsum += w;
#pragma unroll
    for (int c = 0; c < kC; ++c) acc[c] += w * v[p][c];
  }
  const float inv = 1.0f / wsum;
  const int64_t row = static_cast<int64_t>(job.q_row0) + r;
  __nv_bfloat16* dst = out + row * row_stride + static_cast<int64_t>(job.head) * D;
  __nv_bfloat162 lo = __floats2bfloat162_rn(acc[0] * inv, acc[1] * inv);
  if constexpr (kC == 4) {
    __nv_bfloat162 hi = __floats2bfloat162_rn(acc[2] * inv, acc[3] * inv);
    uint2 packed;
    packed.x = *reinterpret_cast<uint32_t*>(&lo);
    packed.y = *reinterpret_cast<uint32_t*>(&hi);
    reinterpret_cast<uint2*>(dst)[lane] = packed;
  } else {
    reinterpret_cast<__nv_bfloat162*>(dst)[lane] = lo;
  }
  if (lse && lane == 0) lse[row * num_heads + job.head] = lmax + logf(wsum);
}

}  // namespace rc
