// cache_fp8.cuh -- the write of the E4M3 reference cache (the approximate
// variant of the exact cache of Sec. 3.3, Eq. 2): the cached rows' K and V
// quantised per (128-row tile of one request, head) with one fp32 scale each:
//   amax = max |x| over the tile's rows and the head's 128 columns
//   s    = amax / 448,  code = E4M3(x * (448 / amax))   (0 when amax = 0)
// with IEEE fp32 division and multiply and round-to-nearest-even conversion.
// Layout of one layer:
//   k8     [rows_pad, H, 128]   codes, rows in cache order
//   vt8    [H, 128, rows_pad]   codes of V, transposed per head (K-major B
//                               operand of the P.V MMA)
//   scales [rows_pad / 128, H]  float4 (s_K, s_V, log2 s_V, 1 / s_V); the last
//                               two (0 when s_V = 0) spare the attention kernel a
//                               logarithm and a division per tile
// Each request's rows start on a 128-row boundary; pad rows hold code 0.
#pragma once
#include <cstdint>
#include <cuda_bf16.h>

#include "ptx.cuh"

namespace rc {

// One 128-row tile of the cache: rows [src_row0, src_row0 + valid) of the
// prefill tensors go to rows [dst_row0, dst_row0 + 128) of the cache.
struct QuantTile {
  int32_t src_row0, valid, dst_row0, pad;
};

__device__ __forceinline__ float block_amax_256(float v, float* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
  __syncthreads();
  float r = red[0];
#pragma unroll
  for (int w = 1; w < 8; ++w) r = fmaxf(r, red[w]);
  return r;
}

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

// grid (tiles, H), 256 threads: thread i holds row (i >> 4) + 16 r, columns
// [8 (i & 15), 8 (i & 15) + 8) of the tile, r = 0..7.
__global__ void __launch_bounds__(256) quantize_cache_kernel(const QuantTile* __restrict__ tiles,
                                                             const uint4* __restrict__ k, const uint4* __restrict__ v,
                                                             uint8_t* __restrict__ k8, uint8_t* __restrict__ vt8,
                                                             float4* __restrict__ scales, int H, int64_t rows_pad) {
  constexpr int D = 128;
  __shared__ float red[2][8];
  __shared__ __align__(16) uint8_t vt[D][128 + 16];  // V^T codes of the tile: [d][row]
  const QuantTile t = tiles[blockIdx.x];
  const int h = blockIdx.y;
  const int c = threadIdx.x & 15;
  const int r0 = threadIdx.x >> 4;
  const int64_t row_u4 = static_cast<int64_t>(H) * D / 8;
  uint4 kv[8], vv[8];
  float ka = 0.f, va = 0.f;
#pragma unroll
  for (int r = 0; r < 8; ++r) {
    const int row = r0 + 16 * r;
    if (row < t.valid) {
      const int64_t at = static_cast<int64_t>(t.src_row0 + row) * row_u4 + h * (D / 8) + c;
      kv[r] = k[at];
      vv[r] = v[at];
    } else {
      kv[r] = make_uint4(0, 0, 0, 0);
      vv[r] = make_uint4(0, 0, 0, 0);
    }
    const uint32_t kw[4] = {kv[r].x, kv[r].y, kv[r].z, kv[r].w};
    const uint32_t vw[4] = {vv[r].x, vv[r].y, vv[r].z, vv[r].w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      ka = fmax3(ka, fabsf(bf16_lo(kw[e])), fabsf(bf16_hi(kw[e])));
      va = fmax3(va, fabsf(bf16_lo(vw[e])), fabsf(bf16_hi(vw[e])));
    }
  }
  const float kmax = block_amax_256(ka, red[0]);
  const float vmax = block_amax_256(va, red[1]);
  const float kinv = kmax > 0.f ? __fdiv_rn(448.f, kmax) : 0.f;
  const float vinv = vmax > 0.f ? __fdiv_rn(448.f, vmax) : 0.f;
  uint8_t* krow = k8 + static_cast<int64_t>(t.dst_row0) * H * D + static_cast<int64_t>(h) * D + 8 * c;
#pragma unroll
  for (int r = 0; r < 8; ++r) {
    const int row = r0 + 16 * r;
    const uint32_t kw[4] = {kv[r].x, kv[r].y, kv[r].z, kv[r].w};
    const uint32_t vw[4] = {vv[r].x, vv[r].y, vv[r].z, vv[r].w};
    const uint32_t k_lo = pack_e4m3x4(__fmul_rn(bf16_lo(kw[0]), kinv), __fmul_rn(bf16_hi(kw[0]), kinv),
                                      __fmul_rn(bf16_lo(kw[1]), kinv), __fmul_rn(bf16_hi(kw[1]), kinv));
    const uint32_t k_hi = pack_e4m3x4(__fmul_rn(bf16_lo(kw[2]), kinv), __fmul_rn(bf16_hi(kw[2]), kinv),
                                      __fmul_rn(bf16_lo(kw[3]), kinv), __fmul_rn(bf16_hi(kw[3]), kinv));
    *reinterpret_cast<uint2*>(krow + static_cast<int64_t>(row) * H * D) = make_uint2(k_lo, k_hi);
    const uint32_t v_lo = pack_e4m3x4(__fmul_rn(bf16_lo(vw[0]), vinv), __fmul_rn(bf16_hi(vw[0]), vinv),
                                      __fmul_rn(bf16_lo(vw[1]), vinv), __fmul_rn(bf16_hi(vw[1]), vinv));
    const uint32_t v_hi = pack_e4m3x4(__fmul_rn(bf16_lo(vw[2]), vinv), __fmul_rn(bf16_hi(vw[2]), vinv),
                                      __fmul_rn(bf16_lo(vw[3]), vinv), __fmul_rn(bf16_hi(vw[3]), vinv));
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      vt[8 * c + e][row] = static_cast<uint8_t>(v_lo >> (8 * e));
      vt[8 * c + 4 + e][row] = static_cast<uint8_t>(v_hi >> (8 * e));
    }
  }
  __syncthreads();
  // V^T rows: 128 d rows of 128 codes, 16 bytes per thread and step
  uint8_t* vbase = vt8 + static_cast<int64_t>(h) * D * rows_pad + t.dst_row0;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int idx = threadIdx.x + 256 * i;  // 0..1023 = d * 8 + chunk
    const int d = idx >> 3, ch = idx & 7;
    *reinterpret_cast<uint4*>(vbase + static_cast<int64_t>(d) * rows_pad + 16 * ch) =
        *reinterpret_cast<const uint4*>(&vt[d][16 * ch]);
  }
  if (threadIdx.x == 0) {
    const float sv = __fdiv_rn(vmax, 448.f);
    scales[static_cast<int64_t>(t.dst_row0 >> 7) * H + h] =
        make_float4(__fdiv_rn(kmax, 448.f), sv, sv > 0.f ? log2f(sv) : 0.f, sv > 0.f ? __frcp_rn(sv) : 0.f);
  }
}

}  // namespace rc
