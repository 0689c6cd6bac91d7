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

// grid (H, tiles, 2): blockIdx.z = 0 quantises the tile's K, 1 its V (heads
// fastest, so that CTAs running together read neighbouring bytes of the same
// rows); 256 threads.  Thread i takes rows [4 q, 4 q + 4) of the tile (q = i % 32) and
// head-dim columns [16 p, 16 p + 16) (p = i / 32): per row one 32-byte run.
// K codes go out row by row (16 bytes); V codes are transposed through shared
// memory as one 32-bit word (four rows) per column, so the 32 threads of a
// warp store 32 consecutive words.
__global__ void __launch_bounds__(256, 3) quantize_cache_kernel(const QuantTile* __restrict__ tiles,
                                                                const uint4* __restrict__ k, const uint4* __restrict__ v,
                                                                uint8_t* __restrict__ k8, uint8_t* __restrict__ vt8,
                                                                float4* __restrict__ scales, int H, int64_t rows_pad) {
  constexpr int D = 128;
  __shared__ float red[8];
  __shared__ __align__(16) uint32_t vt[D][32 + 4];  // V^T codes of the tile: [d][row / 4], 4 rows per word
  const QuantTile t = tiles[blockIdx.y];
  const int h = blockIdx.x;
  const bool is_v = blockIdx.z != 0;
  const int q = threadIdx.x & 31;   // rows 4 q .. 4 q + 3
  const int p = threadIdx.x >> 5;   // columns 16 p .. 16 p + 15
  const int64_t row_u4 = static_cast<int64_t>(H) * D / 8;
  const uint4* src = is_v ? v : k;
  uint4 x[4][2];
  float a = 0.f;
#pragma unroll
  for (int r = 0; r < 4; ++r) {
    const int row = 4 * q + r;
#pragma unroll
    for (int c = 0; c < 2; ++c) {
      x[r][c] = row < t.valid ? src[static_cast<int64_t>(t.src_row0 + row) * row_u4 + h * (D / 8) + 2 * p + c]
                              : make_uint4(0, 0, 0, 0);
      const uint32_t w[4] = {x[r][c].x, x[r][c].y, x[r][c].z, x[r][c].w};
#pragma unroll
      for (int e = 0; e < 4; ++e) a = fmax3(a, fabsf(bf16_lo(w[e])), fabsf(bf16_hi(w[e])));
    }
  }
  const float amax = block_amax_256(a, red);
  const float inv = amax > 0.f ? __fdiv_rn(448.f, amax) : 0.f;
  // codes of the 16 columns of row r: four words of four codes
  uint32_t cw[4][4];
#pragma unroll
  for (int r = 0; r < 4; ++r)
#pragma unroll
    for (int c = 0; c < 2; ++c) {
      const uint4& y = x[r][c];
      cw[r][2 * c] = pack_e4m3x4(__fmul_rn(bf16_lo(y.x), inv), __fmul_rn(bf16_hi(y.x), inv),
                                 __fmul_rn(bf16_lo(y.y), inv), __fmul_rn(bf16_hi(y.y), inv));
      cw[r][2 * c + 1] = pack_e4m3x4(__fmul_rn(bf16_lo(y.z), inv), __fmul_rn(bf16_hi(y.z), inv),
                                     __fmul_rn(bf16_lo(y.w), inv), __fmul_rn(bf16_hi(y.w), inv));
    }
  if (!is_v) {
    uint8_t* krow = k8 + static_cast<int64_t>(t.dst_row0) * H * D + static_cast<int64_t>(h) * D + 16 * p;
#pragma unroll
    for (int r = 0; r < 4; ++r)
      *reinterpret_cast<uint4*>(krow + static_cast<int64_t>(4 * q + r) * H * D) =
          make_uint4(cw[r][0], cw[r][1], cw[r][2], cw[r][3]);
    if (threadIdx.x == 0) scales[static_cast<int64_t>(t.dst_row0 >> 7) * H + h].x = __fdiv_rn(amax, 448.f);
    return;
  }
  // column 16 p + 4 w + e: byte e of word w of each of the four rows
#pragma unroll
  for (int w = 0; w < 4; ++w)
#pragma unroll
    for (int e = 0; e < 4; ++e)
      vt[16 * p + 4 * w + e][q] = __byte_perm(__byte_perm(cw[0][w], cw[1][w], 0x0040 + e * 0x0011),
                                              __byte_perm(cw[2][w], cw[3][w], 0x0040 + e * 0x0011), 0x5410);
  __syncthreads();
  // V^T rows: 128 d rows of 128 codes, 16 bytes per thread and step
  uint8_t* vbase = vt8 + static_cast<int64_t>(h) * D * rows_pad + t.dst_row0;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int idx = threadIdx.x + 256 * i;  // 0..1023 = d * 8 + chunk
    const int d = idx >> 3, ch = idx & 7;
    *reinterpret_cast<uint4*>(vbase + static_cast<int64_t>(d) * rows_pad + 16 * ch) =
        *reinterpret_cast<const uint4*>(&vt[d][4 * ch]);
  }
  if (threadIdx.x == 0) {
    const float sv = __fdiv_rn(amax, 448.f);
    float4* dst = &scales[static_cast<int64_t>(t.dst_row0 >> 7) * H + h];
    dst->y = sv;
    dst->z = sv > 0.f ? log2f(sv) : 0.f;
    dst->w = sv > 0.f ? __frcp_rn(sv) : 0.f;
  }
}

}  // namespace rc
