// attn_mma.cuh -- the same masked attention on the legacy warp-level tensor
// core path (mma.sync.m16n8k16 bf16, ldmatrix, cp.async), kept as the
// "recompiled pre-Blackwell kernel" comparison point for the tcgen05 kernel.
//
// CTA = 4 warps = 64 query rows (16 per warp) of one (task, head) item;
// blockIdx.x = (rows_per_task / 64) * item + sub, sub selecting rows
// [64 sub, 64 sub + 64) of the task.  Key tiles of 64 rows stream through a double-buffered cp.async
// pipeline (range A, then range B); scores, online softmax (exact running
// maximum, fp32) and the P.V accumulation stay in registers.
#pragma once
#include <cuda_bf16.h>

#include "common.cuh"
#include "ptx.cuh"

namespace rc {

namespace mm {
__device__ __forceinline__ void cp_async16(void* smem, const void* gmem, int src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(static_cast<uint32_t>(
                   __cvta_generic_to_shared(smem))),
               "l"(gmem), "r"(src_bytes)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}
__device__ __forceinline__ void ldsm_x4(uint32_t (&r)[4], const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(static_cast<uint32_t>(__cvta_generic_to_shared(p))));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t (&r)[4], const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(static_cast<uint32_t>(__cvta_generic_to_shared(p))));
}
__device__ __forceinline__ void mma16816(float (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ uint32_t pack2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}
__device__ __forceinline__ float ex2f(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
}  // namespace mm

template <int D>
__global__ void __launch_bounds__(128) attn_mma_kernel(const AttnArgs a) {
  using namespace mm;
  constexpr int kCh = D / 8;  // 16-byte chunks per row
  extern __shared__ __align__(128) uint8_t smem_mm[];
  __nv_bfloat16* sQ = reinterpret_cast<__nv_bfloat16*>(smem_mm);
  __nv_bfloat16* sK = sQ + 64 * D;
  __nv_bfloat16* sV = sK + 2 * 64 * D;
  // element offset of (row, 16-byte chunk) with the chunk XOR-swizzled by row
  auto off = [](int row, int ch) { return row * D + ((ch ^ (row & 7)) << 3); };

  const int per_task = a.rows_per_task / 64;
  const int item = blockIdx.x / per_task, sub = blockIdx.x % per_task;
  if (item >= a.n_items) return;
  const Task t = a.tasks[item / a.num_heads];
  const int head = item % a.num_heads;
  const int r0 = sub * 64;
  if (r0 >= t.q_rows) return;
  const int nrows = min(64, t.q_rows - r0);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t ld = a.row_stride;
  const int na = (t.a_len + 63) / 64, nkv = na + (t.b_len + 63) / 64;

  const int g = lane >> 2, q4 = lane & 3;
  if (nkv == 0) {
    for (int h = 0; h < 2; ++h) {
      const int row = 16 * warp + g + 8 * h;
      if (row < nrows) {
        const int64_t grow = t.q_row0 + r0 + row;
        for (int c = q4; c < D / 2; c += 4)
          reinterpret_cast<uint32_t*>(a.out + grow * ld + head * D)[c] = 0u;
        if (a.lse && q4 == 0) a.lse[grow * a.num_heads + head] = -INFINITY;
      }
    }
    return;
  }

  auto load_rows = [&](__nv_bfloat16* dst, const __nv_bfloat16* src, int row0, int valid) {
    for (int i = threadIdx.x; i < 64 * kCh; i += 128) {
      const int r = i / kCh, ch = i % kCh;
      const int rr = r < valid ? r : 0;
      cp_async16(dst + off(r, ch), src + (row0 + rr) * ld + head * D + ch * 8, r < valid ? 16 : 0);
    }
  };
  auto load_tile = [&](int j, int buf) {
    int row0, valid;
    const __nv_bfloat16 *k, *v;
    if (j < na) {
      row0 = t.a_row0 + 64 * j;
      valid = min(64, t.a_len - 64 * j);
      k = a.ka;
      v = a.va;
    } else {
      row0 = t.b_row0 + 64 * (j - na);
      valid = min(64, t.b_len - 64 * (j - na));
      k = a.kb;
      v = a.vb;
    }
    load_rows(sK + buf * 64 * D, k, row0, valid);
    load_rows(sV + buf * 64 * D, v, row0, valid);
  };
  auto tile_valid = [&](int j) {
    return j < na ? min(64, t.a_len - 64 * j) : min(64, t.b_len - 64 * (j - na));
  };

  load_rows(sQ, a.q, t.q_row0 + r0, nrows);
  load_tile(0, 0);
  cp_async_commit();

  uint32_t qf[D / 16][4];
  float oacc[D / 8][4];
#pragma unroll
  for (int i = 0; i < D / 8; ++i) oacc[i][0] = oacc[i][1] = oacc[i][2] = oacc[i][3] = 0.f;
  float m[2] = {-INFINITY, -INFINITY}, l[2] = {0.f, 0.f};
  const float sl2 = a.scale_log2;
  const int mi = lane >> 3, li = lane & 7;

  for (int j = 0; j < nkv; ++j) {
    const int buf = j & 1;
    if (j + 1 < nkv) {
      load_tile(j + 1, buf ^ 1);
      cp_async_commit();
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    if (j == 0) {
#pragma unroll
      for (int kt = 0; kt < D / 16; ++kt)
        ldsm_x4(qf[kt], sQ + off(16 * warp + (mi & 1) * 8 + li, 2 * kt + (mi >> 1)));
    }
    const __nv_bfloat16* K = sK + buf * 64 * D;
    const __nv_bfloat16* V = sV + buf * 64 * D;
    float s[8][4];
#pragma unroll
    for (int n = 0; n < 8; ++n) s[n][0] = s[n][1] = s[n][2] = s[n][3] = 0.f;
#pragma unroll
    for (int kt = 0; kt < D / 16; ++kt) {
#pragma unroll
      for (int np = 0; np < 4; ++np) {
        uint32_t b[4];
        ldsm_x4(b, K + off(16 * np + (mi >> 1) * 8 + li, 2 * kt + (mi & 1)));
        mma16816(s[2 * np], qf[kt], b[0], b[1]);
        mma16816(s[2 * np + 1], qf[kt], b[2], b[3]);
      }
    }
    const int valid = tile_valid(j);
    if (valid < 64) {
#pragma unroll
      for (int n = 0; n < 8; ++n)
#pragma unroll
        for (int e = 0; e < 4; ++e)
          if (8 * n + 2 * q4 + (e & 1) >= valid) s[n][e] = -INFINITY;
    }
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      float mx = -INFINITY;
#pragma unroll
      for (int n = 0; n < 8; ++n) mx = fmaxf(mx, fmaxf(s[n][2 * h], s[n][2 * h + 1]));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
      const float m_new = fmaxf(m[h], mx * sl2);
      const float alpha = ex2f(m[h] - m_new);
      m[h] = m_new;
      float rs = 0.f;
#pragma unroll
      for (int n = 0; n < 8; ++n) {
        s[n][2 * h] = ex2f(fmaf(s[n][2 * h], sl2, -m_new));
        s[n][2 * h + 1] = ex2f(fmaf(s[n][2 * h + 1], sl2, -m_new));
        rs += s[n][2 * h] + s[n][2 * h + 1];
      }
      l[h] = l[h] * alpha + rs;
#pragma unroll
      for (int dn = 0; dn < D / 8; ++dn) {
        oacc[dn][2 * h] *= alpha;
        oacc[dn][2 * h + 1] *= alpha;
      }
    }
#pragma unroll
    for (int kt = 0; kt < 4; ++kt) {
      uint32_t pa[4] = {pack2(s[2 * kt][0], s[2 * kt][1]), pack2(s[2 * kt][2], s[2 * kt][3]),
                        pack2(s[2 * kt + 1][0], s[2 * kt + 1][1]), pack2(s[2 * kt + 1][2], s[2 * kt + 1][3])};
#pragma unroll
      for (int dp = 0; dp < D / 16; ++dp) {
        uint32_t b[4];
        ldsm_x4_t(b, V + off(16 * kt + (mi & 1) * 8 + li, 2 * dp + (mi >> 1)));
        mma16816(oacc[2 * dp], pa, b[0], b[1]);
        mma16816(oacc[2 * dp + 1], pa, b[2], b[3]);
      }
    }
    __syncthreads();
  }
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    float lt = l[h];
    lt += __shfl_xor_sync(0xffffffffu, lt, 1);
    lt += __shfl_xor_sync(0xffffffffu, lt, 2);
    const int row = 16 * warp + g + 8 * h;
    if (row < nrows) {
      const float inv = 1.f / lt;
      const int64_t grow = t.q_row0 + r0 + row;
      uint32_t* dst = reinterpret_cast<uint32_t*>(a.out + grow * ld + head * D);
#pragma unroll
      for (int dn = 0; dn < D / 8; ++dn)
        dst[4 * dn + q4] = pack2(oacc[dn][2 * h] * inv, oacc[dn][2 * h + 1] * inv);
      if (a.lse && q4 == 0) a.lse[grow * a.num_heads + head] = (m[h] + log2f(lt)) * 0.69314718055994530942f;
    }
  }
}

// Cache write (the copy of the static pass's R rows' K and V into the
// persistent slot of one layer).  One block row per request segment.  It reads
// only the static inputs, so it may run beside the prefill attention: launched
// as a programmatic dependent of that kernel it starts once the prefill's CTAs
// are all running (and so the inputs' producers are complete), and it waits
// for the prefill to complete before it exits, so that the work after it on
// the stream sees both.
struct CopySeg {
  int32_t src_row0, dst_row0, nrows, pad;
};
__global__ void copy_rows_kernel(const CopySeg* segs, const uint4* __restrict__ src_k,
                                 const uint4* __restrict__ src_v, uint4* __restrict__ dst_k,
                                 uint4* __restrict__ dst_v, int row_u4) {
  if (threadIdx.x == 0) grid_launch_dependents();
  const CopySeg s = segs[blockIdx.y];
  const int64_t n = static_cast<int64_t>(s.nrows) * row_u4;
  const int64_t so = static_cast<int64_t>(s.src_row0) * row_u4, d0 = static_cast<int64_t>(s.dst_row0) * row_u4;
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    dst_k[d0 + i] = src_k[so + i];
    dst_v[d0 + i] = src_v[so + i];
  }
  grid_dependency_wait();
}

}  // namespace rc
