// attn_tc.cuh -- the sm_103a attention kernel: TMA-staged Q/K/V tiles,
// tcgen05 MMAs accumulating in tensor memory, fp32 online softmax.
//
// Computes, for every (task, head) item, O = softmax(scale * Q K^T) V over
// the task's visible keys (key ranges A then B; see common.cuh), with the
// scores, softmax and accumulation in fp32 and P rounded to bf16 for P.V.
//
// CTA organisation (one persistent CTA per SM, 320 threads):
//   warps 0-3  softmax group 0: query tile 0 (item rows 0..127), one row per thread
//   warps 4-7  softmax group 1: query tile 1 (item rows 128..255)
//   warp 8     TMA producer: Q tiles once per item, then K_j and V_j tiles
//              of 128 keys into a ring of NS shared-memory slots
//   warp 9     MMA issuer (one thread): S_i = Q_i K_j^T, O_i += P_i V_j;
//              also allocates and frees tensor memory
// Tensor memory (512 columns x 128 lanes of 32 bit):
//   S_0 cols [0,128)   S_1 cols [128,256)   O_0 cols [256,256+D)   O_1 [384,384+D)
//   P_i (bf16, two per column) overwrites the first 64 columns of S_i once
//   the softmax has read S_i; the P.V MMA reads P_i straight from TMEM.
// Per key tile j the MMA thread issues S_0, S_1, then (after each softmax
// group has written P_i) O_0 += P_0 V_j and O_1 += P_1 V_j, so the softmax of
// one query tile overlaps the tensor-core work of the other.
// Rescaling of O is lazy: a row's running maximum is only moved (and its O
// row in TMEM multiplied down) when a new score exceeds it by more than 2^8.
//
// Shared memory: Q_0, Q_1 and NS ring slots of 128 rows x D bf16 each, every
// tile stored as D/64 TMA boxes of 128 rows x 128 bytes with the 128-byte
// swizzle (the canonical K-major layout for Q and K; V is read as the
// MN-major B operand of P.V from the same layout).
//
// Every wait is bounded (AttnArgs::timeout_ns).  A wait that runs out sets
// the device error word and a CTA-wide abort flag; every role then leaves its
// loop, the producer waits (bounded) for its TMA loads in flight, the MMA
// thread for its MMAs in flight, and tensor memory is freed before exit.
#pragma once
#include <cuda.h>
#include <cuda_bf16.h>

#include "common.cuh"
#include "ptx.cuh"

namespace rc {

namespace tc {
constexpr int kThreads = 320;
constexpr int kNumSlots = 4;
constexpr int kTileRows = 128;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kBoxBytes = 128 * 128;  // one TMA box: 128 rows x 128 bytes

template <int D>
struct Smem {
  static constexpr uint32_t kTile = kTileRows * D * 2;
  static constexpr uint32_t kQ0 = 0;
  static constexpr uint32_t kQ1 = kTile;
  static constexpr uint32_t kRing = 2 * kTile;
  static constexpr uint32_t kBars = kRing + kNumSlots * kTile;
  // barrier indices
  static constexpr int kQFull = 0, kQEmpty = 1, kSlotFull = 2, kSlotEmpty = 2 + kNumSlots,
                       kSFull = 2 + 2 * kNumSlots, kPFull = kSFull + 2, kOFull = kPFull + 2,
                       kOFree = kOFull + 2, kMmaDone = kOFree + 2, kNumBars = kMmaDone + 1;
  static constexpr uint32_t kTmemHolder = kBars + 8 * kNumBars;
  static constexpr uint32_t kAbort = kTmemHolder + 4;
  static constexpr uint32_t kUsed = kAbort + 4;
  static constexpr uint32_t kDynamic = kUsed + 1024;  // slack to align the base to 1024
};

struct Ctl {
  volatile int* abort_flag;
  uint64_t timeout_ns;
};

// Bounded wait on one mbarrier phase by one thread.
__device__ __forceinline__ bool wait_one(uint32_t bar, uint32_t parity, const Ctl& c, int where) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (;;) {
    for (int i = 0; i < 16; ++i)
      if (mbar_try_wait(bar, parity)) return true;
    if (*c.abort_flag) return false;
    if (globaltimer_ns() - t0 > c.timeout_ns) {
      *c.abort_flag = 1;
      atomicCAS(&g_rc_status, 0, RC_DEV_TIMEOUT_BASE + where);
      return false;
    }
  }
}
// Bounded wait by a whole warp; the outcome is made warp-uniform.
__device__ __forceinline__ bool wait_warp(uint32_t bar, uint32_t parity, const Ctl& c, int where) {
  const bool ok = wait_one(bar, parity, c, where);
  return __all_sync(0xffffffffu, ok);
}
// Bounded wait used during teardown: ignores the abort flag.
__device__ __forceinline__ void drain_one(uint32_t bar, uint32_t parity, uint64_t timeout_ns) {
  const uint64_t t0 = globaltimer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (globaltimer_ns() - t0 > timeout_ns) break;
  }
}

struct TileSrc {
  int row;    // first key row of the tile in its tensor
  int valid;  // keys of the tile inside the range (1..128)
  bool in_b;  // tile comes from the B tensors
};
__device__ __forceinline__ TileSrc tile_src(const Task& t, int na, int j) {
  TileSrc s;
  if (j < na) {
    s.row = t.a_row0 + j * kTileRows;
    s.valid = min(kTileRows, t.a_len - j * kTileRows);
    s.in_b = false;
  } else {
    const int jj = j - na;
    s.row = t.b_row0 + jj * kTileRows;
    s.valid = min(kTileRows, t.b_len - jj * kTileRows);
    s.in_b = true;
  }
  return s;
}
}  // namespace tc

template <int D>
__global__ void __launch_bounds__(tc::kThreads, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_ka,
                   const __grid_constant__ CUtensorMap tm_va, const __grid_constant__ CUtensorMap tm_kb,
                   const __grid_constant__ CUtensorMap tm_vb, const AttnArgs args) {
  using namespace tc;
  using L = Smem<D>;
  static_assert(D == 64 || D == 128, "head_dim 64 or 128");
  constexpr int kChunks = D / 64;
  constexpr uint32_t kIdescS = idesc_bf16_f32(128, 128, false);
  constexpr uint32_t kIdescO = idesc_bf16_f32(128, D, true);

  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* base_ptr = smem_raw + (base - raw);
  auto bar = [&](int i) -> uint32_t { return base + L::kBars + 8u * static_cast<uint32_t>(i); };
  volatile int* abort_flag = reinterpret_cast<volatile int*>(base_ptr + L::kAbort);
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(base_ptr + L::kTmemHolder);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    mbar_init(bar(L::kQFull), 1);
    mbar_init(bar(L::kQEmpty), 1);
    for (int s = 0; s < kNumSlots; ++s) {
      mbar_init(bar(L::kSlotFull + s), 1);
      mbar_init(bar(L::kSlotEmpty + s), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(bar(L::kSFull + i), 1);
      mbar_init(bar(L::kPFull + i), 128);
      mbar_init(bar(L::kOFull + i), 1);
      mbar_init(bar(L::kOFree + i), 128);
    }
    mbar_init(bar(L::kMmaDone), 1);
    *abort_flag = 0;
    fence_barrier_init();
    fence_proxy_async_smem();
  }
  if (warp == 9) {
    tmem_alloc(smem_u32(tmem_holder), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_holder;
  const Ctl ctl{abort_flag, args.timeout_ns};

  if (warp == 8) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      uint32_t use = 0, q_uses = 0;
      int armed_round[kNumSlots];
      for (int s = 0; s < kNumSlots; ++s) armed_round[s] = -1;
      int q_armed = -1;
      bool skip_next = args.dbg_skip_first_load != 0;
      for (int item = blockIdx.x; item < args.n_items; item += gridDim.x) {
        const Task t = args.tasks[item / args.num_heads];
        const int head = item % args.num_heads;
        const int na = (t.a_len + kTileRows - 1) / kTileRows;
        const int nkv = na + (t.b_len + kTileRows - 1) / kTileRows;
        if (nkv == 0) continue;
        const bool two = t.q_rows > kTileRows;
        if (!wait_one(bar(L::kQEmpty), (q_uses & 1u) ^ 1u, ctl, 1)) goto producer_done;
        mbar_arrive_expect_tx(bar(L::kQFull), (two ? 2u : 1u) * L::kTile);
        for (int c = 0; c < kChunks; ++c) {
          tma_load_2d(base + L::kQ0 + c * kBoxBytes, &tm_q, bar(L::kQFull), head * D + c * 64, t.q_row0);
          if (two)
            tma_load_2d(base + L::kQ1 + c * kBoxBytes, &tm_q, bar(L::kQFull), head * D + c * 64,
                        t.q_row0 + kTileRows);
        }
        q_armed = static_cast<int>(q_uses);
        ++q_uses;
        for (int j = 0; j < nkv; ++j) {
          const TileSrc src = tile_src(t, na, j);
          for (int kv = 0; kv < 2; ++kv, ++use) {
            const int slot = static_cast<int>(use % kNumSlots);
            const uint32_t round = use / kNumSlots;
            if (!wait_one(bar(L::kSlotEmpty + slot), (round & 1u) ^ 1u, ctl, 2)) goto producer_done;
            if (skip_next) {  // fault injection: this load never arrives
              skip_next = false;
              continue;
            }
            const void* map = kv == 0 ? (src.in_b ? &tm_kb : &tm_ka) : (src.in_b ? &tm_vb : &tm_va);
            const uint32_t dst = base + L::kRing + static_cast<uint32_t>(slot) * L::kTile;
            mbar_arrive_expect_tx(bar(L::kSlotFull + slot), L::kTile);
            for (int c = 0; c < kChunks; ++c)
              tma_load_2d(dst + c * kBoxBytes, map, bar(L::kSlotFull + slot), head * D + c * 64, src.row);
            armed_round[slot] = static_cast<int>(round);
          }
        }
      }
    producer_done:
      // Let every TMA load this CTA issued land before the CTA may exit.
      for (int s = 0; s < kNumSlots; ++s)
        if (armed_round[s] >= 0)
          drain_one(bar(L::kSlotFull + s), static_cast<uint32_t>(armed_round[s]) & 1u, args.timeout_ns);
      if (q_armed >= 0) drain_one(bar(L::kQFull), static_cast<uint32_t>(q_armed) & 1u, args.timeout_ns);
    }
    __syncwarp();
  } else if (warp == 9) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      uint32_t use = 0, q_uses = 0;
      uint32_t p_cnt[2] = {0u, 0u}, ofree_cnt[2] = {0u, 0u};
      bool ofree_pending[2] = {false, false};
      bool issued_any = false;
      for (int item = blockIdx.x; item < args.n_items; item += gridDim.x) {
        const Task t = args.tasks[item / args.num_heads];
        const int na = (t.a_len + kTileRows - 1) / kTileRows;
        const int nkv = na + (t.b_len + kTileRows - 1) / kTileRows;
        if (nkv == 0) continue;
        const int ntiles = t.q_rows > kTileRows ? 2 : 1;
        if (!wait_one(bar(L::kQFull), q_uses & 1u, ctl, 3)) goto mma_done;
        ++q_uses;
        tc_fence_after();
        for (int j = 0; j < nkv; ++j) {
          const int kslot = static_cast<int>(use % kNumSlots);
          const uint32_t kround = use / kNumSlots;
          ++use;
          const int vslot = static_cast<int>(use % kNumSlots);
          const uint32_t vround = use / kNumSlots;
          ++use;
          if (!wait_one(bar(L::kSlotFull + kslot), kround & 1u, ctl, 4)) goto mma_done;
          tc_fence_after();
          const uint32_t kaddr = base + L::kRing + static_cast<uint32_t>(kslot) * L::kTile;
          for (int i = 0; i < ntiles; ++i) {
            const uint32_t qaddr = base + (i == 0 ? L::kQ0 : L::kQ1);
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk) {
              const uint32_t off = static_cast<uint32_t>(kk / 4) * kBoxBytes + static_cast<uint32_t>(kk % 4) * 32u;
              tc_mma_ss(tmem + 128u * i, sdesc_sw128(qaddr + off, 16, 1024), sdesc_sw128(kaddr + off, 16, 1024),
                        kIdescS, kk > 0 ? 1u : 0u);
            }
            tc_commit(bar(L::kSFull + i));
          }
          issued_any = true;
          tc_commit(bar(L::kSlotEmpty + kslot));
          if (j == nkv - 1) tc_commit(bar(L::kQEmpty));
          if (!wait_one(bar(L::kSlotFull + vslot), vround & 1u, ctl, 5)) goto mma_done;
          const uint32_t vaddr = base + L::kRing + static_cast<uint32_t>(vslot) * L::kTile;
          for (int i = 0; i < ntiles; ++i) {
            if (j == 0 && ofree_pending[i]) {
              if (!wait_one(bar(L::kOFree + i), ofree_cnt[i] & 1u, ctl, 6)) goto mma_done;
              ++ofree_cnt[i];
              ofree_pending[i] = false;
            }
            if (!wait_one(bar(L::kPFull + i), p_cnt[i] & 1u, ctl, 7)) goto mma_done;
            ++p_cnt[i];
            tc_fence_after();
#pragma unroll
            for (int kk = 0; kk < kTileRows / 16; ++kk) {
              tc_mma_ts(tmem + 256u + 128u * i, tmem + 128u * i + 8u * kk,
                        sdesc_sw128(vaddr + 2048u * kk, kBoxBytes, 1024), kIdescO,
                        (j > 0 || kk > 0) ? 1u : 0u);
            }
            tc_commit(bar(L::kOFull + i));
          }
          tc_commit(bar(L::kSlotEmpty + vslot));
        }
        for (int i = 0; i < ntiles; ++i) ofree_pending[i] = true;
      }
    mma_done:
      if (issued_any) {  // every MMA issued must finish before TMEM is freed
        tc_commit(bar(L::kMmaDone));
        drain_one(bar(L::kMmaDone), 0u, args.timeout_ns);
      }
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ softmax groups
    const int grp = warp >> 2;               // query tile of this group
    const int trow = threadIdx.x & 127;      // row within the tile (= TMEM lane)
    const uint32_t lane_off = static_cast<uint32_t>((warp & 3) * 32) << 16;
    const uint32_t t_s = tmem + lane_off + 128u * grp;
    const uint32_t t_o = tmem + lane_off + 256u + 128u * grp;
    const float sl2 = args.scale_log2;
    uint32_t s_cnt = 0, o_cnt = 0;
    for (int item = blockIdx.x; item < args.n_items; item += gridDim.x) {
      const Task t = args.tasks[item / args.num_heads];
      const int head = item % args.num_heads;
      if (grp == 1 && t.q_rows <= kTileRows) continue;
      const int na = (t.a_len + kTileRows - 1) / kTileRows;
      const int nkv = na + (t.b_len + kTileRows - 1) / kTileRows;
      const int row = grp * kTileRows + trow;
      const bool row_ok = row < t.q_rows;
      const int64_t grow = static_cast<int64_t>(t.q_row0) + row;
      __nv_bfloat16* orow = args.out + grow * args.row_stride + static_cast<int64_t>(head) * D;
      if (nkv == 0) {
        if (row_ok) {
          uint4 z = make_uint4(0, 0, 0, 0);
          for (int c = 0; c < D / 8; ++c) reinterpret_cast<uint4*>(orow)[c] = z;
          if (args.lse) args.lse[grow * args.num_heads + head] = -INFINITY;
        }
        continue;
      }
      float m_run = 0.f, l_run = 0.f;
      for (int j = 0; j < nkv; ++j) {
        const TileSrc src = tile_src(t, na, j);
        if (!wait_warp(bar(L::kSFull + grp), s_cnt & 1u, ctl, 8)) goto softmax_done;
        ++s_cnt;
        tc_fence_after();
        uint32_t r0[32], r1[32], r2[32], r3[32];
        tmem_ld32(t_s + 0u, r0);
        tmem_ld32(t_s + 32u, r1);
        tmem_ld32(t_s + 64u, r2);
        tmem_ld32(t_s + 96u, r3);
        tmem_wait_ld(r0);
        tmem_wait_ld(r1);
        tmem_wait_ld(r2);
        tmem_wait_ld(r3);
        float s[128];
#pragma unroll
        for (int c = 0; c < 32; ++c) {
          s[c] = __uint_as_float(r0[c]);
          s[32 + c] = __uint_as_float(r1[c]);
          s[64 + c] = __uint_as_float(r2[c]);
          s[96 + c] = __uint_as_float(r3[c]);
        }
        if (src.valid < kTileRows) {
#pragma unroll
          for (int c = 0; c < 128; ++c)
            if (c >= src.valid) s[c] = -INFINITY;
        }
        float mx0 = s[0], mx1 = s[1], mx2 = s[2], mx3 = s[3];
#pragma unroll
        for (int c = 4; c < 128; c += 4) {
          mx0 = fmaxf(mx0, s[c]);
          mx1 = fmaxf(mx1, s[c + 1]);
          mx2 = fmaxf(mx2, s[c + 2]);
          mx3 = fmaxf(mx3, s[c + 3]);
        }
        const float m_tile = fmaxf(fmaxf(mx0, mx1), fmaxf(mx2, mx3)) * sl2;
        if (j > 0) {
          // O_i holds P_{j-1} V_{j-1} once S_i of tile j is complete; this
          // wait keeps the phase count in step and returns at once.
          if (!wait_warp(bar(L::kOFull + grp), o_cnt & 1u, ctl, 9)) goto softmax_done;
          ++o_cnt;
          tc_fence_after();
          const bool need = m_tile > m_run + 8.0f;
          if (__any_sync(0xffffffffu, need)) {
            const float m_new = fmaxf(m_run, m_tile);
            const float alpha = ex2_approx(m_run - m_new);
            m_run = m_new;
            l_run *= alpha;
#pragma unroll
            for (int cc = 0; cc < D / 16; ++cc) {
              uint32_t o[16];
              tmem_ld16(t_o + 16u * cc, o);
              tmem_wait_ld(o);
#pragma unroll
              for (int c = 0; c < 16; ++c) o[c] = __float_as_uint(__uint_as_float(o[c]) * alpha);
              tmem_st16(t_o + 16u * cc, o);
            }
          }
        } else {
          m_run = m_tile;
        }
        // P = exp2(scaled S - m) as bf16 pairs, written 16 score columns
        // (8 TMEM columns) at a time over the S columns already consumed.
        const float neg_m = -m_run;
        float ls0 = 0.f, ls1 = 0.f;
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          uint32_t pk[8];
#pragma unroll
          for (int c = 0; c < 8; ++c) {
            const float a = ex2_approx(fmaf(s[16 * q + 2 * c], sl2, neg_m));
            const float b = ex2_approx(fmaf(s[16 * q + 2 * c + 1], sl2, neg_m));
            ls0 += a;
            ls1 += b;
            pk[c] = pack_bf16x2(a, b);
          }
          tmem_st8(t_s + 8u * q, pk);
        }
        l_run += ls0 + ls1;
        tmem_wait_st();
        tc_fence_before();
        mbar_arrive(bar(L::kPFull + grp));
      }
      // epilogue: O_i / l -> bf16 rows
      if (!wait_warp(bar(L::kOFull + grp), o_cnt & 1u, ctl, 10)) goto softmax_done;
      ++o_cnt;
      tc_fence_after();
      {
        const float inv_l = 1.0f / l_run;
        uint32_t packed[D / 2];
#pragma unroll
        for (int cc = 0; cc < D / 32; ++cc) {
          uint32_t o[32];
          tmem_ld32(t_o + 32u * cc, o);
          tmem_wait_ld(o);
#pragma unroll
          for (int c = 0; c < 16; ++c)
            packed[16 * cc + c] =
                pack_bf16x2(__uint_as_float(o[2 * c]) * inv_l, __uint_as_float(o[2 * c + 1]) * inv_l);
        }
        tc_fence_before();
        mbar_arrive(bar(L::kOFree + grp));
        if (row_ok) {
          uint4* dst = reinterpret_cast<uint4*>(orow);
#pragma unroll
          for (int c = 0; c < D / 8; ++c)
            dst[c] = make_uint4(packed[4 * c], packed[4 * c + 1], packed[4 * c + 2], packed[4 * c + 3]);
          if (args.lse)
            args.lse[grow * args.num_heads + head] = (m_run + log2f(l_run)) * 0.69314718055994530942f;
        }
      }
    }
  softmax_done:;
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 9) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

}  // namespace rc
