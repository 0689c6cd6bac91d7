// attn_tc.cuh -- the sm_103a attention kernel: TMA-staged Q/K/V tiles,
// tcgen05 MMAs accumulating in tensor memory, fp32 online softmax.
//
// Computes, for every (task, head) item, O = softmax(scale * Q K^T) V over
// the task's visible keys (key ranges A then B; see common.cuh), with the
// scores, softmax and accumulation in fp32 and P rounded to bf16 for P.V.
//
// CTA organisation (one persistent CTA per SM, 320 threads):
//   warps 0-7  softmax: row r of the item's 128-row query tile is shared by
//              thread r of warps 0-3 (score columns 0-63) and thread r of
//              warps 4-7 (columns 64-127); the two exchange their partial
//              row maxima through shared memory once per tile
//   warp 8     TMA producer: the item's Q tile, then K and V tiles of 128
//              keys into a ring of kNumSlots shared-memory slots
//   warp 9     MMA issuer (one thread); also allocates and frees TMEM
//
// The key tiles of all items a CTA runs form one stream t = 0, 1, 2, ...
// For tile t the MMA thread computes S_t = Q K_t^T and O += P_t V_t.  The
// MMAs are issued in pairs: pair t interleaves, instruction by instruction,
// the 8 MMAs of O += P_t V_t with the MMAs of S_{t+2} = Q K_{t+2}^T (the
// latter may belong to the next item).  The tensor core then runs a stream
// that alternates the two instruction kinds at every MMA, which keeps it at
// full rate, whereas long runs of one kind followed by the other drain its
// pipeline at every switch.  While pair t runs, the softmax turns S_{t+1}
// into P_{t+1}, so the softmax of one tile overlaps the MMAs of the others.
//
// Tensor memory (512 columns x 128 lanes of 32 bit):
//   S buffers  [0,128) [128,256)   tile t uses buffer t % 2 (fp32 scores)
//   P buffers  [256,320) [320,384) tile t uses buffer t % 2 (bf16 pairs,
//              read by the P.V MMA as its A operand)
//   O          [384, 384 + D)      fp32 accumulator of the current item
// Rescaling of O is lazy: a row's running maximum is only moved (and its O
// row multiplied down) when a new score exceeds it by more than 2^8.
//
// Shared memory: two Q tile buffers (item i uses buffer i % 2) and a ring of
// kNumSlots tiles of 128 rows x D bf16; every tile is D/64 TMA boxes of 128
// rows x 128 bytes with the 128-byte swizzle (the canonical K-major layout
// for Q and K; V is read as the MN-major B operand of P.V).
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
constexpr int kSoftmaxThreads = 256;
constexpr int kNumSlots = 5;
constexpr int kTileRows = 128;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kBoxBytes = 128 * 128;  // one TMA box: 128 rows x 128 bytes
constexpr uint32_t kColS = 0, kColP = 256, kColO = 384;

template <int D>
struct Smem {
  static constexpr uint32_t kTile = kTileRows * D * 2;
  static constexpr uint32_t kQ = 0;  // Q buffers 0 and 1
  static constexpr uint32_t kRing = 2 * kTile;
  static constexpr uint32_t kBars = kRing + kNumSlots * kTile;
  // barrier indices
  static constexpr int kQFull = 0, kQEmpty = 2, kSlotFull = 4, kSlotEmpty = 4 + kNumSlots,
                       kSFull = 4 + 2 * kNumSlots, kPFull = kSFull + 2, kOFree = kPFull + 2, kMmaDone = kOFree + 1,
                       kXchg = kMmaDone + 1, kNumBars = kXchg + 4;
  // partial row maxima / sums exchanged by the two threads of a row:
  // float [2 parity][2 halves][128 rows]
  static constexpr uint32_t kXBuf = kBars + 8 * kNumBars;
  static constexpr uint32_t kTmemHolder = kXBuf + 2 * 2 * 128 * 4;
  static constexpr uint32_t kAbort = kTmemHolder + 4;
  static constexpr uint32_t kUsed = kAbort + 4;
  // bytes requested at launch: slack to align the base to 1024, capped at the
  // 227 KB a CTA may have (the kernel checks that the aligned layout fits)
  static constexpr uint32_t kMaxDynamic = 232448;
  static constexpr uint32_t kDynamic = kUsed + 1024 < kMaxDynamic ? kUsed + 1024 : kMaxDynamic;
  static_assert(kUsed <= kMaxDynamic, "shared-memory layout too large");
};

struct Ctl {
  volatile int* abort_flag;
  uint64_t timeout_ns;
  int* status;  // the launching cache's own error word, or null
};

// A bounded wait ran out at `where`: the device word, and the cache's own.
__device__ __forceinline__ void report_timeout(int* status, int where) {
  atomicCAS(&g_rc_status, 0, RC_DEV_TIMEOUT_BASE + where);
  if (status) atomicCAS(status, 0, RC_DEV_TIMEOUT_BASE + where);
}

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
      report_timeout(c.status, where);
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

// Items are enumerated head-major (item = head * n_tasks + task, tasks
// longest first): CTAs that run at the same time then work on few heads, so
// the K/V tiles they all stream stay in L2.  A per-item list is already in
// that order and names the head of every item.
__device__ __forceinline__ void decode_item(const AttnArgs& a, int item, Task& t, int& head) {
  if (a.per_item) {
    t = a.tasks[item];
    head = t.head;
    return;
  }
  head = item / a.n_tasks;
  t = a.tasks[item - head * a.n_tasks];
}

__device__ __forceinline__ int n_key_tiles(const Task& t, int& na) {
  na = (t.a_len + kTileRows - 1) / kTileRows;
  return na + (t.b_len + kTileRows - 1) / kTileRows;
}

// Position in a CTA's key-tile stream: items first, first + stride, ...
// with at least one key tile; qi counts those items, t the tiles.
struct Cursor {
  Task task;
  int head, item, stride, qi, j, na, nkv, t;
  bool valid;
  __device__ __forceinline__ void seek(const AttnArgs& a) {
    for (; item < a.n_items; item += stride) {
      decode_item(a, item, task, head);
      nkv = n_key_tiles(task, na);
      if (nkv > 0) {
        j = 0;
        valid = true;
        return;
      }
    }
    valid = false;
  }
  __device__ __forceinline__ void init(const AttnArgs& a, int first, int step) {
    item = first;
    stride = step;
    qi = 0;
    t = 0;
    seek(a);
  }
  __device__ __forceinline__ bool last_of_item() const { return j == nkv - 1; }
  __device__ __forceinline__ void advance(const AttnArgs& a) {
    ++t;
    if (++j == nkv) {
      item += stride;
      ++qi;
      seek(a);
    }
  }
};
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
  if (base - raw + L::kUsed > L::kDynamic) {  // the allocation cannot hold the aligned layout
    if (threadIdx.x == 0) report_timeout(args.status, 99);
    return;
  }

  if (threadIdx.x == 0) {
    for (int i = 0; i < 2; ++i) {
      mbar_init(bar(L::kQFull + i), 1);
      mbar_init(bar(L::kQEmpty + i), 1);
      mbar_init(bar(L::kSFull + i), 1);
      mbar_init(bar(L::kPFull + i), kSoftmaxThreads);
    }
    for (int s = 0; s < kNumSlots; ++s) {
      mbar_init(bar(L::kSlotFull + s), 1);
      mbar_init(bar(L::kSlotEmpty + s), 1);
    }
    mbar_init(bar(L::kOFree), kSoftmaxThreads);
    for (int q = 0; q < 4; ++q) mbar_init(bar(L::kXchg + q), 64);  // warps q and q + 4
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
  const Ctl ctl{abort_flag, args.timeout_ns, args.status};

  if (warp == 8) {
    // ------------------------------------------------------------ producer
    // Ring order = the MMA thread's order of use: K_0, K_1, then V_t, K_t+2
    // for t = 0, 1, ...; an item's Q tile goes out just before its first K.
    if (lane == 0) {
      uint32_t use = 0;
      int armed_round[kNumSlots];
      for (int s = 0; s < kNumSlots; ++s) armed_round[s] = -1;
      int q_armed[2] = {-1, -1};
      bool skip_next = args.dbg_skip_first_load != 0;
      Cursor kc, vc;
      kc.init(args, blockIdx.x, gridDim.x);
      vc.init(args, blockIdx.x, gridDim.x);
      // load K (kv = 0) or V (kv = 1) of the tile at cursor c into the next ring slot
      auto load_tile = [&](const Cursor& c, int kv) -> bool {
        const int slot = static_cast<int>(use % kNumSlots);
        const uint32_t round = use / kNumSlots;
        ++use;
        if (!wait_one(bar(L::kSlotEmpty + slot), (round & 1u) ^ 1u, ctl, 2)) return false;
        if (kv == 0 && skip_next) {  // fault injection: this load never arrives
          skip_next = false;
          return true;
        }
        const TileSrc src = tile_src(c.task, c.na, c.j);
        const void* map = kv == 0 ? (src.in_b ? &tm_kb : &tm_ka) : (src.in_b ? &tm_vb : &tm_va);
        const uint32_t dst = base + L::kRing + static_cast<uint32_t>(slot) * L::kTile;
        mbar_arrive_expect_tx(bar(L::kSlotFull + slot), L::kTile);
        for (int ch = 0; ch < kChunks; ++ch)
          tma_load_2d(dst + ch * kBoxBytes, map, bar(L::kSlotFull + slot), c.head * D + ch * 64, src.row);
        armed_round[slot] = static_cast<int>(round);
        return true;
      };
      auto load_k = [&]() -> bool {
        if (kc.j == 0) {  // the item's Q tile into buffer qi % 2
          const int b = kc.qi & 1;
          const uint32_t u = static_cast<uint32_t>(kc.qi >> 1);
          if (!wait_one(bar(L::kQEmpty + b), (u & 1u) ^ 1u, ctl, 1)) return false;
          mbar_arrive_expect_tx(bar(L::kQFull + b), L::kTile);
          for (int ch = 0; ch < kChunks; ++ch)
            tma_load_2d(base + L::kQ + b * L::kTile + ch * kBoxBytes, &tm_q, bar(L::kQFull + b),
                        kc.head * D + ch * 64, kc.task.q_row0);
          q_armed[b] = static_cast<int>(u);
        }
        if (!load_tile(kc, 0)) return false;
        kc.advance(args);
        return true;
      };
      for (int n = 0; n < 2 && kc.valid; ++n)
        if (!load_k()) goto producer_done;
      while (vc.valid) {
        if (!load_tile(vc, 1)) goto producer_done;
        vc.advance(args);
        if (kc.valid && !load_k()) goto producer_done;
      }
    producer_done:
      // Let every TMA load this CTA issued land before the CTA may exit.
      for (int s = 0; s < kNumSlots; ++s)
        if (armed_round[s] >= 0)
          drain_one(bar(L::kSlotFull + s), static_cast<uint32_t>(armed_round[s]) & 1u, args.timeout_ns);
      for (int b = 0; b < 2; ++b)
        if (q_armed[b] >= 0) drain_one(bar(L::kQFull + b), static_cast<uint32_t>(q_armed[b]) & 1u, args.timeout_ns);
    }
    __syncwarp();
  } else if (warp == 9) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      uint32_t use = 0;
      bool issued_any = false;
      Cursor sc, pc;  // S side (two tiles ahead) and P.V side of the stream
      sc.init(args, blockIdx.x, gridDim.x);
      pc.init(args, blockIdx.x, gridDim.x);
      const uint64_t qdesc0 = sdesc_sw128(base + L::kQ, 16, 1024);
      // wait for the next ring slot to be full; returns its index or -1
      auto next_slot = [&](int where) -> int {
        const int slot = static_cast<int>(use % kNumSlots);
        const uint32_t round = use / kNumSlots;
        ++use;
        return wait_one(bar(L::kSlotFull + slot), round & 1u, ctl, where) ? slot : -1;
      };
      // the first S of an item waits for the item's Q tile
      auto wait_q = [&](const Cursor& c) -> bool {
        if (c.j != 0) return true;
        return wait_one(bar(L::kQFull + (c.qi & 1)), static_cast<uint32_t>(c.qi >> 1) & 1u, ctl, 3);
      };
      // prologue: S_0 and S_1 on their own
      for (int n = 0; n < 2 && sc.valid; ++n) {
        if (!wait_q(sc)) goto mma_done;
        const int ks = next_slot(4);
        if (ks < 0) goto mma_done;
        tc_fence_after();
        const uint64_t qd = qdesc0 + ((static_cast<uint32_t>(sc.qi & 1) * L::kTile) >> 4);
        const uint64_t kd = sdesc_sw128(base + L::kRing + static_cast<uint32_t>(ks) * L::kTile, 16, 1024);
        const uint32_t d_s = tmem + kColS + 128u * static_cast<uint32_t>(sc.t & 1);
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint64_t off = (static_cast<uint32_t>(kk >> 2) * kBoxBytes + static_cast<uint32_t>(kk & 3) * 32u) >> 4;
          tc_mma_ss(d_s, qd + off, kd + off, kIdescS, kk > 0 ? 1u : 0u);
        }
        issued_any = true;
        tc_commit(bar(L::kSlotEmpty + ks));
        if (sc.last_of_item()) tc_commit(bar(L::kQEmpty + (sc.qi & 1)));
        tc_commit(bar(L::kSFull + (sc.t & 1)));
        sc.advance(args);
      }
      // pairs: O += P_t V_t interleaved with S_t+2 = Q K_t+2^T
      while (pc.valid) {
        const int t = pc.t;
        const int vs = next_slot(5);
        if (vs < 0) goto mma_done;
        if (pc.j == 0 && pc.qi > 0)  // the previous item's epilogue has read O
          if (!wait_one(bar(L::kOFree), static_cast<uint32_t>(pc.qi - 1) & 1u, ctl, 6)) goto mma_done;
        if (!wait_one(bar(L::kPFull + (t & 1)), static_cast<uint32_t>(t >> 1) & 1u, ctl, 7)) goto mma_done;
        const bool has_s = sc.valid;
        int ks = -1;
        if (has_s) {
          if (!wait_q(sc)) goto mma_done;
          ks = next_slot(4);
          if (ks < 0) goto mma_done;
        }
        tc_fence_after();
        const uint64_t vd = sdesc_sw128(base + L::kRing + static_cast<uint32_t>(vs) * L::kTile, kBoxBytes, 1024);
        const uint32_t a_p = tmem + kColP + 64u * static_cast<uint32_t>(t & 1);
        const uint32_t first = pc.j == 0 ? 1u : 0u;
        if (has_s) {
          const uint64_t qd = qdesc0 + ((static_cast<uint32_t>(sc.qi & 1) * L::kTile) >> 4);
          const uint64_t kd = sdesc_sw128(base + L::kRing + static_cast<uint32_t>(ks) * L::kTile, 16, 1024);
          const uint32_t d_s = tmem + kColS + 128u * static_cast<uint32_t>(t & 1);
#pragma unroll
          for (int kk = 0; kk < 8; ++kk) {
            // P.V step kk: keys 16 kk .. 16 kk + 15 (2048 bytes of V, 8 TMEM columns of P)
            tc_mma_ts(tmem + kColO, a_p + 8u * kk, vd + ((2048u * kk) >> 4), kIdescO, (first && kk == 0) ? 0u : 1u);
            if (kk < D / 16) {
              // S step kk: 64-column box kk / 4, 32-byte slice kk % 4 of its swizzle atoms
              const uint64_t off =
                  (static_cast<uint32_t>(kk >> 2) * kBoxBytes + static_cast<uint32_t>(kk & 3) * 32u) >> 4;
              tc_mma_ss(d_s, qd + off, kd + off, kIdescS, kk > 0 ? 1u : 0u);
            }
          }
        } else {
#pragma unroll
          for (int kk = 0; kk < 8; ++kk)
            tc_mma_ts(tmem + kColO, a_p + 8u * kk, vd + ((2048u * kk) >> 4), kIdescO, (first && kk == 0) ? 0u : 1u);
        }
        tc_commit(bar(L::kSlotEmpty + vs));
        if (has_s) {
          tc_commit(bar(L::kSlotEmpty + ks));
          if (sc.last_of_item()) tc_commit(bar(L::kQEmpty + (sc.qi & 1)));
          sc.advance(args);
        }
        // buffer t % 2: S_t+2 is ready and pair t (hence O += P_t V_t) is complete
        tc_commit(bar(L::kSFull + (t & 1)));
        pc.advance(args);
      }
    mma_done:
      if (issued_any) {  // every MMA issued must finish before TMEM is freed
        tc_commit(bar(L::kMmaDone));
        drain_one(bar(L::kMmaDone), 0u, args.timeout_ns);
      }
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ softmax
    // s_full[b] phase p completes when S of tile 2p + b is in buffer b; phase
    // p + 1 also means pair 2p + b (O += P V of that tile) is complete.
    const int quarter = warp & 3;
    const int half = warp >> 2;                 // score columns [64 half, 64 half + 64)
    const int trow = quarter * 32 + lane;       // row of the query tile (= TMEM lane)
    const uint32_t lane_off = static_cast<uint32_t>(quarter * 32) << 16;
    const uint32_t col0 = 64u * static_cast<uint32_t>(half);
    constexpr int kOCols = D / 2;               // O columns this thread rescales / stores
    const float sl2 = args.scale_log2;
    float* xbuf = reinterpret_cast<float*>(base_ptr + L::kXBuf);
    const uint32_t xbar = bar(L::kXchg + quarter);
    uint32_t x_phase = 0;                       // exchanges done with the partner thread
    uint32_t s_waited[2] = {0u, 0u};            // phases of s_full[b] already waited for
    int t = 0;                                  // position in the key-tile stream
    // wait until phase `ph` of s_full[b] has completed (each phase once, in order)
    auto wait_s = [&](int b, uint32_t ph, int where) -> bool {
      if (s_waited[b] > ph) return true;
      if (!wait_warp(bar(L::kSFull + b), ph & 1u, ctl, where)) return false;
      s_waited[b] = ph + 1;
      return true;
    };
    // combine a value with the partner thread's (the other half of the row)
    auto exchange = [&](float v, float& other, int where) -> bool {
      float* slot = xbuf + (x_phase & 1u) * 256;
      slot[half * 128 + trow] = v;
      mbar_arrive(xbar);
      if (!wait_warp(xbar, x_phase & 1u, ctl, where)) return false;
      other = slot[(half ^ 1) * 128 + trow];
      ++x_phase;
      return true;
    };
    for (int item = blockIdx.x; item < args.n_items; item += gridDim.x) {
      Task tk;
      int head;
      decode_item(args, item, tk, head);
      int na;
      const int nkv = n_key_tiles(tk, na);
      const bool row_ok = trow < tk.q_rows;
      const int64_t grow = static_cast<int64_t>(tk.q_row0) + trow;
      __nv_bfloat16* orow = args.out + grow * args.row_stride + static_cast<int64_t>(head) * D + half * kOCols;
      if (nkv == 0) {
        if (row_ok) {
          uint4 z = make_uint4(0, 0, 0, 0);
          for (int c = 0; c < kOCols / 8; ++c) reinterpret_cast<uint4*>(orow)[c] = z;
          if (args.lse && half == 0) args.lse[grow * args.num_heads + head] = -INFINITY;
        }
        continue;
      }
      float m_run = 0.f, l_run = 0.f;  // l_run: this thread's half of the row sum
      for (int j = 0; j < nkv; ++j, ++t) {
        const int b = t & 1;
        const TileSrc src = tile_src(tk, na, j);
        if (!wait_s(b, static_cast<uint32_t>(t >> 1), 8)) goto softmax_done;
        tc_fence_after();
        const uint32_t t_s = tmem + lane_off + kColS + 128u * b + col0;
        uint32_t r0[32], r1[32];
        tmem_ld32(t_s + 0u, r0);
        tmem_ld32(t_s + 32u, r1);
        tmem_wait_ld(r0);
        tmem_wait_ld(r1);
        float s[64];
#pragma unroll
        for (int c = 0; c < 32; ++c) {
          s[c] = __uint_as_float(r0[c]);
          s[32 + c] = __uint_as_float(r1[c]);
        }
        const int valid = src.valid - static_cast<int>(col0);  // keys of this half inside the range
        if (valid < 64) {
#pragma unroll
          for (int c = 0; c < 64; ++c)
            if (c >= valid) s[c] = -INFINITY;
        }
        // this half's maximum as a tree (depth 6), then the whole row's
        float mx[32];
#pragma unroll
        for (int c = 0; c < 32; ++c) mx[c] = fmaxf(s[c], s[c + 32]);
#pragma unroll
        for (int w = 16; w >= 1; w >>= 1)
#pragma unroll
          for (int c = 0; c < w; ++c) mx[c] = fmaxf(mx[c], mx[c + w]);
        float mo;
        if (!exchange(mx[0], mo, 11)) goto softmax_done;
        const float m_tile = fmaxf(mx[0], mo) * sl2;
        if (j == 0) {
          m_run = m_tile;
        } else if (__any_sync(0xffffffffu, m_tile > m_run + 8.0f)) {
          // both threads of a row see the same m_tile, so warps q and q + 4 decide alike.
          // Move the running maximum: O must first hold P_{t-1} V_{t-1}
          // (pair t-1 complete = phase (t+1)/2 of s_full[(t+1) % 2])
          if (!wait_s((t + 1) & 1, static_cast<uint32_t>((t + 1) >> 1), 9)) goto softmax_done;
          tc_fence_after();
          const float m_new = fmaxf(m_run, m_tile);
          const float alpha = ex2_approx(m_run - m_new);
          m_run = m_new;
          l_run *= alpha;
          const uint32_t t_o = tmem + lane_off + kColO + static_cast<uint32_t>(half * kOCols);
#pragma unroll
          for (int cc = 0; cc < kOCols / 16; ++cc) {
            uint32_t o[16];
            tmem_ld16(t_o + 16u * cc, o);
            tmem_wait_ld(o);
#pragma unroll
            for (int c = 0; c < 16; ++c) o[c] = __float_as_uint(__uint_as_float(o[c]) * alpha);
            tmem_st16(t_o + 16u * cc, o);
          }
        }
        // P = exp2(scaled S - m) as bf16 pairs into P buffer b (this half: 32 columns)
        const float neg_m = -m_run;
        const uint32_t t_p = tmem + lane_off + kColP + 64u * b + 32u * static_cast<uint32_t>(half);
        float ls[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          uint32_t pk[8];
#pragma unroll
          for (int c = 0; c < 8; ++c) {
            const float x = ex2_approx(fmaf(s[16 * q + 2 * c], sl2, neg_m));
            const float y = ex2_approx(fmaf(s[16 * q + 2 * c + 1], sl2, neg_m));
            ls[(2 * c) & 3] += x;
            ls[(2 * c + 1) & 3] += y;
            pk[c] = pack_bf16x2(x, y);
          }
          tmem_st8(t_p + 8u * q, pk);
        }
        l_run += (ls[0] + ls[1]) + (ls[2] + ls[3]);
        tmem_wait_st();
        tc_fence_before();
        mbar_arrive(bar(L::kPFull + b));
      }
      // epilogue: wait for the item's last pair, then O / l -> bf16 rows
      {
        float l_other;
        if (!exchange(l_run, l_other, 12)) goto softmax_done;
        const float l_row = l_run + l_other;
        const int tl = t - 1;
        if (!wait_s(tl & 1, static_cast<uint32_t>(tl >> 1) + 1u, 10)) goto softmax_done;
        tc_fence_after();
        const float inv_l = 1.0f / l_row;
        const uint32_t t_o = tmem + lane_off + kColO + static_cast<uint32_t>(half * kOCols);
        uint32_t packed[kOCols / 2];
#pragma unroll
        for (int cc = 0; cc < kOCols / 32; ++cc) {
          uint32_t o[32];
          tmem_ld32(t_o + 32u * cc, o);
          tmem_wait_ld(o);
#pragma unroll
          for (int c = 0; c < 16; ++c)
            packed[16 * cc + c] =
                pack_bf16x2(__uint_as_float(o[2 * c]) * inv_l, __uint_as_float(o[2 * c + 1]) * inv_l);
        }
        tc_fence_before();
        mbar_arrive(bar(L::kOFree));
        if (row_ok) {
          uint4* dst = reinterpret_cast<uint4*>(orow);
#pragma unroll
          for (int c = 0; c < kOCols / 8; ++c)
            dst[c] = make_uint4(packed[4 * c], packed[4 * c + 1], packed[4 * c + 2], packed[4 * c + 3]);
          if (args.lse && half == 0)
            args.lse[grow * args.num_heads + head] = (m_run + log2f(l_row)) * 0.69314718055994530942f;
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
