// attn_tc2.cuh -- the tcgen05 attention kernel on CTA pairs: for every
// (task, head) item, O = softmax(scale * Q K^T) V over the task's visible keys
// (key ranges A then B; see common.cuh), scores, softmax and accumulation in
// fp32 and P rounded to bf16 for P.V, with every MMA issued over two CTAs on
// neighbouring SMs (tcgen05 cta_group::2, M = 256).  Head dim 128, or 64
// padded to 128 inside shared memory (see the kernel's kDG).
//
// Why pairs: with one 128-row query tile per SM, each S/P.V pair of MMAs
// (1024 tensor cycles at 128-key tiles) needs a fresh 32 KB K tile and 32 KB
// V tile in that SM's shared memory.  The tensor core's operand reads (about
// 96 KB per pair) plus those 64 KB of TMA fills exceed what one SM's shared
// memory delivers in 1024 cycles (128 bytes per cycle), so the tensor core
// waits for data.  A CTA pair shares every K/V tile: CTA r holds keys
// [kBN/2 r, kBN/2 (r + 1)) of each K tile and head-dim columns [64 r, 64 r +
// 64) of each V tile (the B operand of a cta_group::2 MMA is split along N
// between the two CTAs), while each CTA keeps its own 128 query rows (A is
// split along M).  Per SM this halves the tile bytes fetched and the
// B-operand bytes read, for the same MMA work.
//
// Key tiles (kBN): 192 keys for the bf16 cache, 128 for the E4M3 cache and
// the 128-key comparison variant.  At 192 keys P is written over the first
// half of its own S buffer, which is what makes two 192-column S buffers and
// the 128-column O fit in the 512 TMEM columns; each handshake then carries
// 1536 tensor cycles of MMAs instead of 1024 (see Cfg).
//
// Cluster of 2 CTAs (rank 0 = leader), 224 threads each (352 in the E4M3
// kernel, whose 8 softmax warps split each row's columns, see below):
//   warps 0-3  softmax: thread l of warp w owns row 32 w + l of this CTA's
//              128 rows (its TMEM lane), all kBN score columns of a tile
//   warp 4     TMA producer: this CTA's Q rows and its halves of the K and V
//              tiles; completion is counted on the leader's barriers
//   warp 5     both CTAs: TMEM allocation (a pair operation); leader only:
//              the MMA warp (lane 0 issues every MMA and commit)
//   warp 6     leader only: the gate warp, which does every mbarrier wait
//              the MMAs depend on and hands each group to the MMA warp
//              through a named barrier
// One softmax warp per SM sub-partition leaves the MMA warp's sub-partition
// with a single busy warp beside it, and a row needs no partner thread.
// An item is a task of up to 256 query rows: CTA r takes rows
// [128 r, 128 r + 128).  Items come from a per-item list ordered on the host
// or, head-major, from the task list: with a work counter each CTA pair takes
// the next item of the list whenever it starts one (the leader's producer
// takes it and passes it on through a ring in shared memory), else pair c
// takes items c, c + n_pairs, ...
//
// Work is done item by item (an item = a task of up to 256 rows x one
// head).  An item with n key tiles is a sequence of n + 2 MMA groups:
//   group G + 0, G + 1     S_0 = Q K_0^T, S_1 = Q K_1^T (the second is empty
//                          when n = 1)
//   group G + 2 + j        O += P_j V_j with S_j+2 = Q K_j+2^T when j + 2 < n
//                          (all P.V MMAs first when S_j+2 overwrites P_j,
//                          else interleaved MMA by MMA)
// numbered g = 0, 1, 2, ... over all items of the cluster.  Group g reads
// ring stage g % kStages (K of its S, V of its P.V; 48 KB per CTA at 192-key
// tiles, 32 KB at 128).  Tiles are also numbered over all items (t); S_t and
// P_t live in TMEM buffer t % 2.
//
// Synchronisation is built so that the MMA thread does as little as possible
// between its MMAs: a tcgen05.mma blocks its thread until the tensor core
// takes it, and the tensor core queues almost nothing, so every cycle the
// MMA thread spends between two groups idles the tensor core.  An mbarrier
// wait whose result the MMA thread needs costs it far more than a
// named-barrier handshake, so all mbarrier waits are done by the gate warp:
// per group, the gate warp waits for what the group needs and then meets the
// MMA warp at `bar.red.or` (which also carries an abort bit: both warps walk
// the same group sequence and leave together, so neither can be left waiting);
// the MMA thread then issues the group and commits once:
//   pair_done[g % 4]   one commit per group (multicast to both CTAs): its S
//                      is in TMEM, its P.V is in O, its stage and the P
//                      buffer it read are free.  Four barriers, so that no
//                      waiter can miss a phase: a waiter for group g holds up
//                      group g + 4.
//   p_full[t % 2]      one arrival per softmax warp of both CTAs.  Its phase
//                      for tile t means P_t is in TMEM, every softmax thread
//                      has finished reading O for the previous item, and (the
//                      leader's warp 0 waited for it) the stage of P_t V_t's
//                      group is full.
//   stage_full[s]      the producers' TMA bytes of both CTAs (leader's barrier)
//   q_full / q_empty   per Q buffer, once per item
//
// E4M3 cache (kF8): key range B is the quantised reference cache -- K as
// E4M3 codes [rows_pad, H, 128] and V transposed per head [H, 128, rows_pad],
// both K-major operands, with one fp32 scale (s_K, s_V) per 128-row tile and
// head.  Its tiles run as kind::f8f6f4 MMAs (K = 32 per instruction, half
// the tensor cycles of bf16); range A (the live rows) stays bf16.  At the
// start of an item with cached tiles every softmax thread quantises its own
// query row of this head into an E4M3 Q tile (one scale per row), and the
// first cached tile's S waits for it (q8_full, one arrival per softmax warp
// of both CTAs).  The producer also feeds each CTA a small shared-memory ring
// of the cached tiles' scales (16-byte bulk copies), so that the softmax loop
// touches no global memory.  The scales enter the softmax, so one O
// accumulator serves both ranges: with
// s_ref = s_V of the item's first cached tile, the weights written are
//   live tile:    exp2(u - m) / s_ref                   (bf16, u = scaled score)
//   cached tile:  exp2(u + delta - m), delta = log2(s_V / s_ref)   (E4M3)
// where the running maximum m is taken over u + delta, so E4M3 weights stay
// at most 2^8; each tile adds its unshifted weight sum to l, and
// O = s_ref * acc / l.
#pragma once
#include "attn_tc.cuh"

namespace rc {

namespace tc2 {
using tc::Ctl;
constexpr int kD = 128;
constexpr uint32_t kQTile = 128 * 128 * 2;
// Warp roles: softmax warps first (4, or 8 in the E4M3 kernel, two per SM
// sub-partition), then the producer, the MMA warp and the gate warp.
//
// kBN = keys per tile: 128, or 192 for the bf16 cache.  With 192-key tiles P
// is written over the first half of its own S buffer, so that tensor memory
// holds S_0 [0, 192), S_1 [192, 384) and O [384, 512); an MMA group is then
// 12 P.V MMAs and 8 S MMAs of N = 192 (1536 tensor cycles per handshake
// instead of 1024), and since the S MMAs that reuse a buffer overwrite the P
// that the group's P.V MMAs read, a group issues all its P.V MMAs first.
// With 128-key tiles P has buffers of its own and the two kinds interleave.
template <bool kF8, int kBN>
struct Cfg {
  static_assert(kBN == 128 || (kBN == 192 && !kF8), "key tiles of 128 keys, or 192 with the bf16 cache");
  static constexpr int kHalves = kF8 ? 2 : 1;         // softmax warps per 32 rows
  static constexpr int kSoftmaxWarps = 4 * kHalves;
  static constexpr int kProducerWarp = kSoftmaxWarps, kMmaWarp = kSoftmaxWarps + 1, kGateWarp = kSoftmaxWarps + 2;
  static constexpr int kThreads = 32 * (kSoftmaxWarps + 3);
  static constexpr int kWarpArrivals = 2 * kSoftmaxWarps;  // p_full / q8_full: every softmax warp of both CTAs
  // warps that take each item from the ring (work counter): the leader's
  // gate and softmax warps, the follower's producer and softmax warps
  static constexpr int kItemTakers = 2 + 2 * kSoftmaxWarps;
  static constexpr int kStages = kBN == 128 ? 4 : 3;     // ring stages (shared memory: 2 Q + stages <= 227 KB)
  static constexpr uint32_t kKBox = (kBN / 2) * 128;     // one K box: kBN / 2 rows x 128 bytes
  static constexpr uint32_t kKHalf = 2 * kKBox;          // this CTA's kBN / 2 keys x 128 d of a K tile
  static constexpr uint32_t kVHalf = kBN * 64 * 2;       // kBN keys x this CTA's 64 d of a V tile
  static constexpr uint32_t kStage = kKHalf + kVHalf;
  static constexpr bool kPOverS = kBN != 128;
  static constexpr uint32_t kColS = 0;                   // S buffer b at kColS + b * kBN
  static constexpr uint32_t kColP = kPOverS ? 0u : 256u; // P buffer b at kColP + b * kPStride
  static constexpr uint32_t kPStride = kPOverS ? kBN : 64u;
  static constexpr uint32_t kColO = 384;
  static_assert(2 * kBN <= 384 && kColO + kD <= tc::kTmemCols, "tensor-memory layout");
};
constexpr int kPairDoneBars = 4;          // pair_done[g % 4]: a waiter for group g holds up group g + 4
constexpr uint32_t kGateBarrier = 1;  // named barrier of the MMA and gate warps (0 is __syncthreads)
constexpr uint32_t kKHalf8 = 64 * 128;   // 8 KB: this CTA's 64 keys x 128 d of an E4M3 K tile
constexpr uint32_t kVHalf8 = 64 * 128;   // 8 KB: this CTA's 64 d x 128 keys of an E4M3 V^T tile
constexpr uint32_t kQ8Tile = 128 * 128;  // this CTA's 128 query rows as E4M3
constexpr int kScaleSlots = 8;           // ring of per-tile scales of cached tiles (E4M3 kernel)
constexpr int kItemSlots = 4;            // ring of items taken from the work counter

template <bool kF8, int kBN>
struct SmemT {
  using C = Cfg<kF8, kBN>;
  static constexpr int kStages = C::kStages;
  static constexpr uint32_t kQ = 0;                // Q buffers 0 and 1 (this CTA's 128 rows)
  static constexpr uint32_t kRing = 2 * kQTile;    // stage s: [K half | V half]
  static constexpr uint32_t kQ8 = kRing + kStages * C::kStage;  // E4M3 Q tile (kF8 only)
  static constexpr uint32_t kScales = kQ8 + (kF8 ? kQ8Tile : 0u);  // ring of kScaleSlots x 16 B (kF8 only)
  static constexpr uint32_t kLX = kScales + (kF8 ? kScaleSlots * 16u : 0u);  // [2][128] fp32 partial row sums
  static constexpr uint32_t kBars = kLX + (kF8 ? 2u * 128u * 4u : 0u);
  static constexpr int kQFull = 0, kQEmpty = 2, kStageFull = 4, kPairDone = 4 + kStages,
                       kPFull = kPairDone + kPairDoneBars, kMmaDone = kPFull + 2, kQ8Full = kMmaDone + 1,
                       kLXFull = kQ8Full + 1, kScaleFull = kLXFull + 1, kScaleEmpty = kScaleFull + kScaleSlots,
                       kItemFull = kScaleEmpty + kScaleSlots, kItemEmpty = kItemFull + kItemSlots,
                       kNumBars = kItemEmpty + kItemSlots;
  static constexpr uint32_t kTmemHolder = kBars + 8 * kNumBars;
  static constexpr uint32_t kAbort = kTmemHolder + 4;
  // load record of each CTA of the pair (leader's copy read at teardown):
  // per CTA [loads per stage (kStages) | own bytes of the last load per stage
  // (kStages) | the other CTA's bytes of that load (kStages) | loads per Q
  // buffer (2)]
  static constexpr uint32_t kRecWords = 3 * kStages + 2;
  static constexpr uint32_t kLoadRec = kAbort + 4;
  // ring of taken items (work counter): slot k % kItemSlots holds item k of
  // this cluster (-1: none left); the gate warp passes the MMA warp its item
  static constexpr uint32_t kItemRing = kLoadRec + 2 * kRecWords * 4;
  static constexpr uint32_t kGateItem = kItemRing + 4 * kItemSlots;
  static constexpr uint32_t kUsed = kGateItem + 4;
  static constexpr uint32_t kMaxDynamic = 232448;
  static constexpr uint32_t kDynamic = kUsed + 1024 < kMaxDynamic ? kUsed + 1024 : kMaxDynamic;
  static_assert(kUsed <= kMaxDynamic, "shared-memory layout too large");
  static_assert(C::kStage % 1024 == 0 && C::kKBox % 1024 == 0, "swizzle atoms start on 1024-byte boundaries");
};

// Key tiles of kBN keys: tile j of an item (range A first, then range B).
template <int kBN>
__device__ __forceinline__ tc::TileSrc tile_src(const Task& t, int na, int j) {
  tc::TileSrc s;
  if (j < na) {
    s.row = t.a_row0 + j * kBN;
    s.valid = min(kBN, t.a_len - j * kBN);
    s.in_b = false;
  } else {
    const int jj = j - na;
    s.row = t.b_row0 + jj * kBN;
    s.valid = min(kBN, t.b_len - jj * kBN);
    s.in_b = true;
  }
  return s;
}
template <int kBN>
__device__ __forceinline__ int n_key_tiles(const Task& t, int& na) {
  na = (t.a_len + kBN - 1) / kBN;
  return na + (t.b_len + kBN - 1) / kBN;
}

// Phase parity of pair_done[g % 4] for group g.
__device__ __forceinline__ uint32_t group_parity(int g) { return static_cast<uint32_t>(g >> 2) & 1u; }
// Ring stage of group g and the phase parity of its stage_full barrier.
template <int kStages>
__device__ __forceinline__ int stage_of(int g) { return g % kStages; }
template <int kStages>
__device__ __forceinline__ uint32_t stage_parity(int g) { return static_cast<uint32_t>(g / kStages) & 1u; }

// Bounded wait with cluster-scope acquire (barriers other CTAs arrive on).
__device__ __forceinline__ bool wait_cl(uint32_t bar, uint32_t parity, const Ctl& c, int where) {
  if (mbar_try_wait_cluster(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (;;) {
    for (int i = 0; i < 16; ++i)
      if (mbar_try_wait_cluster(bar, parity)) return true;
    if (*c.abort_flag) return false;
    if (globaltimer_ns() - t0 > c.timeout_ns) {
      *c.abort_flag = 1;
      tc::report_timeout(c.status, where);
      return false;
    }
  }
}
__device__ __forceinline__ bool wait_cl_warp(uint32_t bar, uint32_t parity, const Ctl& c, int where) {
  const bool ok = wait_cl(bar, parity, c, where);
  return __all_sync(0xffffffffu, ok);
}
// Work counter [next item, clusters done]: this cluster has finished (every
// item it took is done or abandoned); the last cluster resets both words for
// the next launch, which reads them only after this grid has completed.
__device__ __forceinline__ void work_done(int* work, int n_clusters) {
  __threadfence();
  if (atomicAdd(work + 1, 1) == n_clusters - 1) {
    __threadfence();
    atomicExch(work, 0);
    atomicExch(work + 1, 0);
  }
}
}  // namespace tc2

// kDG: the tensors' head dim.  At 64 the tiles keep the layout of head dim
// 128 with the upper 64 columns as zero padding: Q and K tiles load only
// their first 64-column box (S = Q K^T takes the first four K = 16 steps), the
// second CTA of a pair holds the upper half of V's columns, which it never
// loads but zeroes once (P V keeps N = 128; O's upper 64 columns stay zero and
// are never read).
template <bool kF8, int kBN, int kDG>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(tc2::Cfg<kF8, kBN>::kThreads, 1)
    attn_tc2_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_ka,
                    const __grid_constant__ CUtensorMap tm_va, const __grid_constant__ CUtensorMap tm_kb,
                    const __grid_constant__ CUtensorMap tm_vb, const AttnArgs args) {
  using namespace tc;
  using tc2::kQTile;
  using Cfg = tc2::Cfg<kF8, kBN>;
  constexpr uint32_t kKBox = Cfg::kKBox;
  constexpr uint32_t kKHalf = Cfg::kKHalf;
  constexpr uint32_t kVHalf = Cfg::kVHalf;
  constexpr uint32_t kStage = Cfg::kStage;
  constexpr int kStages = Cfg::kStages;
  constexpr uint32_t kColS = Cfg::kColS, kColP = Cfg::kColP, kPStride = Cfg::kPStride, kColO = Cfg::kColO;
  constexpr int kWarpArrivals = Cfg::kWarpArrivals;
  using tc2::group_parity;
  using tc2::wait_cl;
  using tc2::wait_cl_warp;
  using tc2::kKHalf8;
  using tc2::kVHalf8;
  using L = tc2::SmemT<kF8, kBN>;
  constexpr int D = tc2::kD;   // head-dim columns of the tiles (P V's N)
  constexpr int DG = kDG;      // head dim of the tensors
  static_assert(DG == D || (DG == 64 && !kF8), "head dim 128, or 64 (bf16 cache) padded to 128");
  constexpr int kQBoxes = DG / 64;  // 64-column boxes of a Q or K row loaded
  auto stage_of = [](int g) -> int { return tc2::stage_of<kStages>(g); };
  auto stage_parity = [](int g) -> uint32_t { return tc2::stage_parity<kStages>(g); };
  constexpr uint32_t kIdescS = idesc_bf16_f32(256, kBN, false);
  constexpr uint32_t kIdescO = idesc_bf16_f32(256, D, true);
  constexpr uint32_t kIdesc8 = idesc_e4m3_f32(256, 128);  // S and O of cached tiles (N = 128 keys or d)

  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* base_ptr = smem_raw + (base - raw);
  auto bar = [&](int i) -> uint32_t { return base + L::kBars + 8u * static_cast<uint32_t>(i); };
  volatile int* abort_flag = reinterpret_cast<volatile int*>(base_ptr + L::kAbort);
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(base_ptr + L::kTmemHolder);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const bool leader = rank == 0;
  const int cluster = static_cast<int>(blockIdx.x >> 1);
  const int n_clusters = static_cast<int>(gridDim.x >> 1);
  // Both CTAs of a pair get the same layout, so both leave here together.
  if (base - raw + L::kUsed > L::kDynamic) {
    if (threadIdx.x == 0) tc::report_timeout(args.status, 99);
    if (threadIdx.x == 0 && leader && args.work != nullptr) tc2::work_done(args.work, n_clusters);
    return;
  }

  if (threadIdx.x == 0) {
    for (int i = 0; i < 2; ++i) {
      mbar_init(bar(L::kQFull + i), 1);
      mbar_init(bar(L::kQEmpty + i), 1);
      mbar_init(bar(L::kPFull + i), kWarpArrivals);
    }
    for (int s = 0; s < kStages; ++s) mbar_init(bar(L::kStageFull + s), 1);
    for (int s = 0; s < tc2::kPairDoneBars; ++s) mbar_init(bar(L::kPairDone + s), 1);
    mbar_init(bar(L::kMmaDone), 1);
    mbar_init(bar(L::kQ8Full), kWarpArrivals);
    mbar_init(bar(L::kLXFull), Cfg::kSoftmaxWarps);
    for (int s = 0; s < tc2::kScaleSlots; ++s) {
      mbar_init(bar(L::kScaleFull + s), 1);
      mbar_init(bar(L::kScaleEmpty + s), Cfg::kSoftmaxWarps);
    }
    for (int s = 0; s < tc2::kItemSlots; ++s) {
      mbar_init(bar(L::kItemFull + s), 1);
      mbar_init(bar(L::kItemEmpty + s), Cfg::kItemTakers);
    }
    *abort_flag = 0;
    fence_barrier_init();
    fence_proxy_async_smem();
  }
  if constexpr (DG != D) {
    // head dim 64: the second CTA's V half of every stage is the zero padding
    // of the upper 64 head-dim columns (written once; that CTA never loads V)
    if (rank == 1) {
      constexpr uint32_t kChunks = kVHalf / 16;
      for (uint32_t i = threadIdx.x; i < kStages * kChunks; i += blockDim.x)
        st_shared_v4(base + L::kRing + (i / kChunks) * kStage + kKHalf + (i % kChunks) * 16u, make_uint4(0, 0, 0, 0));
      fence_proxy_async_smem();
    }
  }
  if (warp == Cfg::kMmaWarp) {
    tmem_alloc_pair(smem_u32(tmem_holder), kTmemCols);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // both CTAs' barriers exist before any cross-CTA arrival
  tc_fence_after();
  // launched as a programmatic dependent of the previous kernel on the stream:
  // everything above overlaps its tail, nothing below reads memory before it
  // is complete; and the next kernel may start its CTAs (they wait likewise)
  grid_dependency_wait();
  if (threadIdx.x == 0) grid_launch_dependents();
  const uint32_t tmem = *tmem_holder;
  const Ctl ctl{abort_flag, args.timeout_ns, args.status};
  auto lbar = [&](int i) -> uint32_t { return mapa_shared(bar(i), 0); };  // leader's barrier i
  // Item k of this cluster (k = 0, 1, ...; -1 once there is none, -2 after a
  // failed wait).  Static order: cluster + k * n_clusters.  With a work
  // counter the leader's producer takes the next item of the list for each k
  // (atomic increment) and writes it to ring slot k % kItemSlots of both CTAs;
  // the other warps read it there.  A slot is reused once every taker has
  // read it (item_empty, on the leader).
  const bool dyn = args.work != nullptr;
  volatile int* item_ring = reinterpret_cast<volatile int*>(base_ptr + L::kItemRing);
  auto static_item = [&](int k) -> int {
    const int64_t it = static_cast<int64_t>(cluster) + static_cast<int64_t>(k) * n_clusters;
    return it < args.n_items ? static_cast<int>(it) : -1;
  };
  auto publish_item = [&](int k) -> int {  // leader's producer (one thread)
    const int s = k % tc2::kItemSlots;
    if (k >= tc2::kItemSlots &&
        !wait_cl(bar(L::kItemEmpty + s), static_cast<uint32_t>(k / tc2::kItemSlots - 1) & 1u, ctl, 21))
      return -2;
    int it = atomicAdd(args.work, 1);
    if (it >= args.n_items) it = -1;
    item_ring[s] = it;
    st_cluster_u32(mapa_shared(base + L::kItemRing + 4u * static_cast<uint32_t>(s), 1), static_cast<uint32_t>(it));
    mbar_arrive(bar(L::kItemFull + s));
    mbar_arrive_release_cluster(mapa_shared(bar(L::kItemFull + s), 1));
    return it;
  };
  auto take_item = [&](int k, int where) -> int {  // one thread of a taking warp
    const int s = k % tc2::kItemSlots;
    if (!wait_cl(bar(L::kItemFull + s), static_cast<uint32_t>(k / tc2::kItemSlots) & 1u, ctl, where)) return -2;
    const int it = item_ring[s];
    mbar_arrive_release_cluster(lbar(L::kItemEmpty + s));
    return it;
  };
  auto take_item_warp = [&](int k, int where) -> int {
    int it = 0;
    if (lane == 0) it = dyn ? take_item(k, where) : static_item(k);
    return __shfl_sync(0xffffffffu, it, 0);
  };

  if (warp == Cfg::kProducerWarp) {
    // ------------------------------------------------------------ producer (both CTAs)
    // This CTA's halves of the stages of every group, in group order, and an
    // item's Q rows just before its first stage.
    if (lane == 0) {
      // loads this CTA issued per stage and per Q buffer, and its bytes of the
      // last load of each stage; the leader arms every phase for both CTAs'
      // bytes right before it issues its own half
      int n_stage[kStages];
      uint32_t own_bytes[kStages], other_bytes[kStages];
      for (int s = 0; s < kStages; ++s) {
        n_stage[s] = 0;
        own_bytes[s] = 0;
        other_bytes[s] = 0;
      }
      int n_q[2] = {0, 0};
      int scale_armed[tc2::kScaleSlots];
      for (int s = 0; s < tc2::kScaleSlots; ++s) scale_armed[s] = -1;
      bool skip_next = leader && args.dbg_skip_first_load != 0;
      int g = 0, qi = 0, si = 0;  // si: cached tiles whose scales went into the ring
      Task tk;
      int head = 0, na = 0;
      // stage of group g: K tile kj (if kj >= 0) and V tile vj (if vj >= 0) of the item
      auto load_stage = [&](int kj, int vj) -> bool {
        const int slot = stage_of(g);
        // the stage's previous group (g - kStages) must be complete
        if (g >= kStages &&
            !wait_one(bar(L::kPairDone + ((g - kStages) & 3)), group_parity(g - kStages), ctl, 2))
          return false;
        const uint32_t dst = base + L::kRing + static_cast<uint32_t>(slot) * kStage;
        const uint32_t full = lbar(L::kStageFull + slot);
        const TileSrc ks = tc2::tile_src<kBN>(tk, na, kj >= 0 ? kj : 0);
        const TileSrc vs = tc2::tile_src<kBN>(tk, na, vj >= 0 ? vj : 0);
        const bool k8 = kF8 && kj >= 0 && ks.in_b, v8 = kF8 && vj >= 0 && vs.in_b;
        // each CTA's K bytes; a V half (at head dim 64 only the first CTA loads one)
        const uint32_t kb = kj >= 0 ? (k8 ? kKHalf8 : kKBox * kQBoxes) : 0u;
        const uint32_t vb = vj >= 0 ? (v8 ? kVHalf8 : kVHalf) : 0u;
        const bool v_here = DG == D || rank == 0;
        const uint32_t bytes = 2 * kb + (DG == D ? 2 : 1) * vb;  // both CTAs
        if (k8) {
          // this CTA's softmax warps read the cached tile's scales from ring slot
          // si % kScaleSlots; the slot's previous tile must have been read
          const int sl = si % tc2::kScaleSlots, use = si / tc2::kScaleSlots;
          if (use > 0 && !wait_one(bar(L::kScaleEmpty + sl), static_cast<uint32_t>(use - 1) & 1u, ctl, 16)) return false;
          mbar_arrive_expect_tx(bar(L::kScaleFull + sl), 16u);
          scale_armed[sl] = use & 1;
          bulk_load(base + L::kScales + 16u * static_cast<uint32_t>(sl),
                    args.b_scales + ((tk.b_row0 >> 7) + (kj - na)) * args.num_heads + head, 16u,
                    bar(L::kScaleFull + sl));
          ++si;
        }
        if (skip_next) {  // fault injection: the leader never arms or loads this stage
          skip_next = false;
        } else {
          if (leader) mbar_arrive_expect_tx(bar(L::kStageFull + slot), bytes);
          ++n_stage[slot];
          own_bytes[slot] = kb + (v_here ? vb : 0u);
          other_bytes[slot] = kb + (DG == D || rank == 1 ? vb : 0u);
          if (k8) {  // E4M3 keys [64 r, 64 r + 64): one box of 64 rows x 128 bytes
            tma_load_2d_pair(dst, &tm_kb, full, head * D, ks.row + 64 * static_cast<int>(rank));
          } else if (kj >= 0) {  // keys [kBN/2 r, kBN/2 (r + 1)) of the tile, both head-dim boxes
            const void* map = ks.in_b ? &tm_kb : &tm_ka;
            for (int ch = 0; ch < kQBoxes; ++ch)
              tma_load_2d_pair(dst + ch * kKBox, map, full, head * DG + ch * 64,
                               ks.row + (kBN / 2) * static_cast<int>(rank));
          }
          if (v8) {  // E4M3 V^T rows d in [64 r, 64 r + 64), all 128 keys
            tma_load_2d_pair(dst + kKHalf, &tm_vb, full, vs.row, head * D + 64 * static_cast<int>(rank));
          } else if (vj >= 0 && v_here) {  // head-dim columns [64 r, 64 r + 64) of all kBN keys
            const void* map = vs.in_b ? &tm_vb : &tm_va;
            tma_load_2d_pair(dst + kKHalf, map, full, head * DG + 64 * static_cast<int>(rank), vs.row);
          }
        }
        ++g;
        return true;
      };
      for (int k = 0;; ++k) {
        const int item = !dyn ? static_item(k) : leader ? publish_item(k) : take_item(k, 18);
        if (item == -2) goto producer_done;
        if (item < 0) break;
        decode_item(args, item, tk, head);
        const int nkv = tc2::n_key_tiles<kBN>(tk, na);
        if (nkv == 0) continue;
        {  // this CTA's 128 query rows into Q buffer qi % 2
          const int b = qi & 1;
          const uint32_t n = static_cast<uint32_t>(qi >> 1);
          if (!wait_one(bar(L::kQEmpty + b), (n & 1u) ^ 1u, ctl, 1)) goto producer_done;
          if (leader) mbar_arrive_expect_tx(bar(L::kQFull + b), 2 * kQBoxes * kBoxBytes);
          ++n_q[b];
          const uint32_t qfull = lbar(L::kQFull + b);
          for (int ch = 0; ch < kQBoxes; ++ch)
            tma_load_2d_pair(base + L::kQ + b * kQTile + ch * kBoxBytes, &tm_q, qfull, head * DG + ch * 64,
                             tk.q_row0 + 128 * static_cast<int>(rank));
        }
        if (!load_stage(0, -1)) goto producer_done;
        if (!load_stage(nkv > 1 ? 1 : -1, -1)) goto producer_done;
        for (int j = 0; j < nkv; ++j)
          if (!load_stage(j + 2 < nkv ? j + 2 : -1, j)) goto producer_done;
        ++qi;
      }
    producer_done:
      // the scale ring's barriers are this CTA's own
      for (int s = 0; s < tc2::kScaleSlots; ++s)
        if (scale_armed[s] >= 0) drain_one(bar(L::kScaleFull + s), static_cast<uint32_t>(scale_armed[s]), args.timeout_ns);
      // stage and Q loads of both CTAs complete on the leader's barriers: record
      // this CTA's loads in the leader's shared memory, where the leader
      // settles and drains them after the teardown's first cluster barrier
      const uint32_t rec = mapa_shared(base + L::kLoadRec + rank * (L::kRecWords * 4u), 0);
      for (int s = 0; s < kStages; ++s) {
        st_cluster_u32(rec + 4u * s, static_cast<uint32_t>(n_stage[s]));
        st_cluster_u32(rec + 4u * (kStages + s), own_bytes[s]);
        st_cluster_u32(rec + 4u * (2 * kStages + s), other_bytes[s]);
      }
      st_cluster_u32(rec + 4u * (3 * kStages), static_cast<uint32_t>(n_q[0]));
      st_cluster_u32(rec + 4u * (3 * kStages + 1), static_cast<uint32_t>(n_q[1]));
    }
    __syncwarp();
  } else if (warp == Cfg::kMmaWarp) {
    // ------------------------------------------------------------ MMA warp (leader)
    if (leader) {
      // descriptors of stage 0 (stage s: + s * kStage / 16) and of Q buffer 0
      const uint64_t kd0 = sdesc_sw128(base + L::kRing, 16, 1024);
      const uint64_t vd0 = sdesc_sw128(base + L::kRing + kKHalf, Cfg::kVHalf, 1024);
      const uint64_t qdesc0 = sdesc_sw128(base + L::kQ, 16, 1024);
      // E4M3 operands: Q8 (128 rows x 128 B), K8 half (64 rows x 128 B), V^T half (64 d x 128 B); a
      // K = 32 step advances 32 bytes inside the swizzle atom
      const uint64_t q8d = sdesc_sw128(base + L::kQ8, 16, 1024);
      const uint64_t vd80 = sdesc_sw128(base + L::kRing + kKHalf, 16, 1024);
      // S step kk: A = Q (128-row boxes of 16 KB), B = this CTA's kBN / 2 keys (boxes of kBN / 2 rows)
      auto q_off = [](int kk) -> uint64_t {
        return (static_cast<uint32_t>(kk >> 2) * kBoxBytes + static_cast<uint32_t>(kk & 3) * 32u) >> 4;
      };
      auto k_off = [](int kk) -> uint64_t {
        return (static_cast<uint32_t>(kk >> 2) * kKBox + static_cast<uint32_t>(kk & 3) * 32u) >> 4;
      };
      bool issued = false;
      int g = 0, t0 = 0, qi = 0;
      const volatile int* gate_item = reinterpret_cast<const volatile int*>(base_ptr + L::kGateItem);
      for (;;) {
        // the gate warp names the next item with key tiles at this handshake;
        // none left (or a failed wait) ends both warps
        if (bar_red_or(tc2::kGateBarrier, 64, false)) goto mma_done;
        Task tk;
        int head, na;
        decode_item(args, *gate_item, tk, head);
        const int nkv = tc2::n_key_tiles<kBN>(tk, na);
        const int qb = qi & 1;
        const uint64_t qd = qdesc0 + ((static_cast<uint32_t>(qb) * kQTile) >> 4);
        // groups G, G + 1: S_0, S_1 (the gate warp has seen the Q tile and stage g land)
        for (int n = 0; n < 2; ++n, ++g) {
          if (bar_red_or(tc2::kGateBarrier, 64, false)) goto mma_done;
          const int slot = stage_of(g);
          if (lane == 0) {
            if (n < nkv) {
              tc_fence_after();
              const uint64_t kd = kd0 + static_cast<uint64_t>(slot) * (kStage >> 4);
              const uint32_t d_s = tmem + kColS + static_cast<uint32_t>((t0 + n) & 1) * kBN;
              if (kF8 && n >= na) {
#pragma unroll
                for (int kk = 0; kk < 4; ++kk)
                  tc2_mma_ss_f8(d_s, q8d + ((32u * kk) >> 4), kd + ((32u * kk) >> 4), kIdesc8, kk > 0 ? 1u : 0u);
              } else {
#pragma unroll
                for (int kk = 0; kk < DG / 16; ++kk)
                  tc2_mma_ss(d_s, qd + q_off(kk), kd + k_off(kk), kIdescS, kk > 0 ? 1u : 0u);
              }
              if (n == nkv - 1) tc2_commit_mc(bar(L::kQEmpty + qb), 3);
            }
            tc2_commit_mc(bar(L::kPairDone + (g & 3)), 3);
          }
          issued = true;
          __syncwarp();
        }
        // groups G + 2 + j: P_j V_j (+ S_j+2) (the gate warp has seen P_t, which
        // also covers this group's stage and the previous item's O reads)
        for (int j = 0; j < nkv; ++j, ++g) {
          if (bar_red_or(tc2::kGateBarrier, 64, false)) goto mma_done;
          if (lane == 0) {
            const int t = t0 + j;
            tc_fence_after();
            const int slot = stage_of(g);
            const uint64_t soff = static_cast<uint64_t>(slot) * (kStage >> 4);
            const uint64_t vd = vd0 + soff;
            const uint32_t a_p = tmem + kColP + static_cast<uint32_t>(t & 1) * kPStride;
            const uint32_t acc0 = j > 0 ? 1u : 0u;
            const bool pv8 = kF8 && j >= na;      // P_j V_j on E4M3 operands
            const bool s8 = kF8 && j + 2 >= na;   // S_j+2 on E4M3 operands
            const uint64_t vd8 = vd80 + soff;
            if (j + 2 < nkv) {
              const uint64_t kd = kd0 + soff;
              const uint32_t d_s = tmem + kColS + static_cast<uint32_t>(t & 1) * kBN;
              if (!s8 && Cfg::kPOverS) {
                // S_j+2 overwrites P_j: every P.V MMA of the group goes first
#pragma unroll
                for (int kk = 0; kk < kBN / 16; ++kk)
                  tc2_mma_ts(tmem + kColO, a_p + 8u * kk, vd + ((2048u * kk) >> 4), kIdescO, kk > 0 ? 1u : acc0);
#pragma unroll
                for (int kk = 0; kk < DG / 16; ++kk)
                  tc2_mma_ss(d_s, qd + q_off(kk), kd + k_off(kk), kIdescS, kk > 0 ? 1u : 0u);
              } else if (!s8) {
#pragma unroll
                for (int kk = 0; kk < 8; ++kk) {
                  tc2_mma_ts(tmem + kColO, a_p + 8u * kk, vd + ((2048u * kk) >> 4), kIdescO, kk > 0 ? 1u : acc0);
                  if (kk < DG / 16) tc2_mma_ss(d_s, qd + q_off(kk), kd + k_off(kk), kIdescS, kk > 0 ? 1u : 0u);
                }
              } else if (pv8) {
#pragma unroll
                for (int kk = 0; kk < 4; ++kk) {
                  tc2_mma_ts_f8(tmem + kColO, a_p + 8u * kk, vd8 + ((32u * kk) >> 4), kIdesc8, kk > 0 ? 1u : acc0);
                  tc2_mma_ss_f8(d_s, q8d + ((32u * kk) >> 4), kd + ((32u * kk) >> 4), kIdesc8, kk > 0 ? 1u : 0u);
                }
              } else {  // the last live tiles' P.V beside the first cached tiles' S
#pragma unroll
                for (int kk = 0; kk < 8; ++kk) {
                  tc2_mma_ts(tmem + kColO, a_p + 8u * kk, vd + ((2048u * kk) >> 4), kIdescO, kk > 0 ? 1u : acc0);
                  if (kk < 4)
                    tc2_mma_ss_f8(d_s, q8d + ((32u * kk) >> 4), kd + ((32u * kk) >> 4), kIdesc8, kk > 0 ? 1u : 0u);
                }
              }
              if (j + 2 == nkv - 1) tc2_commit_mc(bar(L::kQEmpty + qb), 3);
            } else if (pv8) {
#pragma unroll
              for (int kk = 0; kk < 4; ++kk)
                tc2_mma_ts_f8(tmem + kColO, a_p + 8u * kk, vd8 + ((32u * kk) >> 4), kIdesc8, kk > 0 ? 1u : acc0);
            } else {
#pragma unroll
              for (int kk = 0; kk < kBN / 16; ++kk)
                tc2_mma_ts(tmem + kColO, a_p + 8u * kk, vd + ((2048u * kk) >> 4), kIdescO, kk > 0 ? 1u : acc0);
            }
            tc2_commit_mc(bar(L::kPairDone + (g & 3)), 3);
          }
          __syncwarp();
        }
        t0 += nkv;
        ++qi;
      }
    mma_done:
      if (issued && lane == 0) {  // every MMA must finish before TMEM is freed
        tc2_commit_mc(bar(L::kMmaDone), 1);
        drain_one(bar(L::kMmaDone), 0u, args.timeout_ns);
      }
    }
    __syncwarp();
  } else if (warp == Cfg::kGateWarp) {
    // ------------------------------------------------------------ gate warp (leader)
    // The same group sequence as the MMA warp; every wait is bounded, and a
    // failed wait is passed on through the handshake, after which both leave.
    if (leader) {
      int g = 0, t0 = 0, qi = 0, q8i = 0;
      volatile int* gate_item = reinterpret_cast<volatile int*>(base_ptr + L::kGateItem);
      for (int k = 0;; ++k) {
        const int item = take_item_warp(k, 19);
        Task tk;
        int head = 0, na = 0, nkv = 0;
        if (item >= 0) {
          decode_item(args, item, tk, head);
          nkv = tc2::n_key_tiles<kBN>(tk, na);
          if (nkv == 0) continue;
        }
        // the MMA warp takes the item from here; the end of the list, or a
        // failed wait, ends both warps
        if (lane == 0) *gate_item = item;
        if (bar_red_or(tc2::kGateBarrier, 64, item < 0)) goto gate_done;
        // the first cached tile's S also needs the E4M3 Q tile of both CTAs
        const bool q8 = kF8 && nkv > na;
        const uint32_t q8_parity = static_cast<uint32_t>(q8i) & 1u;
        bool ok = wait_cl_warp(bar(L::kQFull + (qi & 1)), static_cast<uint32_t>(qi >> 1) & 1u, ctl, 3);
        for (int n = 0; n < 2; ++n, ++g) {
          ok = ok && wait_cl_warp(bar(L::kStageFull + stage_of(g)), stage_parity(g), ctl, 4);
          if (q8 && n == na) ok = ok && wait_cl_warp(bar(L::kQ8Full), q8_parity, ctl, 14);
          if (bar_red_or(tc2::kGateBarrier, 64, !ok)) goto gate_done;
        }
        for (int j = 0; j < nkv; ++j, ++g) {
          const int t = t0 + j;
          ok = wait_cl_warp(bar(L::kPFull + (t & 1)), static_cast<uint32_t>(t >> 1) & 1u, ctl, 7);
          if (q8 && j + 2 == na) ok = ok && wait_cl_warp(bar(L::kQ8Full), q8_parity, ctl, 14);
          if (bar_red_or(tc2::kGateBarrier, 64, !ok)) goto gate_done;
        }
        t0 += nkv;
        ++qi;
        if (q8) ++q8i;
      }
    gate_done:;
    }
  } else {
    // ------------------------------------------------------------ softmax (both CTAs)
    // kH = 1: warp w (0-3) owns rows 32 w .. 32 w + 31 of this CTA's 128 rows
    // (its TMEM lanes) and all 128 key columns.  kH = 2 (E4M3 kernel): warps w
    // and w + 4 share those rows, warp w + 4 hh taking key columns and O
    // columns [64 hh, 64 hh + 64), so that two warps per SM sub-partition share
    // the exponentials.  Both read the whole S row, find the same row maximum
    // and take the same rescale decisions; their partial row sums meet in the
    // epilogue through shared memory.
    constexpr int kH = Cfg::kHalves;
    constexpr int kC = kBN / kH;  // key columns of this thread
    constexpr int kOC = DG / kH;  // O columns of this thread
    const int quarter = warp & 3, hh = warp >> 2;
    const int col0 = hh * kC, ocol0 = hh * kOC;
    const int trow = quarter * 32 + lane;                  // row within this CTA's 128 rows (= TMEM lane)
    const int prow = 128 * static_cast<int>(rank) + trow;  // row within the item
    const uint32_t lane_off = static_cast<uint32_t>(quarter * 32) << 16;
    const float sl2 = args.scale_log2;
    const f32x2 sl2x2 = make_f32x2(sl2, sl2);
    float* lx = reinterpret_cast<float*>(base_ptr + L::kLX);  // [2][128] partial row sums (kH = 2)
    int t = 0;     // tiles of earlier items
    int G = 0;     // first group of the item
    int n_lx = 0;  // row-sum exchanges so far (kH = 2)
    int si = 0;    // cached tiles read from the scale ring so far
    // wait until group g is complete (both CTAs see the multicast commit)
    auto wait_group = [&](int g, int where) -> bool {
      return wait_cl_warp(bar(L::kPairDone + (g & 3)), group_parity(g), ctl, where);
    };
    for (int k = 0;; ++k) {
      const int item = take_item_warp(k, 20);
      if (item == -2) goto softmax_done;
      if (item < 0) break;
      Task tk;
      int head;
      decode_item(args, item, tk, head);
      int na;
      const int nkv = tc2::n_key_tiles<kBN>(tk, na);
      const bool row_ok = prow < tk.q_rows;
      const int64_t grow = static_cast<int64_t>(tk.q_row0) + prow;
      __nv_bfloat16* orow = args.out + grow * args.row_stride + static_cast<int64_t>(head) * DG + ocol0;
      if (nkv == 0) {
        if (row_ok) {
          uint4 z = make_uint4(0, 0, 0, 0);
          for (int c = 0; c < kOC / 8; ++c) reinterpret_cast<uint4*>(orow)[c] = z;
          if (args.lse && hh == 0) args.lse[grow * args.num_heads + head] = -INFINITY;
        }
        continue;
      }
      float m_run = 0.f, l_run = 0.f;
      // E4M3 cache: this row's query scale (folded into sl2) and the weight scale s_ref
      float c_row = sl2, s_ref = 1.f, l2_ref = 0.f;
      const int scale_row0 = kF8 ? (tk.b_row0 >> 7) * args.num_heads + head : 0;
      if (kF8 && nkv > na) {
        // quantise this thread's query row of this head into the E4M3 Q tile:
        // s = amax / 448, code = E4M3(x * (448 / amax)), round to nearest even
        // (the maximum over the whole row; each half writes its own columns)
        uint4 raw[16];
        if (row_ok) {
          const uint4* src = reinterpret_cast<const uint4*>(args.q + grow * args.row_stride + static_cast<int64_t>(head) * D);
#pragma unroll
          for (int c = 0; c < 16; ++c) raw[c] = src[c];
        } else {
#pragma unroll
          for (int c = 0; c < 16; ++c) raw[c] = make_uint4(0, 0, 0, 0);
        }
        float amax = 0.f;
#pragma unroll
        for (int c = 0; c < 16; ++c) {
          const uint32_t w4[4] = {raw[c].x, raw[c].y, raw[c].z, raw[c].w};
#pragma unroll
          for (int e = 0; e < 4; ++e)
            amax = fmax3(amax, fabsf(__uint_as_float(w4[e] << 16)), fabsf(__uint_as_float(w4[e] & 0xFFFF0000u)));
        }
        const float inv = amax > 0.f ? __fdiv_rn(448.f, amax) : 0.f;
        const uint32_t q8_row = base + L::kQ8 + static_cast<uint32_t>(trow) * 128u;
#pragma unroll
        for (int c = 0; c < 8; ++c) {  // 16 codes per 16-byte chunk, 128-byte swizzle
          if (kH == 2 && (c >> 2) != hh) continue;
          uint32_t w[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const uint32_t x0 = e < 2 ? (&raw[2 * c].x)[2 * e] : (&raw[2 * c + 1].x)[2 * e - 4];
            const uint32_t x1 = e < 2 ? (&raw[2 * c].x)[2 * e + 1] : (&raw[2 * c + 1].x)[2 * e - 3];
            w[e] = pack_e4m3x4(__fmul_rn(__uint_as_float(x0 << 16), inv), __fmul_rn(__uint_as_float(x0 & 0xFFFF0000u), inv),
                               __fmul_rn(__uint_as_float(x1 << 16), inv), __fmul_rn(__uint_as_float(x1 & 0xFFFF0000u), inv));
          }
          st_shared_v4(q8_row + ((static_cast<uint32_t>(c) ^ static_cast<uint32_t>(trow & 7)) << 4),
                       make_uint4(w[0], w[1], w[2], w[3]));
        }
        // visible to the tensor core, then one arrival per warp of both CTAs
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive_release_cluster(mapa_shared(bar(L::kQ8Full), 0));
        c_row = sl2 * __fdiv_rn(amax, 448.f);
        const float4 sc0 = args.b_scales[scale_row0];
        s_ref = sc0.y > 0.f ? sc0.y : 1.f;
        l2_ref = sc0.y > 0.f ? sc0.z : 0.f;
      }
      for (int j = 0; j < nkv; ++j, ++t) {
        const int b = t & 1;
        const TileSrc src = tc2::tile_src<kBN>(tk, na, j);
        // per-tile constants: u = c * s + shift is the shifted scaled score, the
        // weight written is exp2(u - m + wshift), the tile adds lscale * sum to l
        const bool t8 = kF8 && j >= na;
        float c_t = sl2, shift = 0.f, wshift = -l2_ref, lscale = s_ref;
        if (t8) {
          // the producer's ring of tile scales (no global access here: an
          // ordinary load still in flight would hold up the next P arrival)
          const int sl = si % tc2::kScaleSlots;
          if (!wait_warp(bar(L::kScaleFull + sl), static_cast<uint32_t>(si / tc2::kScaleSlots) & 1u, ctl, 17))
            goto softmax_done;
          const float4 sc = ld_shared_f4(base + L::kScales + 16u * static_cast<uint32_t>(sl));
          __syncwarp();
          if (lane == 0) mbar_arrive(bar(L::kScaleEmpty + sl));
          ++si;
          c_t = fmaxf(c_row * sc.x, 1e-30f);
          // delta = log2(s_V / s_ref); an all-zero V tile (s_V = 0) takes delta = 0
          const bool nz = sc.y > 0.f;
          shift = nz ? sc.z - l2_ref : 0.f;
          wshift = 0.f;
          lscale = nz ? s_ref * sc.w : 1.f;  // 2^-delta
        }
        // S_j is ready and P buffer b is free once group G + j is complete
        if (!wait_group(G + j, 8)) goto softmax_done;
        tc_fence_after();
        const uint32_t t_s = tmem + lane_off + kColS + static_cast<uint32_t>(kBN) * b;
        // this thread's columns of S in s[]; with two halves, the other half's
        // maximum in m_other
        float s[kC];
        float m_other = -INFINITY;
        if constexpr (kH == 1) {
          uint32_t r[kC / 32][32];
#pragma unroll
          for (int k = 0; k < kC / 32; ++k) tmem_ld32(t_s + 32u * k, r[k]);
#pragma unroll
          for (int k = 0; k < kC / 32; ++k) tmem_wait_ld(r[k]);
#pragma unroll
          for (int k = 0; k < kC / 32; ++k)
#pragma unroll
            for (int c = 0; c < 32; ++c) s[32 * k + c] = __uint_as_float(r[k][c]);
          if (src.valid < kBN) {  // keys past the end of the range
#pragma unroll
            for (int c = 0; c < kC; ++c)
              if (c >= src.valid) s[c] = -INFINITY;
          }
        } else {
          // own 64 columns, and the other half's 64 for the maximum only
          const uint32_t other = static_cast<uint32_t>(kC - col0);
          uint32_t r0[32], r1[32], x0[32], x1[32];
          tmem_ld32(t_s + static_cast<uint32_t>(col0), r0);
          tmem_ld32(t_s + static_cast<uint32_t>(col0) + 32u, r1);
          tmem_ld32(t_s + other, x0);
          tmem_ld32(t_s + other + 32u, x1);
          tmem_wait_ld(r0);
          tmem_wait_ld(r1);
          tmem_wait_ld(x0);
          tmem_wait_ld(x1);
          float o[64];
#pragma unroll
          for (int c = 0; c < 32; ++c) {
            s[c] = __uint_as_float(r0[c]);
            s[32 + c] = __uint_as_float(r1[c]);
            o[c] = __uint_as_float(x0[c]);
            o[32 + c] = __uint_as_float(x1[c]);
          }
          if (src.valid < 128) {  // keys past the end of the range
#pragma unroll
            for (int c = 0; c < 64; ++c) {
              if (col0 + c >= src.valid) s[c] = -INFINITY;
              if (static_cast<int>(other) + c >= src.valid) o[c] = -INFINITY;
            }
          }
          float mx[2];
#pragma unroll
          for (int k = 0; k < 2; ++k) {
            mx[k] = fmax3(o[32 * k], o[32 * k + 1], o[32 * k + 2]);
#pragma unroll
            for (int c = 3; c < 31; c += 2) mx[k] = fmax3(mx[k], o[32 * k + c], o[32 * k + c + 1]);
            mx[k] = fmaxf(mx[k], o[32 * k + 31]);
          }
          m_other = fmaxf(mx[0], mx[1]);
        }
        // the row maximum of the raw scores: four independent chains of
        // 3-input max over this thread's columns (and the other half's maximum)
        auto row_max = [&]() -> float {
          constexpr int kChains = kC / 32;
          float mx[kChains];
#pragma unroll
          for (int k = 0; k < kChains; ++k) {
            mx[k] = fmax3(s[32 * k], s[32 * k + 1], s[32 * k + 2]);
#pragma unroll
            for (int c = 3; c < 31; c += 2) mx[k] = fmax3(mx[k], s[32 * k + c], s[32 * k + c + 1]);
            mx[k] = fmaxf(mx[k], s[32 * k + 31]);
          }
          if constexpr (kChains == 6)
            return fmax3(fmax3(mx[0], mx[1], mx[2]), fmax3(mx[3], mx[4], mx[5]), -INFINITY);
          else if constexpr (kChains == 4)
            return fmax3(mx[0], mx[1], fmaxf(mx[2], mx[3]));
          else
            return fmax3(mx[0], mx[1], m_other);
        };
        // rescale this row's O columns and l for a new running maximum m_new (O
        // must first hold P_j-1 V_j-1: group G + j + 1 complete)
        auto rescale = [&](float m_new) -> bool {
          if (!wait_group(G + j + 1, 9)) return false;
          tc_fence_after();
          const float alpha = ex2_approx(m_run - m_new);
          const f32x2 alpha2 = make_f32x2(alpha, alpha);
          m_run = m_new;
          l_run *= alpha;
          const uint32_t t_o = tmem + lane_off + kColO + static_cast<uint32_t>(ocol0);
#pragma unroll
          for (int cc = 0; cc < kOC / 16; ++cc) {
            uint32_t o[16];
            tmem_ld16(t_o + 16u * cc, o);
            tmem_wait_ld(o);
#pragma unroll
            for (int c = 0; c < 16; c += 2) {
              f32x2 v = mul_f32x2(make_f32x2(__uint_as_float(o[c]), __uint_as_float(o[c + 1])), alpha2);
              float lo, hi;
              split_f32x2(v, lo, hi);
              o[c] = __float_as_uint(lo);
              o[c + 1] = __float_as_uint(hi);
            }
            tmem_st16(t_o + 16u * cc, o);
          }
          return true;
        };
        // P = exp2(c * S + shift - m) into P buffer b: bf16 pairs (32 keys = 16
        // columns at a time), or for a cached tile E4M3 quads (32 keys = 8
        // columns); returns this thread's sum of the weights written
        const uint32_t t_p = tmem + lane_off + kColP + kPStride * b;
        auto write_p = [&]() -> float {
          const float bias = (kF8 ? shift + wshift : 0.f) - m_run;
          const f32x2 negm = make_f32x2(bias, bias);
          const f32x2 c2 = kF8 ? make_f32x2(c_t, c_t) : sl2x2;
          f32x2 lacc[4];
#pragma unroll
          for (int i = 0; i < 4; ++i) lacc[i] = make_f32x2(0.f, 0.f);
          if (t8) {
#pragma unroll
            for (int k = 0; k < kC / 32; ++k) {
              uint32_t pk[8];
#pragma unroll
              for (int c = 0; c < 8; ++c) {
                const f32x2 e01 = fma_f32x2(make_f32x2(s[32 * k + 4 * c], s[32 * k + 4 * c + 1]), c2, negm);
                const f32x2 e23 = fma_f32x2(make_f32x2(s[32 * k + 4 * c + 2], s[32 * k + 4 * c + 3]), c2, negm);
                float e0, e1, e2, e3;
                split_f32x2(e01, e0, e1);
                split_f32x2(e23, e2, e3);
                const float x0 = ex2_approx(e0), x1 = ex2_approx(e1), x2 = ex2_approx(e2), x3 = ex2_approx(e3);
                lacc[(2 * c) & 3] = add_f32x2(lacc[(2 * c) & 3], make_f32x2(x0, x1));
                lacc[(2 * c + 1) & 3] = add_f32x2(lacc[(2 * c + 1) & 3], make_f32x2(x2, x3));
                pk[c] = pack_e4m3x4(x0, x1, x2, x3);
              }
              tmem_st8(t_p + static_cast<uint32_t>(col0 / 4) + 8u * k, pk);
            }
          } else {
#pragma unroll
            for (int k = 0; k < kC / 32; ++k) {
              uint32_t pk[16];
#pragma unroll
              for (int c = 0; c < 16; ++c) {
                const f32x2 e = fma_f32x2(make_f32x2(s[32 * k + 2 * c], s[32 * k + 2 * c + 1]), c2, negm);
                float e0, e1;
                split_f32x2(e, e0, e1);
                const float x = ex2_approx(e0), y = ex2_approx(e1);
                lacc[c & 3] = add_f32x2(lacc[c & 3], make_f32x2(x, y));
                pk[c] = pack_bf16x2(x, y);
              }
              tmem_st16(t_p + static_cast<uint32_t>(col0 / 2) + 16u * k, pk);
            }
          }
          const f32x2 l2 = add_f32x2(add_f32x2(lacc[0], lacc[1]), add_f32x2(lacc[2], lacc[3]));
          float lo, hi;
          split_f32x2(l2, lo, hi);
          return lo + hi;
        };
        // running maximum from the row maximum (lazy: moves only when a tile's
        // maximum exceeds it by more than 2^8)
        const float m_tile = fmaf(row_max(), c_t, shift);
        if (j == 0) {
          m_run = m_tile;
        } else if (__any_sync(0xffffffffu, m_tile > m_run + 8.0f)) {
          if (!rescale(fmaxf(m_run, m_tile))) goto softmax_done;
        }
        const float l_tile = write_p();
        l_run += kF8 ? l_tile * lscale : l_tile;
        // the MMA thread waits only for P: the leader's warp 0 first makes
        // sure that the stage of P_j V_j's group (G + j + 2) has landed
        if (leader && warp == 0 &&
            !wait_warp(bar(L::kStageFull + stage_of(G + j + 2)), stage_parity(G + j + 2), ctl, 13))
          goto softmax_done;
        tmem_wait_st();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive_cluster(mapa_shared(bar(L::kPFull + b), 0));
      }
      {
        // the row's place: the bf16 kernels read it again from the work list, so
        // that it is not kept live through the tile loop
        bool e_row_ok = row_ok;
        int64_t e_grow = grow;
        __nv_bfloat16* e_orow = orow;
        int e_head = head, e_part = tk.part;
        if constexpr (!kF8) {
          Task et;
          decode_item(args, item, et, e_head);
          e_row_ok = prow < et.q_rows;
          e_grow = static_cast<int64_t>(et.q_row0) + prow;
          e_orow = args.out + e_grow * args.row_stride + static_cast<int64_t>(e_head) * DG + ocol0;
          e_part = et.part;
        }
        if (!wait_group(G + nkv + 1, 10)) goto softmax_done;  // the item's last group
        tc_fence_after();
        float l_tot = l_run;
        if constexpr (kH == 2) {
          // the two halves' partial row sums (relative to the same maximum)
          lx[hh * 128 + trow] = l_run;
          __syncwarp();
          if (lane == 0) mbar_arrive(bar(L::kLXFull));
          if (!wait_warp(bar(L::kLXFull), static_cast<uint32_t>(n_lx) & 1u, ctl, 15)) goto softmax_done;
          ++n_lx;
          l_tot = l_run + lx[(1 - hh) * 128 + trow];
        }
        const float inv_l = kF8 ? s_ref / l_tot : 1.0f / l_tot;
        const uint32_t t_o = tmem + lane_off + kColO + static_cast<uint32_t>(ocol0);
        if (e_part > 0) {
          // a part of a split item: O / l in fp32 and m + log l to its workspace slot
          const int64_t prow_ws = static_cast<int64_t>(e_part - 1) * args.rows_per_task + prow;
          float4* dst = reinterpret_cast<float4*>(args.part_o + prow_ws * DG + ocol0);
#pragma unroll
          for (int cc = 0; cc < kOC / 32; ++cc) {
            uint32_t o[32];
            tmem_ld32(t_o + 32u * cc, o);
            tmem_wait_ld(o);
            if (e_row_ok) {
#pragma unroll
              for (int c = 0; c < 8; ++c)
                dst[8 * cc + c] = make_float4(__uint_as_float(o[4 * c]) * inv_l, __uint_as_float(o[4 * c + 1]) * inv_l,
                                              __uint_as_float(o[4 * c + 2]) * inv_l,
                                              __uint_as_float(o[4 * c + 3]) * inv_l);
            }
          }
          tc_fence_before();
          if (e_row_ok && hh == 0) args.part_lse[prow_ws] = (m_run + log2f(l_tot)) * 0.69314718055994530942f;
          G += nkv + 2;
          continue;
        }
        uint32_t packed[kOC / 2];
#pragma unroll
        for (int cc = 0; cc < kOC / 32; ++cc) {
          uint32_t o[32];
          tmem_ld32(t_o + 32u * cc, o);
          tmem_wait_ld(o);
#pragma unroll
          for (int c = 0; c < 16; ++c)
            packed[16 * cc + c] =
                pack_bf16x2(__uint_as_float(o[2 * c]) * inv_l, __uint_as_float(o[2 * c + 1]) * inv_l);
        }
        // (the next arrival on p_full, after the next tile's P, tells the MMA
        // thread that these O reads are done)
        tc_fence_before();
        if (e_row_ok) {
          uint4* dst = reinterpret_cast<uint4*>(e_orow);
#pragma unroll
          for (int c = 0; c < kOC / 8; ++c)
            dst[c] = make_uint4(packed[4 * c], packed[4 * c + 1], packed[4 * c + 2], packed[4 * c + 3]);
          if (args.lse && hh == 0)
            args.lse[e_grow * args.num_heads + e_head] = (m_run + log2f(l_tot)) * 0.69314718055994530942f;
        }
      }
      G += nkv + 2;
    }
  softmax_done:;
  }

  tc_fence_before();
  __syncthreads();
  // the pair's MMAs and TMEM reads are over in both CTAs, and both producers'
  // load records are in the leader's shared memory
  cluster_sync();
  if (warp == Cfg::kMmaWarp) {
    tc_fence_after();
    tmem_dealloc_pair(tmem, kTmemCols);
  }
  if (leader && warp == Cfg::kProducerWarp && lane == 0) {
    // Every stage and Q load of either CTA must land before that CTA exits.
    // The leader arms a phase for both halves before it issues its own, and
    // each CTA issues its half after the same wait; after an abort the two can
    // differ by one phase.  A phase the follower loaded but the leader never
    // armed is armed now for the follower's bytes; a phase the leader armed
    // whose follower half was never issued has those bytes counted as
    // arrived.  Then the last phase of every barrier is drained (bounded).
    const volatile uint32_t* rec = reinterpret_cast<const volatile uint32_t*>(base_ptr + L::kLoadRec);
    const volatile uint32_t* peer = rec + L::kRecWords;
    // missing: the follower's bytes of the leader's last phase; loaded: the
    // follower's own bytes of its last load
    auto settle = [&](uint32_t b, int mine, int theirs, uint32_t missing, uint32_t loaded) {
      if (theirs == mine + 1) {
        mbar_arrive_expect_tx(b, loaded);
        mine = theirs;
      } else if (mine == theirs + 1 && missing > 0) {
        mbar_complete_tx(b, missing);
      }
      if (mine > 0) drain_one(b, static_cast<uint32_t>(mine - 1) & 1u, args.timeout_ns);
    };
    for (int s = 0; s < kStages; ++s)
      settle(bar(L::kStageFull + s), static_cast<int>(rec[s]), static_cast<int>(peer[s]), rec[2 * kStages + s],
             peer[kStages + s]);
    constexpr uint32_t kQCta = kQBoxes * kBoxBytes;  // each CTA's bytes of a Q load
    for (int b = 0; b < 2; ++b)
      settle(bar(L::kQFull + b), static_cast<int>(rec[3 * kStages + b]), static_cast<int>(peer[3 * kStages + b]),
             kQCta, kQCta);
  }
  // the follower leaves only once the leader has seen every load of the pair land
  cluster_sync();
  if (dyn && leader && threadIdx.x == 0) tc2::work_done(args.work, n_clusters);
}

}  // namespace rc
