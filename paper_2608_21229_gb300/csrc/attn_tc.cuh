// attn_tc.cuh -- pieces shared by the tcgen05 attention kernel
// (attn_tc2.cuh): bounded mbarrier waits that report a timeout instead of
// hanging, and the decoding of work items.
//
// Every wait is bounded (AttnArgs::timeout_ns).  A wait that runs out sets
// the device error word (and the launching cache's own word) and a CTA-wide
// abort flag; every role then leaves its loop, the producer waits (bounded)
// for its TMA loads in flight, the MMA thread for its MMAs in flight, and
// tensor memory is freed before exit.
#pragma once
#include <cuda.h>
#include <cuda_bf16.h>

#include "common.cuh"
#include "ptx.cuh"

namespace rc {

namespace tc {
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kBoxBytes = 128 * 128;  // one TMA box: 128 rows x 128 bytes

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

// A key tile of an item: where it starts in its tensor and how many of its
// keys are inside the item's key range.
struct TileSrc {
  int row;    // first key row of the tile in its tensor
  int valid;  // keys of the tile inside the range
  bool in_b;  // tile comes from the B tensors
};

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

}  // namespace tc

}  // namespace rc
