// common.cuh -- work description shared by the attention kernels.
//
// One task is a run of at most 256 consecutive query rows that all see the
// same keys: a key range A in one K/V pair and an optional key range B in a
// second K/V pair.  The joint masks of the paper reduce to such tasks
// (Sec. 3.3, App. C):
//   step (live rows [LT; X_t])     A = the request's live rows, B = its cached rows
//   prefill (rows [ST; R])         A = the request's [ST; R] rows (anchor rows
//                                  of the alternative reading: A = [ST] only)
//   full (rows [LT; X_t; R])       A = the request's whole sequence
// so the mask is never materialised: a key is visible exactly when it lies in
// A or B, and keys past the end of a range are cut off inside the last tile.
// A launch enumerates items = tasks x heads, item i -> task i / H, head i % H.
#pragma once
#include <cstdint>
#include <cuda_bf16.h>

namespace rc {

struct Task {
  int32_t q_row0;  // first query row (row of the Q/O tensors)
  int32_t q_rows;  // rows in this task, 1..rows_per_task (128 or 256)
  int32_t a_row0;  // key range A: first row in the A tensors
  int32_t a_len;   //              length
  int32_t b_row0;  // key range B (in the B tensors)
  int32_t b_len;   //              length, 0 = none
  int32_t pad0, pad1;
};
static_assert(sizeof(Task) == 32, "Task layout is part of the device work list");

struct AttnArgs {
  const Task* tasks;
  int32_t n_tasks;
  int32_t num_heads;
  int32_t n_items;
  int32_t dbg_skip_first_load;  // tcgen05 kernel: producer skips its first K load
  __nv_bfloat16* out;           // [rows, H, D]
  float* lse;                   // [rows, H] or null
  int64_t row_stride;           // elements between rows of Q/K/V/O (= H * D)
  float scale_log2;             // softmax_scale * log2(e)
  int32_t rows_per_task;        // 128 or 256 (the mma.sync kernel splits tasks into 64-row CTAs)
  uint64_t timeout_ns;          // bound of every in-kernel wait
  // raw pointers, used by the mma.sync kernel (the tcgen05 kernel reads
  // through tensor maps)
  const __nv_bfloat16* q;
  const __nv_bfloat16* ka;
  const __nv_bfloat16* va;
  const __nv_bfloat16* kb;
  const __nv_bfloat16* vb;
};

// Device error word (one per device that loads the library); kernels set it
// when a bounded wait runs out, refcache_status() reads and clears it.
#define RC_DEV_TIMEOUT_BASE 0x1000
__device__ int g_rc_status;

}  // namespace rc
