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
// A launch enumerates items = tasks x heads, item i -> head i / n_tasks, task
// i % n_tasks; or, when AttnArgs::per_item is set, an explicit list with one
// task per item that names its head.  Such a list can also hold *parts* of an
// item (a sub-range of its key tiles): a part writes its normalised output and
// log-sum-exp to a workspace slot, and a combine kernel merges the parts.
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
  int32_t head;    // per-item lists only: the item's head
  int32_t part;    // per-item lists only: 0 = write O, p > 0 = partial result to workspace slot p - 1
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
  int32_t per_item;             // tasks is a per-item list (Task::head, Task::part used)
  float* part_o;                // workspace of partial results: [slot][rows_per_task][D] fp32, O / l
  float* part_lse;              //                               [slot][rows_per_task] fp32, m + log l
  uint64_t timeout_ns;          // bound of every in-kernel wait
  const float4* b_scales;       // E4M3 key range B: (s_K, s_V, log2 s_V, 1/s_V) per (128-row tile, head), tile-major
  // raw pointers, used by the mma.sync kernel (the tcgen05 kernel reads
  // through tensor maps)
  const __nv_bfloat16* q;
  const __nv_bfloat16* ka;
  const __nv_bfloat16* va;
  const __nv_bfloat16* kb;
  const __nv_bfloat16* vb;
  int* status;  // the launching cache's own error word (null: the device word only)
  // CTA-pair kernel: null = static order (cluster c takes items c, c + n, ...);
  // else [next item, clusters done], zero at launch: items are taken in list
  // order by whichever cluster is free, and the last cluster to finish resets
  // both words
  int* work;
};

// One item whose key range was split into parts: the combine kernel merges
// parts [part0, part0 + nparts) of the workspace into rows [q_row0, q_row0 +
// q_rows) of `head`.
struct CombineJob {
  int32_t q_row0, q_rows, head, part0, nparts, pad0, pad1, pad2;
};
static_assert(sizeof(CombineJob) == 32, "CombineJob layout is part of the device work list");

// Device error word (one per device that loads the library); kernels set it
// when a bounded wait runs out, refcache_status() reads and clears it.  A
// launch made for a cache also sets that cache's own word (AttnArgs::status),
// which refcache_cache_status() reads and clears.
#define RC_DEV_TIMEOUT_BASE 0x1000
__device__ int g_rc_status;

}  // namespace rc
