// refcache.cu -- the C ABI declared in include/refcache.h: argument checks,
// the per-request work tables, the persistent per-layer K/V cache (bf16, or
// E4M3 with REFCACHE_CACHE_FP8), TMA tensor maps and the kernel launches.  All
// compute runs in the kernels of attn_tc2.cuh (the tcgen05 kernel on CTA
// pairs, both head dims; attn_tc.cuh holds its bounded waits), attn_mma.cuh
// (the mma.sync comparison kernel and the cache copy), attn_combine.cuh (merge
// of split items) and cache_fp8.cuh (the E4M3 cache write).
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <functional>
#include <mutex>
#include <string>
#include <vector>

#include "refcache.h"
#include "attn_mma.cuh"
#include "attn_tc.cuh"
#include "attn_tc2.cuh"
#include "attn_combine.cuh"
#include "cache_fp8.cuh"
#include "mufu_rate.cuh"

using rc::AttnArgs;
using rc::CombineJob;
using rc::CopySeg;
using rc::QuantTile;
using rc::Task;

namespace {

thread_local std::string g_last_error;
std::atomic<int> g_kernel{REFCACHE_KERNEL_TCGEN05};
std::atomic<uint64_t> g_timeout_ns{1000000000ull};
std::atomic<int> g_dbg_skip{0};

int fail(int code, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return code;
}

int cuda_fail(cudaError_t e, const char* what) {
  return fail(REFCACHE_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

constexpr int kMaxDevices = 64;
constexpr int kWorkOffset = 32;  // ints from a cache's error word to its work counter (a line of its own)

struct DeviceInfo {
  bool checked = false;
  bool ok = false;
  int num_sms = 0;
  bool attr_set[9] = {false, false, false, false, false, false, false, false, false};
  int max_clusters[5] = {0, 0, 0, 0, 0};  // CTA pairs of each attn_tc2_kernel variant that fit at once
};
DeviceInfo g_dev[kMaxDevices];
std::mutex g_dev_mu;

// The kernels are built for sm_103a only: require a compute capability 10.3 device.
int current_device(int* dev_out, DeviceInfo** info) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  if (dev < 0 || dev >= kMaxDevices) return fail(REFCACHE_ERR_UNSUPPORTED, "device index %d", dev);
  std::lock_guard<std::mutex> lk(g_dev_mu);
  DeviceInfo& d = g_dev[dev];
  if (!d.checked) {
    int major = 0, minor = 0, sms = 0;
    if ((e = cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev)) != cudaSuccess ||
        (e = cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev)) != cudaSuccess ||
        (e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
      return cuda_fail(e, "cudaDeviceGetAttribute");
    d.checked = true;
    d.ok = (major == 10 && minor == 3);
    d.num_sms = sms;
    if (!d.ok) {
      d.checked = false;
      return fail(REFCACHE_ERR_UNSUPPORTED, "device %d is sm_%d%d; this library is built for sm_103a", dev,
                  major, minor);
    }
  }
  *dev_out = dev;
  *info = &d;
  return REFCACHE_OK;
}

// ---------------------------------------------------------------- tensor maps
using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                   const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

// THD bf16 tensor [rows, H, D] seen as a 2-D array (H*D columns, rows rows);
// box = 64 columns (128 bytes) x box_rows rows with the 128-byte swizzle.
int make_tmap(CUtensorMap* m, const void* base, int64_t rows, int H, int D, uint32_t box_rows = 128) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return fail(REFCACHE_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable");
  const cuuint64_t dims[2] = {static_cast<cuuint64_t>(H) * D, static_cast<cuuint64_t>(std::max<int64_t>(rows, 1))};
  const cuuint64_t strides[1] = {static_cast<cuuint64_t>(H) * D * 2};
  const cuuint32_t box[2] = {64, box_rows};
  const cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(REFCACHE_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", static_cast<int>(r));
  return REFCACHE_OK;
}

// Byte matrix (E4M3 codes) of `outer` rows x `inner` bytes, row pitch `inner`;
// box = 128 bytes x 64 rows with the 128-byte swizzle.
int make_tmap_u8(CUtensorMap* m, const void* base, int64_t inner, int64_t outer) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return fail(REFCACHE_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable");
  const cuuint64_t dims[2] = {static_cast<cuuint64_t>(inner), static_cast<cuuint64_t>(std::max<int64_t>(outer, 1))};
  const cuuint64_t strides[1] = {static_cast<cuuint64_t>(inner)};
  const cuuint32_t box[2] = {128, 64};
  const cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(REFCACHE_ERR_CUDA, "cuTensorMapEncodeTiled (u8) failed (%d)", static_cast<int>(r));
  return REFCACHE_OK;
}

// ---------------------------------------------------------------- work lists
// Query rows per task: one M = 256 MMA of a CTA pair (both head dims).
int task_rows(int) { return 256; }

void add_rows(std::vector<Task>& v, int rows_per_task, int q0, int qn, int a0, int an, int b0, int bn) {
  for (int r = 0; r < qn; r += rows_per_task) {
    Task t{};
    t.q_row0 = q0 + r;
    t.q_rows = std::min(rows_per_task, qn - r);
    t.a_row0 = a0;
    t.a_len = an;
    t.b_row0 = b0;
    t.b_len = bn;
    v.push_back(t);
  }
}

int64_t task_cost(const Task& t) {
  return static_cast<int64_t>((t.q_rows + 127) / 128) * ((t.a_len + 127) / 128 + (t.b_len + 127) / 128);
}

// Longest tasks first: the order in which the persistent CTAs take items.
void order_tasks(std::vector<Task>& v) {
  std::stable_sort(v.begin(), v.end(), [](const Task& x, const Task& y) { return task_cost(x) > task_cost(y); });
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

int check_dims(int batch, int H, int D) {
  if (batch < 1) return fail(REFCACHE_ERR_INVALID_ARG, "batch must be >= 1 (got %d)", batch);
  if (H < 1) return fail(REFCACHE_ERR_INVALID_ARG, "num_heads must be >= 1 (got %d)", H);
  if (D != 64 && D != 128) return fail(REFCACHE_ERR_UNSUPPORTED, "head_dim must be 64 or 128 (got %d)", D);
  if (static_cast<int64_t>(H) * D > (1 << 20)) return fail(REFCACHE_ERR_INVALID_ARG, "num_heads too large");
  return REFCACHE_OK;
}

int check_cu(const int32_t* cu, int batch, const char* name, int64_t max_rows) {
  if (!cu) return fail(REFCACHE_ERR_INVALID_ARG, "%s is NULL", name);
  if (cu[0] != 0) return fail(REFCACHE_ERR_INVALID_ARG, "%s[0] must be 0", name);
  for (int b = 0; b < batch; ++b)
    if (cu[b + 1] < cu[b]) return fail(REFCACHE_ERR_INVALID_ARG, "%s must be non-decreasing (at %d)", name, b);
  if (cu[batch] > max_rows) return fail(REFCACHE_ERR_INVALID_ARG, "%s total rows too large", name);
  return REFCACHE_OK;
}

int check_scale(float s) {
  if (!(s > 0.f) || !std::isfinite(s)) return fail(REFCACHE_ERR_INVALID_ARG, "softmax_scale must be finite and > 0");
  return REFCACHE_OK;
}

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// ---------------------------------------------------------------- launches
// Keys per tile of the pair kernel: 192 for the bf16 cache
// (REFCACHE_KERNEL_TCGEN05), 128 for the E4M3 cache and for
// REFCACHE_KERNEL_TCGEN05_K128.
int tc2_tile(bool f8) { return f8 || g_kernel.load() == REFCACHE_KERNEL_TCGEN05_K128 ? 128 : 192; }

// CTA pairs of the pair kernel (bf16 key range B, or E4M3 with kF8; kBN keys
// per tile; head dim kDG) that run at once on this device (the persistent
// grid); sets the kernel's shared-memory attribute on first use.
template <bool kF8, int kBN, int kDG>
int tc2_clusters(DeviceInfo* info, int* clusters_out) {
  constexpr uint32_t smem = rc::tc2::SmemT<kF8, kBN>::kDynamic;
  const int variant = kF8 ? 1 : kDG == 128 ? (kBN == 128 ? 0 : 2) : (kBN == 128 ? 3 : 4);
  const int key = 4 + variant;
  if (!info->attr_set[key]) {
    cudaError_t e =
        cudaFuncSetAttribute(rc::attn_tc2_kernel<kF8, kBN, kDG>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute(attn_tc2_kernel)");
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(2 * static_cast<unsigned>(info->num_sms / 2), 1, 1);
    cfg.blockDim = dim3(rc::tc2::Cfg<kF8, kBN>::kThreads, 1, 1);
    cfg.dynamicSmemBytes = smem;
    int clusters = 0;
    e = cudaOccupancyMaxActiveClusters(&clusters, rc::attn_tc2_kernel<kF8, kBN, kDG>, &cfg);
    if (e != cudaSuccess || clusters < 1) clusters = info->num_sms / 2;
    info->max_clusters[variant] = clusters;
    info->attr_set[key] = true;
  }
  *clusters_out = info->max_clusters[variant];
  return REFCACHE_OK;
}

// The CTA-pair kernel: grid = 2 x the clusters that fit at once.
template <bool kF8, int kBN, int kDG>
int launch_tc2(const CUtensorMap (&maps)[5], const AttnArgs& a, DeviceInfo* info, cudaStream_t s) {
  constexpr uint32_t smem = rc::tc2::SmemT<kF8, kBN>::kDynamic;
  int max_clusters = 0;
  int rc = tc2_clusters<kF8, kBN, kDG>(info, &max_clusters);
  if (rc) return rc;
  const int clusters = std::min(a.n_items, max_clusters);
  // a programmatic dependent of the stream's previous kernel: its prologue
  // (barriers, tensor memory) overlaps that kernel's tail
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(2 * static_cast<unsigned>(clusters), 1, 1);
  cfg.blockDim = dim3(rc::tc2::Cfg<kF8, kBN>::kThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaError_t e =
      cudaLaunchKernelEx(&cfg, rc::attn_tc2_kernel<kF8, kBN, kDG>, maps[0], maps[1], maps[2], maps[3], maps[4], a);
  if (e == cudaSuccess) e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "attn_tc2_kernel launch");
  return REFCACHE_OK;
}

template <int D>
int launch_mma(const AttnArgs& a, DeviceInfo* info, cudaStream_t s) {
  constexpr int smem = 5 * 64 * D * 2;
  const int key = D == 64 ? 2 : 3;
  if (!info->attr_set[key]) {
    cudaError_t e = cudaFuncSetAttribute(rc::attn_mma_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute(attn_mma_kernel)");
    info->attr_set[key] = true;
  }
  rc::attn_mma_kernel<D><<<a.n_items * (a.rows_per_task / 64), 128, smem, s>>>(a);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "attn_mma_kernel launch");
  return REFCACHE_OK;
}

struct Operands {
  const void* q;
  int64_t q_rows;
  const void *ka, *va;
  int64_t a_rows;
  const void *kb, *vb;
  int64_t b_rows;
  void* o;
  float* lse;
  int* status = nullptr;  // the cache's own error word, if the launch is for a cache
  int* work = nullptr;    // work counter of the CTA-pair kernel (two ints, zero between launches), or null
};

// Key range B as an E4M3 cache (cache_fp8.cuh): codes of K [rows_pad, H, 128],
// of V transposed [H, 128, rows_pad], and the scales of every tile and head.
struct Fp8B {
  const void* k8 = nullptr;
  const void* vt8 = nullptr;
  const float4* scales = nullptr;
  int64_t rows_pad = 0;
};

// A per-item work list with split items (tcgen05 kernel only):
// the items, the combine jobs of the split ones and their workspace.
struct ItemList {
  const Task* items = nullptr;
  int n_items = 0;
  const CombineJob* jobs = nullptr;
  int n_jobs = 0;
  float* part_o = nullptr;
  float* part_lse = nullptr;
};

// The build's cache write: copy_rows_kernel over the request segments.
struct CopyJob {
  const CopySeg* segs = nullptr;
  int n_segs = 0;
  const void *src_k = nullptr, *src_v = nullptr;
  void *dst_k = nullptr, *dst_v = nullptr;
  int row_u4 = 0;
  int64_t rows = 0;
};

// `beside`: launched as a programmatic dependent of the kernel before it, so
// that it runs next to that kernel (its grid is kept to two CTAs per SM, which
// fit beside the attention kernel's CTAs).
int launch_copy(const CopyJob& c, const DeviceInfo* info, cudaStream_t s, bool beside) {
  const int64_t per_seg = beside ? std::max(1, 2 * info->num_sms / c.n_segs) : 1024;
  dim3 grid(static_cast<unsigned>(std::min<int64_t>(per_seg, (c.rows * c.row_u4 + 255) / 256 / c.n_segs + 1)),
            static_cast<unsigned>(c.n_segs));
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = grid;
  cfg.blockDim = dim3(256, 1, 1);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = beside ? 1 : 0;
  cudaError_t e = cudaLaunchKernelEx(&cfg, rc::copy_rows_kernel, c.segs, static_cast<const uint4*>(c.src_k),
                                     static_cast<const uint4*>(c.src_v), static_cast<uint4*>(c.dst_k),
                                     static_cast<uint4*>(c.dst_v), c.row_u4);
  if (e == cudaSuccess) e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "copy_rows_kernel launch");
  return REFCACHE_OK;
}

// `copy` (the build's cache write, if any) runs beside the pair kernel,
// launched right after it; with the mma.sync kernel it goes first.
int run_attention(const Task* d_tasks, int n_tasks, int H, int D, const Operands& op, float scale, DeviceInfo* info,
                  cudaStream_t s, const ItemList* il = nullptr, const Fp8B* f8 = nullptr,
                  const CopyJob* copy = nullptr) {
  if (n_tasks == 0) return copy ? launch_copy(*copy, info, s, false) : REFCACHE_OK;
  AttnArgs a{};
  a.tasks = d_tasks;
  a.n_tasks = n_tasks;
  a.num_heads = H;
  a.n_items = n_tasks * H;
  a.out = static_cast<__nv_bfloat16*>(op.o);
  a.lse = op.lse;
  a.row_stride = static_cast<int64_t>(H) * D;
  a.scale_log2 = static_cast<float>(static_cast<double>(scale) * 1.4426950408889634074);
  a.rows_per_task = task_rows(D);
  a.timeout_ns = g_timeout_ns.load();
  a.status = op.status;
  a.work = op.work;
  a.q = static_cast<const __nv_bfloat16*>(op.q);
  a.ka = static_cast<const __nv_bfloat16*>(op.ka);
  a.va = static_cast<const __nv_bfloat16*>(op.va);
  a.kb = static_cast<const __nv_bfloat16*>(op.kb ? op.kb : op.ka);
  a.vb = static_cast<const __nv_bfloat16*>(op.vb ? op.vb : op.va);
  if (static_cast<int64_t>(n_tasks) * H > (1ll << 30)) return fail(REFCACHE_ERR_INVALID_ARG, "too many work items");
  if (g_kernel.load() == REFCACHE_KERNEL_MMA_SYNC) {
    if (f8) return fail(REFCACHE_ERR_UNSUPPORTED, "the E4M3 cache runs on the tcgen05 kernel only");
    int rc = copy ? launch_copy(*copy, info, s, false) : REFCACHE_OK;
    if (rc) return rc;
    return D == 64 ? launch_mma<64>(a, info, s) : launch_mma<128>(a, info, s);
  }
  // Key tiles of the CTA-pair kernel: each CTA loads half of a K tile (boxes
  // of tile / 2 rows, one per 64 head-dim columns) and a V box of the whole
  // tile.
  const uint32_t tile = static_cast<uint32_t>(tc2_tile(f8 != nullptr));
  const uint32_t k_rows = tile / 2, v_rows = tile;
  CUtensorMap maps[5];
  int rc;
  if ((rc = make_tmap(&maps[0], op.q, op.q_rows, H, D)) != 0) return rc;
  if ((rc = make_tmap(&maps[1], op.ka, op.a_rows, H, D, k_rows)) != 0) return rc;
  if ((rc = make_tmap(&maps[2], op.va, op.a_rows, H, D, v_rows)) != 0) return rc;
  if (f8) {
    if ((rc = make_tmap_u8(&maps[3], f8->k8, static_cast<int64_t>(H) * D, f8->rows_pad)) != 0) return rc;
    if ((rc = make_tmap_u8(&maps[4], f8->vt8, f8->rows_pad, static_cast<int64_t>(H) * D)) != 0) return rc;
    a.b_scales = f8->scales;
  } else if (op.kb && op.b_rows > 0) {
    if ((rc = make_tmap(&maps[3], op.kb, op.b_rows, H, D, k_rows)) != 0) return rc;
    if ((rc = make_tmap(&maps[4], op.vb, op.b_rows, H, D, v_rows)) != 0) return rc;
  } else {
    maps[3] = maps[1];
    maps[4] = maps[2];
  }
  a.dbg_skip_first_load = g_dbg_skip.exchange(0);
  if (il && il->items) {
    a.tasks = il->items;
    a.per_item = 1;
    a.n_items = il->n_items;
    a.part_o = il->part_o;
    a.part_lse = il->part_lse;
  }
  if (f8)
    rc = launch_tc2<true, 128, 128>(maps, a, info, s);
  else if (D == 128)
    rc = tile == 128 ? launch_tc2<false, 128, 128>(maps, a, info, s) : launch_tc2<false, 192, 128>(maps, a, info, s);
  else
    rc = tile == 128 ? launch_tc2<false, 128, 64>(maps, a, info, s) : launch_tc2<false, 192, 64>(maps, a, info, s);
  if (rc) return rc;
  if (copy && (rc = launch_copy(*copy, info, s, true)) != 0) return rc;
  if (il && il->n_jobs > 0) {
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(static_cast<unsigned>((a.rows_per_task + 7) / 8), static_cast<unsigned>(il->n_jobs));
    cfg.blockDim = dim3(256, 1, 1);
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;  // its CTAs wait for the attention kernel
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    const float* po = static_cast<const float*>(il->part_o);
    const float* pl = static_cast<const float*>(il->part_lse);
    cudaError_t e = D == 128 ? cudaLaunchKernelEx(&cfg, rc::combine_parts_kernel<128>, il->jobs, po, pl, a.rows_per_task,
                                                  a.out, a.lse, a.row_stride, H)
                             : cudaLaunchKernelEx(&cfg, rc::combine_parts_kernel<64>, il->jobs, po, pl, a.rows_per_task,
                                                  a.out, a.lse, a.row_stride, H);
    if (e == cudaSuccess) e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_fail(e, "combine_parts_kernel launch");
  }
  return REFCACHE_OK;
}

// Per-item list of `tasks` x heads (head-major, as the kernels enumerate
// items) for `clusters` CTA pairs.  When the items do not fill the last round
// of the persistent grid, the items of that round are split by key tiles into
// s parts each (s chosen so that the parts fill the clusters best), which run
// after the whole items; their results are merged by combine jobs.
void plan_items(const std::vector<Task>& tasks, int H, int clusters, int tile, std::vector<Task>* items,
                std::vector<CombineJob>* jobs, int* n_parts) {
  items->clear();
  jobs->clear();
  *n_parts = 0;
  const int64_t n = static_cast<int64_t>(tasks.size()) * H;
  if (n == 0 || clusters < 1) return;
  const int64_t rem = n % clusters;
  int best_s = 1;
  double best = 1.0;  // item-times the last round costs
  if (rem > 0) {
    for (int cand : {2, 3, 4, 6, 8}) {
      const double cost = static_cast<double>((rem * cand + clusters - 1) / clusters) / cand;
      if (cost < best - 1e-9) {
        best = cost;
        best_s = cand;
      }
    }
  }
  const int64_t n_whole = rem > 0 && best_s > 1 ? n - rem : n;
  std::vector<Task> parts;
  for (int64_t i = 0; i < n; ++i) {
    const int h = static_cast<int>(i / static_cast<int64_t>(tasks.size()));
    Task t = tasks[static_cast<size_t>(i % static_cast<int64_t>(tasks.size()))];
    t.head = h;
    t.part = 0;
    const int na = (t.a_len + tile - 1) / tile, nb = (t.b_len + tile - 1) / tile, nkv = na + nb;
    const int s_here = std::min(best_s, nkv / 4);  // parts of at least four key tiles
    if (i < n_whole || s_here < 2) {
      items->push_back(t);
      continue;
    }
    CombineJob job{};
    job.q_row0 = t.q_row0;
    job.q_rows = t.q_rows;
    job.head = h;
    job.part0 = *n_parts;
    job.nparts = s_here;
    for (int k = 0; k < s_here; ++k) {
      const int j0 = static_cast<int>(static_cast<int64_t>(nkv) * k / s_here);
      const int j1 = static_cast<int>(static_cast<int64_t>(nkv) * (k + 1) / s_here);
      Task p = t;
      // tiles [j0, j1) of the item's key list (range A, then range B)
      const int a0 = std::min(j0, na), a1 = std::min(j1, na);
      p.a_row0 = t.a_row0 + tile * a0;
      p.a_len = a1 > a0 ? std::min(t.a_len - tile * a0, tile * (a1 - a0)) : 0;
      const int b0 = std::max(j0, na) - na, b1 = std::max(j1, na) - na;
      p.b_row0 = t.b_row0 + tile * b0;
      p.b_len = b1 > b0 ? std::min(t.b_len - tile * b0, tile * (b1 - b0)) : 0;
      p.part = ++*n_parts;
      parts.push_back(p);
    }
    jobs->push_back(job);
  }
  items->insert(items->end(), parts.begin(), parts.end());
}

// Orders a per-item list for the CTA-pair kernel, which hands items out in
// list order to whichever CTA pair is free (a work counter): longest items
// first (MMA groups: key tiles + 2), items of equal length in their order
// (head-major, so that the pairs running at the same time share few heads'
// K/V tiles in L2).  Only the order changes, not any item's arithmetic.
std::vector<Task> longest_first(std::vector<Task> items, int tile) {
  auto groups = [&](const Task& t) -> int64_t {
    const int64_t nkv = (t.a_len + tile - 1) / tile + (t.b_len + tile - 1) / tile;
    return nkv > 0 ? nkv + 2 : 0;
  };
  std::stable_sort(items.begin(), items.end(), [&](const Task& x, const Task& y) { return groups(x) > groups(y); });
  return items;
}

// Work list of full_attention_noalloc: a fixed array in static device memory
// (no allocation at call time), shared by every call on a device.
__device__ __align__(256) static Task g_noalloc_tasks[REFCACHE_NOALLOC_MAX_TASKS];
Task* g_noalloc_dev_ptr[kMaxDevices];
std::mutex g_noalloc_mu;
Task g_noalloc_host[REFCACHE_NOALLOC_MAX_TASKS];  // host staging, guarded by g_noalloc_mu

struct FullScratch {
  Task* buf = nullptr;
  size_t cap = 0;      // tasks
  int* work = nullptr;  // work counter, after the tasks
};
FullScratch g_full[kMaxDevices];
std::mutex g_full_mu;

}  // namespace

// ============================================================== the cache handle
struct refcache {
  int device = 0;
  int num_layers = 0, mode = 0, batch = 0, H = 0, D = 0;
  std::vector<int32_t> cu_live, cu_static, n_anchor;
  std::vector<int64_t> cache_off;  // [batch+1] cached rows per request, prefix sums
  int64_t live_rows = 0, static_rows = 0, cache_rows = 0;
  uint8_t* mem = nullptr;
  bool owns = false;
  Task* d_build = nullptr;
  int n_build = 0;
  // refcache_build_in_slot: the prefill over the cached rows already in the
  // slot (key range B) and the anchors given apart (key range A)
  Task* d_build_slot = nullptr;
  int n_build_slot = 0;
  int64_t anchor_rows = 0;
  int* d_status = nullptr;  // this cache's error word (device int), see refcache_cache_status
  int* d_work = nullptr;    // work counter of its CTA-pair launches (in the same 256-byte region)
  Task* d_step = nullptr;
  int n_step = 0;
  CopySeg* d_copy = nullptr;
  int n_copy = 0;
  // per-item lists of the pair kernel, ordered for the persistent
  // grid (the step's with split items), in a separate allocation:
  // [build items | step items | step jobs | part_o | part_lse]
  uint8_t* aux = nullptr;
  ItemList build_items, step_items;
  __nv_bfloat16* slots = nullptr;
  int64_t slot_elems = 0;
  // E4M3 cache (REFCACHE_CACHE_FP8): per layer [k8 | vt8 | scales] of
  // fp8_layer_bytes at slots8; each request's cached rows padded to 128
  bool f8 = false;
  int64_t rows_pad = 0;
  QuantTile* d_qtiles = nullptr;
  int n_qtiles = 0;
  uint8_t* slots8 = nullptr;
  size_t fp8_layer_bytes = 0;
  std::vector<char> built;
};

namespace {

// Bytes of one layer of an E4M3 cache: codes of K and V^T, and the scales.
size_t fp8_layer_bytes(int64_t rows_pad, int H, int D) {
  return align_up(static_cast<size_t>(rows_pad) * H * D, 256) * 2 +
         align_up(static_cast<size_t>(rows_pad / 128) * H * sizeof(float4), 256);
}

int cache_plan(int num_layers, int mode_flags, const refcache_segments_t* seg, refcache* h,
               std::vector<Task>* build_tasks, std::vector<Task>* step_tasks, std::vector<CopySeg>* copies,
               std::vector<QuantTile>* qtiles, std::vector<Task>* slot_tasks, size_t* total_bytes) {
  if (!seg) return fail(REFCACHE_ERR_INVALID_ARG, "seg is NULL");
  if (num_layers < 1) return fail(REFCACHE_ERR_INVALID_ARG, "num_layers must be >= 1");
  const bool f8 = (mode_flags & REFCACHE_CACHE_FP8) != 0;
  const int mode = mode_flags & ~REFCACHE_CACHE_FP8;
  if (mode != REFCACHE_MASK_BEYOND && mode != REFCACHE_MASK_BEYOND_ALT && mode != REFCACHE_MASK_ISOLATED)
    return fail(REFCACHE_ERR_INVALID_ARG, "unknown mask_mode %d", mode);
  int rc;
  if ((rc = check_dims(seg->batch, seg->num_heads, seg->head_dim)) != 0) return rc;
  const int B = seg->batch;
  const int64_t max_rows = (1ll << 31) - 1 - 512;
  if ((rc = check_cu(seg->cu_live, B, "cu_live", max_rows)) != 0) return rc;
  if ((rc = check_cu(seg->cu_static, B, "cu_static", max_rows)) != 0) return rc;
  if (!seg->n_anchor) return fail(REFCACHE_ERR_INVALID_ARG, "n_anchor is NULL");
  std::vector<int64_t> cache_off(B + 1, 0);
  for (int b = 0; b < B; ++b) {
    const int ns = seg->cu_static[b + 1] - seg->cu_static[b];
    const int na = seg->n_anchor[b];
    if (na < 0 || na > ns) return fail(REFCACHE_ERR_INVALID_ARG, "n_anchor[%d] = %d outside [0, %d]", b, na, ns);
    if (mode == REFCACHE_MASK_ISOLATED && na != 0)
      return fail(REFCACHE_ERR_INVALID_ARG, "isolated cache: n_anchor[%d] must be 0", b);
    if (seg->n_instr) {
      const int nl = seg->cu_live[b + 1] - seg->cu_live[b];
      if (seg->n_instr[b] < 0 || seg->n_instr[b] > nl)
        return fail(REFCACHE_ERR_INVALID_ARG, "n_instr[%d] outside [0, %d]", b, nl);
    }
    const int cached = mode == REFCACHE_MASK_BEYOND_ALT ? ns : ns - na;
    cache_off[b + 1] = cache_off[b] + cached;
  }
  if (cache_off[B] > max_rows) return fail(REFCACHE_ERR_INVALID_ARG, "cache rows too large");
  const int H = seg->num_heads, D = seg->head_dim;
  if (f8 && D != 128) return fail(REFCACHE_ERR_UNSUPPORTED, "the E4M3 cache needs head_dim 128 (got %d)", D);
  // E4M3 cache: request b's cached rows start at off8[b], a multiple of 128
  std::vector<int64_t> off8(B + 1, 0);
  std::vector<QuantTile> qt;
  for (int b = 0; b < B; ++b) {
    const int64_t nc = cache_off[b + 1] - cache_off[b];
    off8[b + 1] = off8[b] + (nc + 127) / 128 * 128;
    if (f8) {
      const int src0 = mode == REFCACHE_MASK_BEYOND_ALT ? seg->cu_static[b] : seg->cu_static[b] + seg->n_anchor[b];
      for (int64_t r = 0; r < nc; r += 128)
        qt.push_back(QuantTile{static_cast<int32_t>(src0 + r), static_cast<int32_t>(std::min<int64_t>(128, nc - r)),
                               static_cast<int32_t>(off8[b] + r), 0});
    }
  }
  if (off8[B] > max_rows) return fail(REFCACHE_ERR_INVALID_ARG, "cache rows too large");
  const int tr = task_rows(D);
  std::vector<Task> bt, st, bs;
  std::vector<CopySeg> cp;
  int a0 = 0;  // first row of request b's anchors in the anchor tensors of refcache_build_in_slot
  for (int b = 0; b < B; ++b) {
    const int s0 = seg->cu_static[b], ns = seg->cu_static[b + 1] - s0, na = seg->n_anchor[b];
    const int l0 = seg->cu_live[b], nl = seg->cu_live[b + 1] - l0;
    const int c0 = static_cast<int>(f8 ? off8[b] : cache_off[b]), nc = static_cast<int>(cache_off[b + 1] - cache_off[b]);
    if (mode == REFCACHE_MASK_BEYOND_ALT) {
      add_rows(bt, tr, s0, na, s0, na, 0, 0);            // anchor rows attend anchors only
      add_rows(bt, tr, s0 + na, ns - na, s0, ns, 0, 0);  // reference rows attend [ST; R]
    } else {
      add_rows(bt, tr, s0, ns, s0, ns, 0, 0);  // [ST; R] rows attend [ST; R] (R only when isolated)
    }
    add_rows(st, tr, l0, nl, l0, nl, c0, nc);  // live rows attend their own rows, then the cache
    if (!f8) {
      // in-slot build: the same rows and visibility, keys read from the slot
      if (mode == REFCACHE_MASK_BEYOND_ALT) {  // the slot holds [ST; R]: key range A is the slot
        add_rows(bs, tr, s0, na, c0, na, 0, 0);
        add_rows(bs, tr, s0 + na, ns - na, c0, ns, 0, 0);
      } else {  // anchors (range A, given apart), then R in the slot (range B)
        add_rows(bs, tr, s0, ns, a0, na, c0, nc);
      }
    }
    a0 += mode == REFCACHE_MASK_BEYOND_ALT ? 0 : na;
    if (nc > 0 && !f8) {
      CopySeg c{};
      c.src_row0 = mode == REFCACHE_MASK_BEYOND_ALT ? s0 : s0 + na;
      c.dst_row0 = c0;
      c.nrows = nc;
      cp.push_back(c);
    }
  }
  order_tasks(bt);
  order_tasks(st);
  order_tasks(bs);
  const size_t slot_elems = static_cast<size_t>(cache_off[B]) * H * D;
  size_t off = 0;
  off = align_up(off + bt.size() * sizeof(Task), 256);
  off = align_up(off + st.size() * sizeof(Task), 256);
  off = align_up(off + cp.size() * sizeof(CopySeg), 256);
  off = align_up(off + qt.size() * sizeof(QuantTile), 256);
  off = align_up(off + bs.size() * sizeof(Task), 256);
  off = align_up(off + sizeof(int), 256);  // the cache's error word and work counter
  const size_t layer_bytes = f8 ? fp8_layer_bytes(off8[B], H, D) : 2 * slot_elems * sizeof(__nv_bfloat16);
  const size_t total = off + static_cast<size_t>(num_layers) * layer_bytes;
  if (h) {
    h->f8 = f8;
    h->rows_pad = off8[B];
    h->n_qtiles = static_cast<int>(qt.size());
    h->fp8_layer_bytes = f8 ? layer_bytes : 0;
    h->num_layers = num_layers;
    h->mode = mode;
    h->batch = B;
    h->H = H;
    h->D = D;
    h->cu_live.assign(seg->cu_live, seg->cu_live + B + 1);
    h->cu_static.assign(seg->cu_static, seg->cu_static + B + 1);
    h->n_anchor.assign(seg->n_anchor, seg->n_anchor + B);
    h->cache_off = cache_off;
    h->live_rows = seg->cu_live[B];
    h->static_rows = seg->cu_static[B];
    h->cache_rows = cache_off[B];
    h->slot_elems = static_cast<int64_t>(slot_elems);
    h->n_build = static_cast<int>(bt.size());
    h->n_build_slot = static_cast<int>(bs.size());
    h->anchor_rows = a0;
    h->n_step = static_cast<int>(st.size());
    h->n_copy = static_cast<int>(cp.size());
  }
  if (build_tasks) *build_tasks = std::move(bt);
  if (step_tasks) *step_tasks = std::move(st);
  if (copies) *copies = std::move(cp);
  if (qtiles) *qtiles = std::move(qt);
  if (slot_tasks) *slot_tasks = std::move(bs);
  *total_bytes = total;
  return REFCACHE_OK;
}

int check_handle_layer(refcache* h, int layer) {
  if (!h) return fail(REFCACHE_ERR_INVALID_ARG, "cache is NULL");
  if (layer < 0 || layer >= h->num_layers)
    return fail(REFCACHE_ERR_INVALID_ARG, "layer %d outside [0, %d)", layer, h->num_layers);
  return REFCACHE_OK;
}

int check_ptrs(std::initializer_list<const void*> ps, int64_t rows, const char* what) {
  if (rows == 0) return REFCACHE_OK;
  for (const void* p : ps) {
    if (!p) return fail(REFCACHE_ERR_INVALID_ARG, "%s: NULL tensor pointer", what);
    if (!aligned16(p)) return fail(REFCACHE_ERR_INVALID_ARG, "%s: tensor pointer not 16-byte aligned", what);
  }
  return REFCACHE_OK;
}

// Per-item lists of a handle for the current device, in one
// allocation of their own (the caller-sized cache memory is not touched):
// the step's, with the last round of items split, and the prefill's, whose
// items are never split: each runs whole on one CTA pair, so a request's
// prefill outputs depend on its own (N_ST, N_R) only -- not on the other
// requests of the batch, nor on the device's SM count -- and the cached block
// is reproduced bit for bit (Sec. 3.3).  Both are ordered by longest_first.
int plan_split_items(refcache* h, DeviceInfo* info, const std::vector<Task>& bt, const std::vector<Task>& st) {
  // planned for the step kernel selected now (key tiles of tc2_tile(); the
  // split and the order stay correct, only less even, if another tile size
  // or grid runs them)
  const bool f8 = h->f8 && h->rows_pad > 0;
  const int tile = tc2_tile(f8), tile_b = tc2_tile(false);
  int clusters = 0;
  int rc = f8 ? tc2_clusters<true, 128, 128>(info, &clusters)
              : tile == 128 ? tc2_clusters<false, 128, 128>(info, &clusters)
                            : tc2_clusters<false, 192, 128>(info, &clusters);
  if (rc) return rc;
  std::vector<Task> si, bi;
  std::vector<CombineJob> sj;
  int parts = 0;
  plan_items(st, h->H, clusters, tile, &si, &sj, &parts);
  si = longest_first(std::move(si), tile);
  for (int hd = 0; hd < h->H; ++hd)
    for (Task t : bt) {
      t.head = hd;
      t.part = 0;
      bi.push_back(t);
    }
  bi = longest_first(std::move(bi), tile_b);
  const int rows = task_rows(h->D);
  size_t off = 0;
  const size_t o_bi = off;
  off = align_up(off + bi.size() * sizeof(Task), 256);
  const size_t o_si = off;
  off = align_up(off + si.size() * sizeof(Task), 256);
  const size_t o_sj = off;
  off = align_up(off + sj.size() * sizeof(CombineJob), 256);
  const size_t o_po = off;
  off = align_up(off + static_cast<size_t>(parts) * rows * h->D * sizeof(float), 256);
  const size_t o_pl = off;
  off = align_up(off + static_cast<size_t>(parts) * rows * sizeof(float), 256);
  cudaError_t e = cudaMalloc(reinterpret_cast<void**>(&h->aux), off);
  if (e != cudaSuccess) {
    h->aux = nullptr;
    return fail(REFCACHE_ERR_OOM, "cudaMalloc(%zu) for the split work list: %s", off, cudaGetErrorString(e));
  }
  auto put = [&](size_t o, const void* src, size_t n) -> cudaError_t {
    return n ? cudaMemcpy(h->aux + o, src, n, cudaMemcpyHostToDevice) : cudaSuccess;
  };
  if ((e = put(o_bi, bi.data(), bi.size() * sizeof(Task))) != cudaSuccess ||
      (e = put(o_si, si.data(), si.size() * sizeof(Task))) != cudaSuccess ||
      (e = put(o_sj, sj.data(), sj.size() * sizeof(CombineJob))) != cudaSuccess) {
    cudaFree(h->aux);
    h->aux = nullptr;
    return cuda_fail(e, "cudaMemcpy(split work list)");
  }
  h->build_items = ItemList{reinterpret_cast<Task*>(h->aux + o_bi), static_cast<int>(bi.size()), nullptr, 0,
                            nullptr, nullptr};
  h->step_items = ItemList{reinterpret_cast<Task*>(h->aux + o_si), static_cast<int>(si.size()),
                           reinterpret_cast<CombineJob*>(h->aux + o_sj), static_cast<int>(sj.size()),
                           reinterpret_cast<float*>(h->aux + o_po), reinterpret_cast<float*>(h->aux + o_pl)};
  return REFCACHE_OK;
}

int enter_device(refcache* h, DeviceInfo** info) {
  int dev = 0;
  int rc = current_device(&dev, info);
  if (rc) return rc;
  if (h && dev != h->device)
    return fail(REFCACHE_ERR_INVALID_ARG, "current device %d is not the cache's device %d", dev, h->device);
  return REFCACHE_OK;
}

}  // namespace

extern "C" {

size_t refcache_bytes(int num_layers, int mask_mode, const refcache_segments_t* seg) {
  size_t total = 0;
  if (cache_plan(num_layers, mask_mode, seg, nullptr, nullptr, nullptr, nullptr, nullptr, nullptr, &total) != 0) return 0;
  return total;
}

int refcache_create(refcache_t** out, int num_layers, int mask_mode, const refcache_segments_t* seg, void* dev_mem,
                    size_t dev_bytes) {
  if (!out) return fail(REFCACHE_ERR_INVALID_ARG, "out is NULL");
  refcache* h = new refcache();
  std::vector<Task> bt, st, bs;
  std::vector<CopySeg> cp;
  std::vector<QuantTile> qt;
  size_t total = 0;
  int rc = cache_plan(num_layers, mask_mode, seg, h, &bt, &st, &cp, &qt, &bs, &total);
  if (rc) {
    delete h;
    return rc;
  }
  if (dev_mem) {
    if (dev_bytes < total) {
      delete h;
      return fail(REFCACHE_ERR_OOM, "given %zu bytes, need %zu", dev_bytes, total);
    }
    if (reinterpret_cast<uintptr_t>(dev_mem) & 255u) {
      delete h;
      return fail(REFCACHE_ERR_INVALID_ARG, "dev_mem must be 256-byte aligned");
    }
  }
  DeviceInfo* info = nullptr;
  if ((rc = current_device(&h->device, &info)) != 0) {
    delete h;
    return rc;
  }
  if (dev_mem) {
    h->mem = static_cast<uint8_t*>(dev_mem);
  } else {
    cudaError_t e = cudaMalloc(reinterpret_cast<void**>(&h->mem), total);
    if (e != cudaSuccess) {
      delete h;
      return fail(REFCACHE_ERR_OOM, "cudaMalloc(%zu): %s", total, cudaGetErrorString(e));
    }
    h->owns = true;
  }
  size_t off = 0;
  h->d_build = reinterpret_cast<Task*>(h->mem + off);
  off = align_up(off + bt.size() * sizeof(Task), 256);
  h->d_step = reinterpret_cast<Task*>(h->mem + off);
  off = align_up(off + st.size() * sizeof(Task), 256);
  h->d_copy = reinterpret_cast<CopySeg*>(h->mem + off);
  off = align_up(off + cp.size() * sizeof(CopySeg), 256);
  h->d_qtiles = reinterpret_cast<QuantTile*>(h->mem + off);
  off = align_up(off + qt.size() * sizeof(QuantTile), 256);
  h->d_build_slot = reinterpret_cast<Task*>(h->mem + off);
  off = align_up(off + bs.size() * sizeof(Task), 256);
  h->d_status = reinterpret_cast<int*>(h->mem + off);
  h->d_work = h->d_status + kWorkOffset;
  off = align_up(off + sizeof(int), 256);
  h->slots = reinterpret_cast<__nv_bfloat16*>(h->mem + off);
  h->slots8 = h->mem + off;
  cudaError_t e = cudaSuccess;
  if (!bt.empty() && e == cudaSuccess) e = cudaMemcpy(h->d_build, bt.data(), bt.size() * sizeof(Task), cudaMemcpyHostToDevice);
  if (!st.empty() && e == cudaSuccess) e = cudaMemcpy(h->d_step, st.data(), st.size() * sizeof(Task), cudaMemcpyHostToDevice);
  if (!cp.empty() && e == cudaSuccess) e = cudaMemcpy(h->d_copy, cp.data(), cp.size() * sizeof(CopySeg), cudaMemcpyHostToDevice);
  if (!qt.empty() && e == cudaSuccess)
    e = cudaMemcpy(h->d_qtiles, qt.data(), qt.size() * sizeof(QuantTile), cudaMemcpyHostToDevice);
  if (!bs.empty() && e == cudaSuccess)
    e = cudaMemcpy(h->d_build_slot, bs.data(), bs.size() * sizeof(Task), cudaMemcpyHostToDevice);
  if (e == cudaSuccess) e = cudaMemset(h->d_status, 0, 256);
  if (e == cudaSuccess) e = cudaDeviceSynchronize();  // zero before any stream's first launch
  if (e != cudaSuccess) {
    if (h->owns) cudaFree(h->mem);
    delete h;
    return cuda_fail(e, "cudaMemcpy(work tables)");
  }
  if ((rc = plan_split_items(h, info, bt, st)) != 0) {
    if (h->owns) cudaFree(h->mem);
    delete h;
    return rc;
  }
  h->built.assign(num_layers, 0);
  *out = h;
  return REFCACHE_OK;
}

void refcache_destroy(refcache_t* h) {
  if (!h) return;
  if ((h->owns && h->mem) || h->aux) {
    int prev = 0;
    cudaGetDevice(&prev);
    cudaSetDevice(h->device);
    cudaDeviceSynchronize();
    if (h->owns && h->mem) cudaFree(h->mem);
    if (h->aux) cudaFree(h->aux);
    cudaSetDevice(prev);
  }
  delete h;
}

int refcache_kv_ptr(refcache_t* h, int layer, void** k_slot, void** v_slot, int64_t* rows) {
  int rc = check_handle_layer(h, layer);
  if (rc) return rc;
  if (h->f8) return fail(REFCACHE_ERR_UNSUPPORTED, "an E4M3 cache has no bf16 slots (see refcache_fp8_ptr)");
  __nv_bfloat16* k = h->slots + static_cast<int64_t>(layer) * 2 * h->slot_elems;
  if (k_slot) *k_slot = k;
  if (v_slot) *v_slot = k + h->slot_elems;
  if (rows) *rows = h->cache_rows;
  return REFCACHE_OK;
}

int refcache_fp8_ptr(refcache_t* h, int layer, void** k8, void** vt8, void** scales, int64_t* rows_pad) {
  int rc = check_handle_layer(h, layer);
  if (rc) return rc;
  if (!h->f8) return fail(REFCACHE_ERR_UNSUPPORTED, "not an E4M3 cache (create it with REFCACHE_CACHE_FP8)");
  uint8_t* base = h->slots8 + static_cast<size_t>(layer) * h->fp8_layer_bytes;
  const size_t codes = align_up(static_cast<size_t>(h->rows_pad) * h->H * h->D, 256);
  if (k8) *k8 = base;
  if (vt8) *vt8 = base + codes;
  if (scales) *scales = base + 2 * codes;
  if (rows_pad) *rows_pad = h->rows_pad;
  return REFCACHE_OK;
}

int refcache_call_launches(refcache_t* h, int call) {
  if (!h) return fail(REFCACHE_ERR_INVALID_ARG, "cache is NULL");
  if (call < 0 || call > 2)
    return fail(REFCACHE_ERR_INVALID_ARG, "call must be 0 (build), 1 (step) or 2 (build in slot)");
  if (call == 2) return h->f8 ? fail(REFCACHE_ERR_UNSUPPORTED, "an E4M3 cache has no in-slot build") : h->n_build_slot > 0;
  const int n_tasks = call == 0 ? h->n_build : h->n_step;
  const int cache_write = call == 0 && (h->n_copy > 0 || h->n_qtiles > 0) ? 1 : 0;
  if (n_tasks == 0) return cache_write;
  const bool tc = g_kernel.load() != REFCACHE_KERNEL_MMA_SYNC;
  const bool combine = call == 1 && tc && h->step_items.items && h->step_items.n_jobs > 0;
  return cache_write + 1 + (combine ? 1 : 0);
}

int refcache_layer_built(refcache_t* h, int layer) {
  int rc = check_handle_layer(h, layer);
  if (rc) return rc;
  return h->built[layer] ? 1 : 0;
}

int refcache_build(refcache_t* h, int layer, const void* q_static, const void* k_static, const void* v_static,
                   void* o_static, float* lse_static, float softmax_scale, void* stream) {
  int rc = check_handle_layer(h, layer);
  if (rc) return rc;
  if ((rc = check_scale(softmax_scale)) != 0) return rc;
  if ((rc = check_ptrs({q_static, k_static, v_static, o_static}, h->static_rows, "refcache_build")) != 0) return rc;
  DeviceInfo* info = nullptr;
  if ((rc = enter_device(h, &info)) != 0) return rc;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (h->f8 && h->n_qtiles > 0) {
    void *k8 = nullptr, *vt8 = nullptr, *sc = nullptr;
    refcache_fp8_ptr(h, layer, &k8, &vt8, &sc, nullptr);
    rc::quantize_cache_kernel<<<dim3(static_cast<unsigned>(h->H), static_cast<unsigned>(h->n_qtiles), 2), 256, 0, s>>>(
        h->d_qtiles, static_cast<const uint4*>(k_static), static_cast<const uint4*>(v_static),
        static_cast<uint8_t*>(k8), static_cast<uint8_t*>(vt8), static_cast<float4*>(sc), h->H, h->rows_pad);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_fail(e, "quantize_cache_kernel launch");
  }
  void *kslot = nullptr, *vslot = nullptr;
  if (!h->f8) refcache_kv_ptr(h, layer, &kslot, &vslot, nullptr);
  CopyJob cj;
  if (h->n_copy > 0) {
    cj.segs = h->d_copy;
    cj.n_segs = h->n_copy;
    cj.src_k = k_static;
    cj.src_v = v_static;
    cj.dst_k = kslot;
    cj.dst_v = vslot;
    cj.row_u4 = h->H * h->D * 2 / 16;
    cj.rows = h->cache_rows;
  }
  Operands op{q_static, h->static_rows, k_static, v_static, h->static_rows, nullptr, nullptr, 0, o_static, lse_static,
              h->d_status, h->d_work};
  rc = run_attention(h->d_build, h->n_build, h->H, h->D, op, softmax_scale, info, s,
                     h->build_items.items ? &h->build_items : nullptr, nullptr, h->n_copy > 0 ? &cj : nullptr);
  if (rc) return rc;
  h->built[layer] = 1;
  return REFCACHE_OK;
}

int refcache_build_in_slot(refcache_t* h, int layer, const void* q_static, const void* k_anchor,
                           const void* v_anchor, void* o_static, float* lse_static, float softmax_scale, void* stream) {
  int rc = check_handle_layer(h, layer);
  if (rc) return rc;
  if (h->f8)
    return fail(REFCACHE_ERR_UNSUPPORTED, "refcache_build_in_slot needs a bf16 cache (an E4M3 cache is written by "
                                          "refcache_build from the bf16 K and V)");
  if ((rc = check_scale(softmax_scale)) != 0) return rc;
  if ((rc = check_ptrs({q_static, o_static}, h->static_rows, "refcache_build_in_slot")) != 0) return rc;
  const bool alt = h->mode == REFCACHE_MASK_BEYOND_ALT;
  if (!alt && (rc = check_ptrs({k_anchor, v_anchor}, h->anchor_rows, "refcache_build_in_slot anchors")) != 0)
    return rc;
  DeviceInfo* info = nullptr;
  if ((rc = enter_device(h, &info)) != 0) return rc;
  void *kslot = nullptr, *vslot = nullptr;
  refcache_kv_ptr(h, layer, &kslot, &vslot, nullptr);
  const bool anchors = !alt && h->anchor_rows > 0;
  const bool range_b = !alt && h->cache_rows > 0;
  Operands op{q_static,
              h->static_rows,
              anchors ? k_anchor : kslot,
              anchors ? v_anchor : vslot,
              anchors ? h->anchor_rows : h->cache_rows,
              range_b ? kslot : nullptr,
              range_b ? vslot : nullptr,
              range_b ? h->cache_rows : 0,
              o_static,
              lse_static,
              h->d_status, h->d_work};
  rc = run_attention(h->d_build_slot, h->n_build_slot, h->H, h->D, op, softmax_scale, info,
                     static_cast<cudaStream_t>(stream));
  if (rc) return rc;
  h->built[layer] = 1;
  return REFCACHE_OK;
}

int step_attention(refcache_t* h, int layer, const void* q_live, const void* k_live, const void* v_live, void* o_live,
                   float* lse_live, float softmax_scale, void* stream) {
  int rc = check_handle_layer(h, layer);
  if (rc) return rc;
  if (!h->built[layer]) return fail(REFCACHE_ERR_NOT_BUILT, "layer %d has not been built", layer);
  if ((rc = check_scale(softmax_scale)) != 0) return rc;
  if ((rc = check_ptrs({q_live, k_live, v_live, o_live}, h->live_rows, "step_attention")) != 0) return rc;
  DeviceInfo* info = nullptr;
  if ((rc = enter_device(h, &info)) != 0) return rc;
  void *kslot = nullptr, *vslot = nullptr;
  Fp8B f8;
  // an E4M3 cache without cached rows has no range B: the bf16 kernel runs
  const bool use_f8 = h->f8 && h->rows_pad > 0;
  if (use_f8) {
    void* sc = nullptr;
    refcache_fp8_ptr(h, layer, const_cast<void**>(&f8.k8), const_cast<void**>(&f8.vt8), &sc, &f8.rows_pad);
    f8.scales = static_cast<const float4*>(sc);
  } else if (!h->f8) {
    refcache_kv_ptr(h, layer, &kslot, &vslot, nullptr);
  }
  Operands op{q_live, h->live_rows, k_live, v_live, h->live_rows, kslot, vslot, h->cache_rows, o_live, lse_live,
              h->d_status, h->d_work};
  return run_attention(h->d_step, h->n_step, h->H, h->D, op, softmax_scale, info, static_cast<cudaStream_t>(stream),
                       h->step_items.items ? &h->step_items : nullptr, use_f8 ? &f8 : nullptr);
}

int full_attention(int batch, int num_heads, int head_dim, const int32_t* cu_seqlens, const void* q, const void* k,
                   const void* v, void* o, float* lse, float softmax_scale, void* stream) {
  int rc = check_dims(batch, num_heads, head_dim);
  if (rc) return rc;
  if ((rc = check_cu(cu_seqlens, batch, "cu_seqlens", (1ll << 31) - 1 - 512)) != 0) return rc;
  if ((rc = check_scale(softmax_scale)) != 0) return rc;
  const int64_t rows = cu_seqlens[batch];
  if ((rc = check_ptrs({q, k, v, o}, rows, "full_attention")) != 0) return rc;
  DeviceInfo* info = nullptr;
  if ((rc = enter_device(nullptr, &info)) != 0) return rc;
  int dev = 0;
  cudaGetDevice(&dev);
  std::vector<Task> tasks;
  for (int b = 0; b < batch; ++b) {
    const int s0 = cu_seqlens[b], n = cu_seqlens[b + 1] - s0;
    add_rows(tasks, task_rows(head_dim), s0, n, s0, n, 0, 0);
  }
  order_tasks(tasks);
  if (tasks.empty()) return REFCACHE_OK;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  Task* d_tasks = nullptr;
  int* work = nullptr;
  {
    std::lock_guard<std::mutex> lk(g_full_mu);
    FullScratch& fs = g_full[dev];
    if (fs.cap < tasks.size()) {
      if (fs.buf) {
        cudaError_t e = cudaStreamSynchronize(s);
        if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
        cudaFree(fs.buf);
        fs.buf = nullptr;
        fs.cap = 0;
      }
      const size_t cap = std::max<size_t>(tasks.size(), 1024);
      cudaError_t e = cudaMalloc(reinterpret_cast<void**>(&fs.buf), cap * sizeof(Task) + 256);
      if (e != cudaSuccess) return fail(REFCACHE_ERR_OOM, "cudaMalloc(work list): %s", cudaGetErrorString(e));
      fs.cap = cap;
      fs.work = reinterpret_cast<int*>(fs.buf + cap);
      e = cudaMemsetAsync(fs.work, 0, 256, s);
      if (e != cudaSuccess) return cuda_fail(e, "cudaMemsetAsync(work counter)");
    }
    d_tasks = fs.buf;
    work = fs.work;
    cudaError_t e = cudaMemcpyAsync(d_tasks, tasks.data(), tasks.size() * sizeof(Task), cudaMemcpyHostToDevice, s);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpyAsync(work list)");
  }
  Operands op{q, rows, k, v, rows, nullptr, nullptr, 0, o, lse, nullptr, work};
  return run_attention(d_tasks, static_cast<int>(tasks.size()), num_heads, head_dim, op, softmax_scale, info, s);
}

int full_attention_noalloc(int batch, int num_heads, int head_dim, const int32_t* cu_seqlens, const void* q,
                           const void* k, const void* v, void* o, float* lse, float softmax_scale, void* stream) {
  int rc = check_dims(batch, num_heads, head_dim);
  if (rc) return rc;
  if ((rc = check_cu(cu_seqlens, batch, "cu_seqlens", (1ll << 31) - 1 - 512)) != 0) return rc;
  if ((rc = check_scale(softmax_scale)) != 0) return rc;
  const int tr = task_rows(head_dim);
  int64_t n_tasks = 0;
  for (int b = 0; b < batch; ++b) n_tasks += (cu_seqlens[b + 1] - cu_seqlens[b] + tr - 1) / tr;
  if (n_tasks > REFCACHE_NOALLOC_MAX_TASKS)
    return fail(REFCACHE_ERR_INVALID_ARG,
                "full_attention_noalloc: %lld work items exceed the static limit of %d (%d query rows each)",
                static_cast<long long>(n_tasks), REFCACHE_NOALLOC_MAX_TASKS, tr);
  const int64_t rows = cu_seqlens[batch];
  if ((rc = check_ptrs({q, k, v, o}, rows, "full_attention_noalloc")) != 0) return rc;
  DeviceInfo* info = nullptr;
  if ((rc = enter_device(nullptr, &info)) != 0) return rc;
  if (n_tasks == 0) return REFCACHE_OK;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  std::lock_guard<std::mutex> lk(g_noalloc_mu);
  if (!g_noalloc_dev_ptr[dev]) {
    // one-time set-up per device, with that device current: the host-side name
    // of a __device__ array is not a device address, so look the address up
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_tasks);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress(work list)");
    g_noalloc_dev_ptr[dev] = static_cast<Task*>(p);
  }
  int n = 0;
  for (int b = 0; b < batch; ++b) {
    const int s0 = cu_seqlens[b], len = cu_seqlens[b + 1] - s0;
    for (int r = 0; r < len; r += tr) {
      Task t{};
      t.q_row0 = s0 + r;
      t.q_rows = std::min(tr, len - r);
      t.a_row0 = s0;
      t.a_len = len;
      g_noalloc_host[n++] = t;
    }
  }
  // the same longest-first order as full_attention (ties by row, so the order is total)
  std::sort(g_noalloc_host, g_noalloc_host + n, [](const Task& x, const Task& y) {
    const int64_t cx = task_cost(x), cy = task_cost(y);
    return cx != cy ? cx > cy : x.q_row0 < y.q_row0;
  });
  // pageable source: the copy is staged before cudaMemcpyAsync returns, so the
  // host array may be reused by the next call
  e = cudaMemcpyAsync(g_noalloc_dev_ptr[dev], g_noalloc_host, static_cast<size_t>(n) * sizeof(Task),
                      cudaMemcpyHostToDevice, s);
  if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpyAsync(work list)");
  Operands op{q, rows, k, v, rows, nullptr, nullptr, 0, o, lse};
  return run_attention(g_noalloc_dev_ptr[dev], n, num_heads, head_dim, op, softmax_scale, info, s);
}

int refcache_status(void* stream) {
  cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
  int v = 0;
  e = cudaMemcpyFromSymbol(&v, rc::g_rc_status, sizeof(int));
  if (e != cudaSuccess) return cuda_fail(e, "read device error word");
  if (v != 0) {
    const int zero = 0;
    e = cudaMemcpyToSymbol(rc::g_rc_status, &zero, sizeof(int));
    if (e != cudaSuccess) return cuda_fail(e, "clear device error word");
    return fail(REFCACHE_ERR_TIMEOUT, "a kernel wait ran out (site %d)", v - RC_DEV_TIMEOUT_BASE);
  }
  return REFCACHE_OK;
}

int refcache_cache_status(refcache_t* h, void* stream) {
  if (!h) return fail(REFCACHE_ERR_INVALID_ARG, "cache is NULL");
  DeviceInfo* info = nullptr;
  int rc = enter_device(h, &info);
  if (rc) return rc;
  cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
  int v = 0;
  e = cudaMemcpy(&v, h->d_status, sizeof(int), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(e, "read the cache's error word");
  if (v != 0) {
    e = cudaMemset(h->d_status, 0, sizeof(int));
    if (e != cudaSuccess) return cuda_fail(e, "clear the cache's error word");
    return fail(REFCACHE_ERR_TIMEOUT, "a kernel wait of a launch for this cache ran out (site %d)",
                v - RC_DEV_TIMEOUT_BASE);
  }
  return REFCACHE_OK;
}

uint64_t refcache_set_wait_timeout_ns(uint64_t ns) { return g_timeout_ns.exchange(ns ? ns : 1); }

int refcache_set_kernel(int kernel) {
  if (kernel != REFCACHE_KERNEL_TCGEN05 && kernel != REFCACHE_KERNEL_MMA_SYNC &&
      kernel != REFCACHE_KERNEL_TCGEN05_K128)
    return fail(REFCACHE_ERR_INVALID_ARG, "unknown kernel %d", kernel);
  return g_kernel.exchange(kernel);
}

void refcache_debug_skip_first_load(int on) { g_dbg_skip.store(on ? 1 : 0); }

int refcache_ex2_rate(double* per_clk_per_sm, void* stream) {
  if (!per_clk_per_sm) return fail(REFCACHE_ERR_INVALID_ARG, "per_clk_per_sm is NULL");
  DeviceInfo* info = nullptr;
  int rc = enter_device(nullptr, &info);
  if (rc) return rc;
  const int blocks = std::min(info->num_sms, rc::kEx2MaxBlocks);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaError_t e = cudaFuncSetAttribute(rc::ex2_rate_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, rc::kEx2Smem);
  if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute(ex2_rate_kernel)");
  rc::ex2_rate_kernel<<<blocks, rc::kEx2Threads, rc::kEx2Smem, s>>>(-1.0f);
  e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "ex2_rate_kernel launch");
  std::vector<long long> cyc(static_cast<size_t>(blocks));
  e = cudaMemcpyFromSymbolAsync(cyc.data(), rc::g_ex2_cycles, cyc.size() * sizeof(long long), 0,
                                cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_fail(e, "read ex2_rate_kernel cycles");
  std::sort(cyc.begin(), cyc.end());
  const long long med = cyc[cyc.size() / 2];
  if (med <= 0) return fail(REFCACHE_ERR_CUDA, "ex2_rate_kernel measured no cycles");
  *per_clk_per_sm = static_cast<double>(rc::kEx2Threads) * rc::kEx2Chains * rc::kEx2Iters / static_cast<double>(med);
  return REFCACHE_OK;
}

int refcache_last_error(char* buf, size_t n) {
  if (buf && n > 0) {
    std::strncpy(buf, g_last_error.c_str(), n - 1);
    buf[n - 1] = '\0';
  }
  return static_cast<int>(g_last_error.size());
}

const char* refcache_version(void) { return "refcache 0.1.0 (sm_103a)"; }

}  // extern "C"
