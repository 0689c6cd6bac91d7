/*
 * refcache.h -- C ABI of the beyond-mask joint attention library for GB300
 * (sm_103a): exact reference K/V caching with static text anchors.
 *
 * The paper's method (Sec. 3.3 "Static Text Anchors", App. C "Derivation"):
 * one request's in-context sequence is [LT, X_t, ST, R] -- live instruction
 * text, the denoising target, static text anchors (the instruction embedded
 * once at t = 0) and the tokens of K reference images R = [R(1); ...; R(K)]
 * (Eq. 1).  R and ST attend each other and nothing else, so their layerwise
 * K and V (Eq. 2) never depend on X_t and are computed once; the live rows
 * [LT, X_t] attend [LT, X_t, R] at every denoising step.
 *
 *   refcache_build   the one-shot static prefill: rows [ST; R] attend keys
 *                    [ST; R]; the R rows' K and V are written into the
 *                    persistent per-layer cache (Sec. 3.3, Eq. cost-pre).
 *   step_attention   one layer of one denoising step: rows [LT; X_t] attend
 *                    their own keys and the cached R keys (App. C, Eq.
 *                    cost-step); no mask is materialised.
 *   full_attention   the full-attention recompute every key of [LT; X_t; R]
 *                    visible to every row (Sec. 3.2, C_full in App. C): the
 *                    baseline the cache is measured against.
 *
 * Conventions shared by every entry point
 *   - Tensors are THD: [tokens, num_heads, head_dim] bf16, head_dim
 *     contiguous, rows of consecutive requests packed back to back.  Base
 *     pointers must be device pointers aligned to 16 bytes.
 *   - head_dim is 64 or 128; num_heads >= 1.
 *   - Every input row must hold finite values (rows of a neighbouring request
 *     may be read into a tile and masked out; they must not be NaN/Inf).
 *   - softmax_scale must be finite and > 0 (1/sqrt(head_dim) is the usual
 *     choice; the paper does not state it).
 *   - lse outputs are optional (NULL = not written): fp32 [tokens, num_heads],
 *     natural-log log-sum-exp of the scaled scores of each row.
 *   - Outputs are bf16 rounded to nearest-even; scores, softmax and
 *     accumulation are fp32; P is rounded to bf16 before the P.V product.
 *   - Calls are asynchronous on `stream` (a cudaStream_t passed as void*;
 *     NULL = legacy default stream) and return a status code below.  A
 *     non-zero return means nothing was launched.  Device-side faults of a
 *     launched kernel (a bounded wait that ran out) are reported later by
 *     refcache_status().
 *   - Host arrays (segment tables) are read during the call only; the library
 *     keeps its own copies.
 *   - No entry point allocates device memory except refcache_create (the
 *     cache, unless it is given memory, and a separate work
 *     list with a workspace for split items, see refcache_create) and
 *     full_attention (a per-device work-list buffer that it keeps and grows).
 *   - The refcache_build, refcache_build_in_slot and step_attention calls of
 *     one cache share that workspace and the cache's work counter: issue them
 *     in stream order (one stream, or streams ordered by events), not
 *     concurrently.  Calls for different caches may run concurrently.
 *   - The tcgen05 attention kernel and the merge of split items are
 *     launched as programmatic dependents of the previous kernel on the
 *     stream: they wait for it to complete before they read memory, and they
 *     allow the kernel after them to start early.  A caller's kernel launched
 *     with programmatic stream serialization after a library call must
 *     therefore wait for its grid dependencies (griddepcontrol.wait) before it
 *     reads the library's outputs; ordinary launches need nothing.
 *   - refcache_build, refcache_build_in_slot and step_attention only launch
 *     kernels (no allocation, no copy), so they can be captured in a CUDA graph and replayed, once a
 *     first call on the device has run outside the capture (the kernels'
 *     attributes are set on first use).  full_attention is not capturable
 *     (it copies its work list from host memory).
 */
#ifndef REFCACHE_H
#define REFCACHE_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define REFCACHE_API __attribute__((visibility("default")))
#else
#define REFCACHE_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

/* ---- status codes ------------------------------------------------------ */
#define REFCACHE_OK 0
#define REFCACHE_ERR_INVALID_ARG (-1) /* null/misaligned pointer, bad sizes or offsets */
#define REFCACHE_ERR_UNSUPPORTED (-2) /* head_dim not 64/128, no sm_103 device */
#define REFCACHE_ERR_NOT_BUILT (-3)   /* step_attention on a layer whose cache was not built */
#define REFCACHE_ERR_CUDA (-4)        /* a CUDA runtime/driver call failed */
#define REFCACHE_ERR_OOM (-5)         /* device allocation failed or given memory too small */
#define REFCACHE_ERR_TIMEOUT (-6)     /* a kernel's bounded wait ran out (see refcache_status) */

/* ---- mask modes (who the static rows and the live rows attend) ---------- */
/* Sec. 3.3: ST <-> R both ways, live rows attend [LT, X_t, R], not ST.      */
#define REFCACHE_MASK_BEYOND 0
/* Alternative anchor reading: ST rows attend only ST, R rows attend [ST, R],
 * live rows attend [LT, X_t, ST, R]; the cache then keeps ST's K/V too.     */
#define REFCACHE_MASK_BEYOND_ALT 1
/* Sec. 4.1 isolated cache (prior-art topology): R attends only R; every
 * request must have zero anchors.                                            */
#define REFCACHE_MASK_ISOLATED 2

/* Cache format flag, OR-ed into mask_mode of refcache_bytes/refcache_create.
 * An explicitly approximate variant of the paper's exact cache (Sec. 3.3
 * reuses the cached K/V exactly): the cached rows are stored as OCP FP8 E4M3
 * codes with one fp32 scale per (128-row tile of one request, head):
 *   amax = max |x| over the tile's rows and the head's 128 columns,
 *   s = amax / 448, code = E4M3(x * (448 / amax)) (round to nearest even,
 *   IEEE fp32 divide and multiply; code 0 and s = 0 when amax = 0).
 * Layout of one layer (refcache_fp8_ptr): K codes [rows_pad, H, 128], V codes
 * transposed per head [H, 128, rows_pad], scales float32 [rows_pad / 128, H, 4]
 * = (s_K, s_V, log2 s_V, 1 / s_V) (the last two 0 when s_V = 0); each
 * request's cached rows start on a 128-row boundary and pad rows hold code 0.  head_dim must be 128 and the tcgen05 kernel selected.
 * step_attention then quantises each live query row per head the same way
 * (one scale per row), attends the cached keys on E4M3 tensor-core MMAs with
 * E4M3 softmax weights, and the live keys exactly as in the bf16 cache; the
 * prefill (refcache_build's outputs) is unchanged.  Half the cache bytes. */
#define REFCACHE_CACHE_FP8 0x100

/* Kernel selection (refcache_set_kernel): the tcgen05/TMEM/TMA kernel is the
 * default (on CTA pairs with 192-key tiles for the bf16 cache; head_dim 64
 * runs on the same kernel with the head dim padded to 128 inside shared
 * memory); the mma.sync kernel is the recompiled legacy-tensor-core baseline;
 * TCGEN05_K128 is the same tcgen05 pair kernel with 128-key tiles, kept as a
 * comparison point (the E4M3 cache always uses 128-key tiles). */
#define REFCACHE_KERNEL_TCGEN05 0
#define REFCACHE_KERNEL_MMA_SYNC 1
#define REFCACHE_KERNEL_TCGEN05_K128 2

/*
 * Segment table of a batch of requests (Eq. 1 layout, Sec. 3.3 order).
 * All arrays are HOST memory.
 *   cu_live[batch+1]   offsets of each request's [LT; X_t] rows in the step
 *                      tensors (cu_seqlens style, cu_live[0] = 0, non-decreasing)
 *   cu_static[batch+1] offsets of each request's [ST; R] rows in the prefill
 *                      tensors
 *   n_anchor[batch]    N_ST: the first n_anchor[b] rows of request b's static
 *                      segment are anchors, the rest are R (N_R >= 0)
 *   n_instr[batch]     N_LT (may be NULL): the first rows of each live segment
 *                      are instruction text; LT and X_t are attended alike, so
 *                      it is informational
 */
typedef struct {
  int32_t batch;
  int32_t num_heads;
  int32_t head_dim;
  const int32_t* cu_live;
  const int32_t* cu_static;
  const int32_t* n_anchor;
  const int32_t* n_instr;
} refcache_segments_t;

typedef struct refcache refcache_t; /* opaque; owns the per-layer K/V slots */

/*
 * Device bytes a cache needs for `num_layers` layers (Sec. 3.3: per layer the
 * R rows' K and V, bf16, [cache_rows, num_heads, head_dim] each, plus the
 * anchors' rows in REFCACHE_MASK_BEYOND_ALT; with REFCACHE_CACHE_FP8 the E4M3
 * layout above), plus its small work tables.  Returns 0 for invalid arguments.
 */
REFCACHE_API size_t refcache_bytes(int num_layers, int mask_mode, const refcache_segments_t* seg);

/*
 * Create a cache.  If dev_mem is NULL the library allocates refcache_bytes()
 * with cudaMalloc on the current device and frees it in refcache_destroy;
 * otherwise it uses dev_mem (>= refcache_bytes(), 256-byte aligned, owned by
 * the caller, not freed).  Synchronous.  *out is set only on success.
 *
 * It also plans, for the current device, the per-item work
 * lists of the prefill and the step, (query tile, head) items longest first;
 * a launch hands them out in that order to whichever CTA pair is free,
 * through a work counter kept in the cache's memory (reset by the launch
 * itself when it ends), so the pair that computes an item varies but its
 * arithmetic does not.  full_attention does the same with a counter kept
 * beside its work list; full_attention_noalloc takes items in a fixed order
 * (the same results, bit for bit).  When the step's
 * items do not fill the last round of the GPU's CTA pairs evenly, the items of
 * that round are split by key range into 2-8 parts whose outputs a combine
 * kernel merges.  These lists and an fp32 workspace for the parts (parts x 256
 * rows x (head_dim + 1) x 4 bytes, e.g. 27 MB at 1024^2 with five references)
 * are one more cudaMalloc, freed by refcache_destroy.  Which step items are split depends on the whole
 * batch and the device, so a step output's last bits may differ between
 * batches (never by more than the rounding of a split).  The prefill is never
 * split: refcache_build's outputs and cache bytes for a request depend only on
 * that request's own inputs, whatever else is in the batch and on any GPU.
 */
REFCACHE_API int refcache_create(refcache_t** out, int num_layers, int mask_mode, const refcache_segments_t* seg,
                    void* dev_mem, size_t dev_bytes);

/* Free the cache (waits for the device to finish using it).  NULL is a no-op. */
REFCACHE_API void refcache_destroy(refcache_t* cache);

/*
 * Device pointers of layer `layer`'s K and V slots, each a THD bf16 tensor of
 * *rows rows: request b's cached rows follow request b-1's.  Cached rows are
 * R (Eq. 2), or [ST; R] in REFCACHE_MASK_BEYOND_ALT.  Any output may be NULL.
 * REFCACHE_ERR_UNSUPPORTED for an E4M3 cache.
 */
REFCACHE_API int refcache_kv_ptr(refcache_t* cache, int layer, void** k_slot, void** v_slot, int64_t* rows);

/*
 * Device pointers of layer `layer` of an E4M3 cache (REFCACHE_CACHE_FP8): the
 * K codes [rows_pad, H, 128] (uint8), the V codes [H, 128, rows_pad] (uint8)
 * and the scales [rows_pad / 128, H, 4] (float32), owned by the cache.  Any
 * output may be NULL.  REFCACHE_ERR_UNSUPPORTED for a bf16 cache.
 */
REFCACHE_API int refcache_fp8_ptr(refcache_t* cache, int layer, void** k8, void** vt8, void** scales,
                                  int64_t* rows_pad);

/* 1 if `layer` has been built, 0 if not, < 0 on error. */
REFCACHE_API int refcache_layer_built(refcache_t* cache, int layer);

/*
 * Number of kernels one refcache_build (call = 0), step_attention (call = 1)
 * or refcache_build_in_slot (call = 2) on this cache launches with the kernel
 * family currently selected (refcache_set_kernel): the attention kernel, the
 * cache write (refcache_build, when there are cached rows: a copy, or the
 * E4M3 quantisation) and the combine of split items (step_attention, when the
 * cache's work list has any).  < 0 on error.
 */
REFCACHE_API int refcache_call_launches(refcache_t* cache, int call);

/*
 * Static prefill of one layer (Sec. 3.3; cost (N_R + N_ST)^2 per head,
 * Eq. cost-pre).  q_static/k_static/v_static: [cu_static[batch], H, d] bf16,
 * each request's [ST; R] rows.  Writes o_static (same shape) for every ST and
 * R row, lse_static if non-NULL, and copies the cached rows' K and V into the
 * layer's slots (an E4M3 cache: quantises them).  The result does not depend
 * on any live input, and repeated builds with the same inputs produce the
 * same bytes.
 */
REFCACHE_API int refcache_build(refcache_t* cache, int layer, const void* q_static, const void* k_static,
                   const void* v_static, void* o_static, float* lse_static, float softmax_scale,
                   void* stream);

/*
 * The static prefill of one layer for a caller that projects the cached rows'
 * K and V straight into the cache (the zero-copy path of Sec. 3.3: only R's
 * K/V are kept, so they may be written where they are kept): before the call
 * the layer's slots (refcache_kv_ptr) must hold the cached rows' K and V --
 * R, or [ST; R] in REFCACHE_MASK_BEYOND_ALT -- of every request, in the
 * slot's row order.  Computes what refcache_build computes (rows [ST; R] over
 * keys [ST; R] under the cache's mask mode) and marks the layer built, but
 * reads R's keys and values from the slots and launches no cache write.
 *   q_static: [cu_static[batch], H, d] bf16, each request's [ST; R] queries.
 *   k_anchor, v_anchor: [sum n_anchor, H, d] bf16, the anchors' K and V,
 *     request b's n_anchor[b] rows after request b-1's; NULL when there are
 *     no anchor rows, and ignored (may be NULL) in REFCACHE_MASK_BEYOND_ALT,
 *     whose slots hold the anchors too.
 *   o_static / lse_static as in refcache_build.
 * The keys are tiled from the anchors and from R separately, so the outputs
 * equal refcache_build's up to the rounding order of the sums, and repeated
 * calls on the same inputs give the same bytes.  The slots are only read.
 * REFCACHE_ERR_UNSUPPORTED for an E4M3 cache (REFCACHE_CACHE_FP8), which
 * refcache_build writes from bf16 K and V.
 */
REFCACHE_API int refcache_build_in_slot(refcache_t* cache, int layer, const void* q_static, const void* k_anchor,
                                        const void* v_anchor, void* o_static, float* lse_static, float softmax_scale,
                                        void* stream);

/*
 * One denoising step of one layer (App. C: [LT, X_t] queries over
 * [LT, X_t, R]; cost S (N_R + S) per head, Eq. cost-step).  q_live, k_live,
 * v_live: [cu_live[batch], H, d] bf16, each request's [LT; X_t] rows.  Keys
 * are the request's own live rows followed by its cached rows of `layer`.
 * Writes o_live (same shape) and lse_live if non-NULL.
 * Returns REFCACHE_ERR_NOT_BUILT if the layer was never built, and
 * REFCACHE_ERR_UNSUPPORTED for an E4M3 cache while the mma.sync kernel is
 * selected.
 */
REFCACHE_API int step_attention(refcache_t* cache, int layer, const void* q_live, const void* k_live,
                   const void* v_live, void* o_live, float* lse_live, float softmax_scale,
                   void* stream);

/*
 * Full attention (Sec. 3.2; C_full = T (N_R + S)^2 over T steps, App. C):
 * every row of request b attends every key of request b.  cu_seqlens is a
 * HOST array [batch+1]; q, k, v, o are [cu_seqlens[batch], H, d] bf16.
 * Uses (and on first use or growth allocates) a per-device work-list buffer
 * kept by the library; calls on one device must be ordered on one stream.
 */
REFCACHE_API int full_attention(int batch, int num_heads, int head_dim, const int32_t* cu_seqlens, const void* q,
                   const void* k, const void* v, void* o, float* lse, float softmax_scale,
                   void* stream);

/*
 * full_attention for callers that cannot allocate device memory -- e.g. code
 * running under a custom or pooled allocator that forbids cudaMalloc, or a
 * host runtime that must not grow GPU memory after start-up.  The paper has
 * no counterpart; this is a deployment variant of full_attention above.
 *
 * Same arguments, semantics and results as full_attention, but the work list
 * lives in a fixed array in the library's static device memory (held by every
 * GPU that loads the library until the process exits), so the call allocates
 * nothing: no cudaMalloc, no cudaFree, no allocating library routine.  The
 * caller still passes (and owns) q, k, v, o and lse.
 *   - The array holds REFCACHE_NOALLOC_MAX_TASKS work items (512 KiB).  One
 *     item covers up to 256 query rows of a request (either head_dim), so a
 *     request of n rows needs ceil(n / 256) items: at most 16384 x 256 rows
 *     per call (fewer when requests end mid-item).  Larger inputs are
 *     rejected with REFCACHE_ERR_INVALID_ARG and a message naming the limit.
 *   - The first call on each device looks up the array's device address with
 *     that device current (a one-time set-up).
 *   - Every call rewrites the whole work list it uses, so no state carries
 *     over, but all calls share the one array: calls whose kernels overlap on
 *     the GPU (different streams, or other threads) race.  Order them on one
 *     stream.
 */
#define REFCACHE_NOALLOC_MAX_TASKS 16384
REFCACHE_API int full_attention_noalloc(int batch, int num_heads, int head_dim, const int32_t* cu_seqlens,
                                        const void* q, const void* k, const void* v, void* o, float* lse,
                                        float softmax_scale, void* stream);

/*
 * Synchronise `stream`, then read and clear the current device's error word
 * written by kernels whose bounded waits ran out.  Returns REFCACHE_OK,
 * REFCACHE_ERR_TIMEOUT or REFCACHE_ERR_CUDA.
 * The word is one per device: every kernel of this library on the device (any
 * cache, any stream, full_attention too) writes it, and the first
 * refcache_status call that reads it clears it.  To learn which cache's launch
 * gave up, use refcache_cache_status.
 */
REFCACHE_API int refcache_status(void* stream);

/*
 * The same for one cache: synchronise `stream`, then read and clear the error
 * word of `cache`, which the kernels launched by refcache_build,
 * refcache_build_in_slot and step_attention on this cache set (besides the
 * device word) when a bounded wait runs out.  Returns REFCACHE_OK,
 * REFCACHE_ERR_TIMEOUT, REFCACHE_ERR_INVALID_ARG (NULL cache, or the current
 * device is not the cache's) or REFCACHE_ERR_CUDA.  It clears only this
 * cache's word, and refcache_status only the device word.
 */
REFCACHE_API int refcache_cache_status(refcache_t* cache, void* stream);

/* Wait limit of every in-kernel wait, nanoseconds (default 1e9).  Returns the old value. */
REFCACHE_API uint64_t refcache_set_wait_timeout_ns(uint64_t ns);

/* Select the kernel for subsequent calls (REFCACHE_KERNEL_*); returns the old one or < 0. */
REFCACHE_API int refcache_set_kernel(int kernel);

/*
 * Debug fault injection on the host side of the wait protocol: when `on` is
 * non-zero, the next launch's TMA producer skips its first K-tile load, so
 * the consumers' bounded waits run out and the kernel reports
 * REFCACHE_ERR_TIMEOUT through refcache_status() instead of hanging.  The
 * switch clears itself after one launch.  Only the tcgen05 kernel has it.
 */
REFCACHE_API void refcache_debug_skip_first_load(int on);

/*
 * Diagnostic: the rate of the GPU's exponential unit (ex2.approx.f32, the
 * special-function unit) on the current device, in exponentials per clock per
 * SM (median over the SMs), written to *per_clk_per_sm (host).  The softmax
 * of the attention kernels evaluates one exponential per visible (query, key)
 * pair of one head; this rate gives that work's floor beside the tensor-core
 * roofline.  The paper has no counterpart.  Runs one short kernel (one CTA
 * per SM, about 0.1 ms) on `stream` and synchronises it; allocates nothing.
 * Returns REFCACHE_ERR_INVALID_ARG for a NULL pointer.
 */
REFCACHE_API int refcache_ex2_rate(double* per_clk_per_sm, void* stream);

/* Copy the calling thread's last error message into buf (NUL-terminated); returns its length. */
REFCACHE_API int refcache_last_error(char* buf, size_t n);

/* Library version string. */
REFCACHE_API const char* refcache_version(void);

#ifdef __cplusplus
}
#endif

#endif /* REFCACHE_H */
