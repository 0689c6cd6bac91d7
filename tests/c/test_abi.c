/*
 * test_abi.c -- the C ABI of librefcache.so (include/refcache.h) called from
 * plain C, without the Python binding.
 *
 *   test_abi cpu   sizing and argument checks; needs no device
 *   test_abi gpu   refcache_create / refcache_build (and refcache_build_in_slot) / step_attention of a small
 *                  ragged batch on the current GPU, head dims 64 and 128, both
 *                  outputs compared with the oracle's joint attention
 *                  (oracle/oracle.c, linked in) on the same input bytes
 *
 * Inputs come from a seeded xorshift generator in this file (no attention
 * arithmetic).  Exit status 0 = pass.
 */
#include <math.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <cuda_runtime.h>

#include "refcache.h"

/* the oracle's entry point (oracle/oracle.c) */
int oracle_joint_attention(const uint16_t* q, const uint16_t* k, const uint16_t* v, int n_lt, int n_x, int n_st,
                           int n_r, int H, int d, int mode, double scale, const int32_t* pairs, long n_pairs,
                           double* out, double* lse);

#define CHECK(cond, ...)                                   \
  do {                                                     \
    if (!(cond)) {                                         \
      fprintf(stderr, "FAIL %s:%d: ", __FILE__, __LINE__); \
      fprintf(stderr, __VA_ARGS__);                        \
      fprintf(stderr, "\n");                               \
      exit(1);                                             \
    }                                                      \
  } while (0)

static uint64_t rng_state = 88172645463325252ull;
static uint64_t xorshift(void) {
  rng_state ^= rng_state << 13;
  rng_state ^= rng_state >> 7;
  rng_state ^= rng_state << 17;
  return rng_state;
}
/* roughly N(0,1): sum of four uniforms, centred and scaled */
static float randn(void) {
  double s = 0;
  for (int i = 0; i < 4; ++i) s += (double)(xorshift() >> 11) / 9007199254740992.0;
  return (float)((s - 2.0) * 1.7320508);
}
/* fp32 -> bf16 bits, round to nearest even (finite inputs) */
static uint16_t to_bf16(float f) {
  uint32_t u;
  memcpy(&u, &f, 4);
  u += 0x7FFFu + ((u >> 16) & 1u);
  return (uint16_t)(u >> 16);
}
static float from_bf16(uint16_t b) {
  uint32_t u = (uint32_t)b << 16;
  float f;
  memcpy(&f, &u, 4);
  return f;
}
static uint16_t* rand_bf16(size_t n) {
  uint16_t* p = (uint16_t*)malloc(n * 2);
  for (size_t i = 0; i < n; ++i) p[i] = to_bf16(randn());
  return p;
}

static int run_cpu(void) {
  int32_t cu_live[2] = {0, 320}, cu_static[2] = {0, 288}, n_anchor[1] = {32};
  refcache_segments_t seg = {1, 4, 64, cu_live, cu_static, n_anchor, NULL};
  const size_t bytes = refcache_bytes(2, REFCACHE_MASK_BEYOND, &seg);
  /* two layers of K and V for 256 cached rows, 4 heads x 64: 2 x 2 x 256 x 4 x 64 x 2 bytes, plus tables */
  CHECK(bytes >= 2u * 2u * 256u * 4u * 64u * 2u && bytes < 2u * 2u * 256u * 4u * 64u * 2u + 65536u,
        "refcache_bytes %zu", bytes);
  CHECK(refcache_bytes(1, REFCACHE_MASK_BEYOND | REFCACHE_CACHE_FP8, &seg) == 0, "E4M3 cache with head_dim 64");
  int32_t bad_cu[2] = {1, 320};
  refcache_segments_t bad = seg;
  bad.cu_live = bad_cu;
  refcache_t* h = NULL;
  CHECK(refcache_create(&h, 1, REFCACHE_MASK_BEYOND, &bad, NULL, 0) == REFCACHE_ERR_INVALID_ARG && !h,
        "bad cu_live accepted");
  char msg[256];
  CHECK(refcache_last_error(msg, sizeof msg) > 0 && strstr(msg, "cu_live"), "last error: %s", msg);
  bad = seg;
  bad.head_dim = 96;
  CHECK(refcache_create(&h, 1, REFCACHE_MASK_BEYOND, &bad, NULL, 0) == REFCACHE_ERR_UNSUPPORTED, "head_dim 96");
  CHECK(refcache_create(&h, 1, 7, &seg, NULL, 0) == REFCACHE_ERR_INVALID_ARG, "unknown mask mode");
  CHECK(refcache_create(NULL, 1, REFCACHE_MASK_BEYOND, &seg, NULL, 0) == REFCACHE_ERR_INVALID_ARG, "null out");
  CHECK(full_attention(1, 4, 64, cu_live, NULL, NULL, NULL, NULL, NULL, 0.125f, NULL) == REFCACHE_ERR_INVALID_ARG,
        "null tensors");
  CHECK(refcache_set_kernel(9) == REFCACHE_ERR_INVALID_ARG, "unknown kernel");
  CHECK(strstr(refcache_version(), "sm_103a") != NULL, "version %s", refcache_version());
  refcache_destroy(NULL);
  printf("cpu ok\n");
  return 0;
}

typedef struct {
  int n_st, n_lt, n_x, n_r;
} req_t;

static double compare(const uint16_t* gpu, const double* ref, size_t n, double* mean_out) {
  double mx = 0, sum = 0;
  for (size_t i = 0; i < n; ++i) {
    const double e = fabs((double)from_bf16(gpu[i]) - ref[i]);
    if (!(e <= mx)) mx = e; /* NaN propagates */
    sum += e;
  }
  *mean_out = n ? sum / (double)n : 0;
  return mx;
}

static int run_gpu_dim(int d) {
  const req_t reqs[] = {{5, 7, 150, 300}, {0, 0, 64, 129}, {16, 20, 1, 0}, {1, 3, 200, 260}};
  const int B = (int)(sizeof reqs / sizeof reqs[0]), H = 2;
  int32_t cu_live[8], cu_static[8], n_anchor[8], n_instr[8];
  cu_live[0] = cu_static[0] = 0;
  for (int b = 0; b < B; ++b) {
    cu_live[b + 1] = cu_live[b] + reqs[b].n_lt + reqs[b].n_x;
    cu_static[b + 1] = cu_static[b] + reqs[b].n_st + reqs[b].n_r;
    n_anchor[b] = reqs[b].n_st;
    n_instr[b] = reqs[b].n_lt;
  }
  const size_t row = (size_t)H * d, n_s = (size_t)cu_static[B] * row, n_l = (size_t)cu_live[B] * row;
  uint16_t *qs = rand_bf16(n_s), *ks = rand_bf16(n_s), *vs = rand_bf16(n_s);
  uint16_t *ql = rand_bf16(n_l), *kl = rand_bf16(n_l), *vl = rand_bf16(n_l);
  void* dev[8];
  const size_t sizes[8] = {n_s * 2, n_s * 2, n_s * 2, n_s * 2, n_l * 2, n_l * 2, n_l * 2, n_l * 2};
  const void* host[8] = {qs, ks, vs, NULL, ql, kl, vl, NULL};
  for (int i = 0; i < 8; ++i) {
    CHECK(cudaMalloc(&dev[i], sizes[i] ? sizes[i] : 16) == cudaSuccess, "cudaMalloc");
    if (host[i]) CHECK(cudaMemcpy(dev[i], host[i], sizes[i], cudaMemcpyHostToDevice) == cudaSuccess, "copy in");
  }
  refcache_segments_t seg = {B, H, d, cu_live, cu_static, n_anchor, n_instr};
  refcache_t* h = NULL;
  int rc = refcache_create(&h, 1, REFCACHE_MASK_BEYOND, &seg, NULL, 0);
  CHECK(rc == REFCACHE_OK && h, "refcache_create %d", rc);
  const float scale = 1.0f / sqrtf((float)d);
  rc = step_attention(h, 0, dev[4], dev[5], dev[6], dev[7], NULL, scale, NULL);
  CHECK(rc == REFCACHE_ERR_NOT_BUILT, "step before build: %d", rc);
  rc = refcache_build(h, 0, dev[0], dev[1], dev[2], dev[3], NULL, scale, NULL);
  CHECK(rc == REFCACHE_OK, "refcache_build %d", rc);
  rc = step_attention(h, 0, dev[4], dev[5], dev[6], dev[7], NULL, scale, NULL);
  CHECK(rc == REFCACHE_OK, "step_attention %d", rc);
  /* the same prefill for a caller that writes the cached rows' K/V straight
     into the slots (here by copying R's rows there) and passes the anchors apart */
  refcache_t* h2 = NULL;
  rc = refcache_create(&h2, 1, REFCACHE_MASK_BEYOND, &seg, NULL, 0);
  CHECK(rc == REFCACHE_OK && h2, "refcache_create (in-slot) %d", rc);
  void *kslot = NULL, *vslot = NULL, *da[2], *os2_d, *ol2_d;
  int64_t crows = 0, na_tot = 0;
  CHECK(refcache_kv_ptr(h2, 0, &kslot, &vslot, &crows) == REFCACHE_OK, "refcache_kv_ptr");
  for (int b = 0; b < B; ++b) na_tot += reqs[b].n_st;
  for (int i = 0; i < 2; ++i) CHECK(cudaMalloc(&da[i], na_tot ? (size_t)na_tot * row * 2 : 16) == cudaSuccess, "cudaMalloc");
  CHECK(cudaMalloc(&os2_d, n_s * 2) == cudaSuccess && cudaMalloc(&ol2_d, n_l * 2) == cudaSuccess, "cudaMalloc");
  int64_t c_rows = 0, a_rows = 0;
  for (int b = 0; b < B; ++b) {
    const size_t src_r = ((size_t)cu_static[b] + reqs[b].n_st) * row * 2, src_a = (size_t)cu_static[b] * row * 2;
    const size_t nr = (size_t)reqs[b].n_r * row * 2, na = (size_t)reqs[b].n_st * row * 2;
    CHECK(cudaMemcpy((char*)kslot + c_rows * row * 2, (char*)dev[1] + src_r, nr, cudaMemcpyDeviceToDevice) == cudaSuccess &&
              cudaMemcpy((char*)vslot + c_rows * row * 2, (char*)dev[2] + src_r, nr, cudaMemcpyDeviceToDevice) == cudaSuccess &&
              cudaMemcpy((char*)da[0] + a_rows * row * 2, (char*)dev[1] + src_a, na, cudaMemcpyDeviceToDevice) == cudaSuccess &&
              cudaMemcpy((char*)da[1] + a_rows * row * 2, (char*)dev[2] + src_a, na, cudaMemcpyDeviceToDevice) == cudaSuccess,
          "slot copy");
    c_rows += reqs[b].n_r;
    a_rows += reqs[b].n_st;
  }
  CHECK(c_rows == crows, "slot rows %lld, expected %lld", (long long)crows, (long long)c_rows);
  rc = refcache_build_in_slot(h2, 0, dev[0], da[0], da[1], os2_d, NULL, scale, NULL);
  CHECK(rc == REFCACHE_OK, "refcache_build_in_slot %d", rc);
  rc = step_attention(h2, 0, dev[4], dev[5], dev[6], ol2_d, NULL, scale, NULL);
  CHECK(rc == REFCACHE_OK, "step_attention (in-slot cache) %d", rc);
  rc = refcache_status(NULL);
  CHECK(rc == REFCACHE_OK, "refcache_status %d", rc);
  uint16_t* os = (uint16_t*)malloc(n_s * 2 + 2);
  uint16_t* ol = (uint16_t*)malloc(n_l * 2 + 2);
  uint16_t* os2 = (uint16_t*)malloc(n_s * 2 + 2);
  uint16_t* ol2 = (uint16_t*)malloc(n_l * 2 + 2);
  CHECK(cudaMemcpy(os, dev[3], n_s * 2, cudaMemcpyDeviceToHost) == cudaSuccess, "copy out");
  CHECK(cudaMemcpy(ol, dev[7], n_l * 2, cudaMemcpyDeviceToHost) == cudaSuccess, "copy out");
  CHECK(cudaMemcpy(os2, os2_d, n_s * 2, cudaMemcpyDeviceToHost) == cudaSuccess, "copy out");
  CHECK(cudaMemcpy(ol2, ol2_d, n_l * 2, cudaMemcpyDeviceToHost) == cudaSuccess, "copy out");
  double worst = 0;
  for (int b = 0; b < B; ++b) {
    const req_t r = reqs[b];
    const int n_live = r.n_lt + r.n_x, n_stat = r.n_st + r.n_r, n = n_live + n_stat;
    if (n == 0) continue;
    /* the joint sequence [LT; X; ST; R] of this request (Sec. 3.3 order) */
    uint16_t *q = calloc((size_t)n * row + 1, 2), *k = calloc((size_t)n * row + 1, 2), *v = calloc((size_t)n * row + 1, 2);
    memcpy(q, ql + (size_t)cu_live[b] * row, (size_t)n_live * row * 2);
    memcpy(k, kl + (size_t)cu_live[b] * row, (size_t)n_live * row * 2);
    memcpy(v, vl + (size_t)cu_live[b] * row, (size_t)n_live * row * 2);
    memcpy(q + (size_t)n_live * row, qs + (size_t)cu_static[b] * row, (size_t)n_stat * row * 2);
    memcpy(k + (size_t)n_live * row, ks + (size_t)cu_static[b] * row, (size_t)n_stat * row * 2);
    memcpy(v + (size_t)n_live * row, vs + (size_t)cu_static[b] * row, (size_t)n_stat * row * 2);
    double* out = malloc(sizeof(double) * ((size_t)n * row + 1));
    /* oracle mode 0: the paper's beyond mask (Sec. 3.3) */
    CHECK(oracle_joint_attention(q, k, v, r.n_lt, r.n_x, r.n_st, r.n_r, H, d, 0, (double)scale, NULL, 0, out,
                                 NULL) == 0,
          "oracle");
    double mean_l, mean_s;
    const double mx_l = compare(ol + (size_t)cu_live[b] * row, out, (size_t)n_live * row, &mean_l);
    const double mx_s = compare(os + (size_t)cu_static[b] * row, out + (size_t)n_live * row, (size_t)n_stat * row, &mean_s);
    CHECK(mx_l <= 2e-2 && mean_l <= 2e-3, "d=%d request %d step: max %.3e mean %.3e", d, b, mx_l, mean_l);
    CHECK(mx_s <= 2e-2 && mean_s <= 2e-3, "d=%d request %d prefill: max %.3e mean %.3e", d, b, mx_s, mean_s);
    double mean_l2, mean_s2;
    const double mx_l2 = compare(ol2 + (size_t)cu_live[b] * row, out, (size_t)n_live * row, &mean_l2);
    const double mx_s2 = compare(os2 + (size_t)cu_static[b] * row, out + (size_t)n_live * row, (size_t)n_stat * row, &mean_s2);
    CHECK(mx_l2 <= 2e-2 && mean_l2 <= 2e-3, "d=%d request %d step (in-slot cache): max %.3e", d, b, mx_l2);
    CHECK(mx_s2 <= 2e-2 && mean_s2 <= 2e-3, "d=%d request %d in-slot prefill: max %.3e", d, b, mx_s2);
    if (mx_s2 > worst) worst = mx_s2;
    if (mx_l > worst) worst = mx_l;
    if (mx_s > worst) worst = mx_s;
    free(q);
    free(k);
    free(v);
    free(out);
  }
  refcache_destroy(h);
  refcache_destroy(h2);
  for (int i = 0; i < 8; ++i) cudaFree(dev[i]);
  cudaFree(da[0]);
  cudaFree(da[1]);
  cudaFree(os2_d);
  cudaFree(ol2_d);
  free(qs); free(ks); free(vs); free(ql); free(kl); free(vl); free(os); free(ol); free(os2); free(ol2);
  printf("gpu d=%d ok (max abs %.3e)\n", d, worst);
  return 0;
}

int main(int argc, char** argv) {
  if (argc < 2) {
    fprintf(stderr, "usage: %s cpu|gpu\n", argv[0]);
    return 2;
  }
  if (!strcmp(argv[1], "cpu")) return run_cpu();
  if (!strcmp(argv[1], "gpu")) return run_gpu_dim(64) || run_gpu_dim(128);
  return 2;
}
