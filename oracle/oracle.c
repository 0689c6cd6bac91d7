/*
 * oracle.c -- plain CPU oracle for the masked joint attention of the
 * beyond-mask in-context diffusion transformer (static text anchors with exact
 * reference K/V caching).
 *
 * TEST INFRASTRUCTURE ONLY.  Only the tests, the smoke check and the
 * benchmark's CPU-baseline leg load this file.  It shares no code, header,
 * table or constant with the CUDA library, and the library never calls it.
 *
 * It computes the plain definition of masked softmax attention, in fp64,
 * without tiling, online softmax or any reordering:
 *
 *   for every computed query row i and head h
 *     s_j = scale * sum_c q[i,h,c] * k[j,h,c]     over the keys j visible to i
 *     m   = max_j s_j
 *     p_j = exp(s_j - m)
 *     l   = sum_j p_j                             (j in increasing index order)
 *     o[i,h,:] = (sum_j p_j * v[j,h,:]) / l
 *     lse[i,h] = m + log(l)
 *   and o = 0, lse = -inf when no key is visible.
 *
 * Inputs are raw bf16 bit patterns (uint16), converted to double exactly.
 *
 * The visibility of one request's joint sequence follows the paper:
 *   Sec. 3.3 "Static Text Anchors": sequence [LT, X_t, ST, R]; R and ST see
 *     each other; neither sees LT or X_t; LT and X_t see each other and R but
 *     not ST.
 *   App. C "Derivation": per step, [LT, X_t] queries attend [LT, X_t, R]; the
 *     static block [ST, R] is evaluated once.
 *   Sec. 4.1 / Table 1 "isolated cache": the prior-art cacheable topology, R
 *     sees only R.
 *   Sec. 3.2 / App. C: full attention, every token of [LT, X_t, R] sees every
 *     other.
 * plus one alternative reading of the anchor rows (anchors see only anchors,
 * live rows also see the anchors) kept as a separate mode.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

enum { ORC_BLK_LT = 0, ORC_BLK_X = 1, ORC_BLK_ST = 2, ORC_BLK_R = 3 };

enum {
  ORC_MODE_BEYOND = 0,      /* Sec. 3.3 */
  ORC_MODE_BEYOND_ALT = 1,  /* anchors see anchors only; live rows see anchors */
  ORC_MODE_ISOLATED = 2,    /* Sec. 4.1: R sees only R */
  ORC_MODE_FULL = 3         /* every block sees every block */
};

/* attends[mode][query block][key block], blocks ordered LT, X, ST, R. */
static const unsigned char orc_attends[4][4][4] = {
    /* BEYOND (Sec. 3.3) */
    {{1, 1, 0, 1}, {1, 1, 0, 1}, {0, 0, 1, 1}, {0, 0, 1, 1}},
    /* BEYOND_ALT */
    {{1, 1, 1, 1}, {1, 1, 1, 1}, {0, 0, 1, 0}, {0, 0, 1, 1}},
    /* ISOLATED (prior-art cache; ST rows, if any, see only ST) */
    {{1, 1, 0, 1}, {1, 1, 0, 1}, {0, 0, 1, 0}, {0, 0, 0, 1}},
    /* FULL */
    {{1, 1, 1, 1}, {1, 1, 1, 1}, {1, 1, 1, 1}, {1, 1, 1, 1}},
};

int oracle_block_visible(int mode, int q_block, int k_block) {
  if (mode < 0 || mode > 3 || q_block < 0 || q_block > 3 || k_block < 0 || k_block > 3) return -1;
  return orc_attends[mode][q_block][k_block];
}

int oracle_max_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}

void oracle_set_threads(int n) {
#ifdef _OPENMP
  if (n > 0) omp_set_num_threads(n);
#else
  (void)n;
#endif
}

static double bf16_to_double(uint16_t bits) {
  uint32_t u = (uint32_t)bits << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return (double)f;
}

/*
 * The definition above for one (row, head): the keys visible to the row are
 * given by a callback-free byte vector vis[0..nk).
 */
static void attend_one(const uint16_t* q, const uint16_t* k, const uint16_t* v, int row, int head,
                       int nk, int H, int d, const unsigned char* vis, double scale, double* s,
                       double* out_row, double* lse) {
  const size_t rs = (size_t)H * d; /* THD row stride in elements */
  const uint16_t* qi = q + (size_t)row * rs + (size_t)head * d;
  int any = 0;
  double m = -INFINITY;
  for (int j = 0; j < nk; ++j) {
    if (!vis[j]) continue;
    const uint16_t* kj = k + (size_t)j * rs + (size_t)head * d;
    double dot = 0.0;
    for (int c = 0; c < d; ++c) dot += bf16_to_double(qi[c]) * bf16_to_double(kj[c]);
    s[j] = scale * dot;
    if (!any || s[j] > m) m = s[j];
    any = 1;
  }
  for (int c = 0; c < d; ++c) out_row[c] = 0.0;
  if (!any) {
    if (lse) *lse = -INFINITY;
    return;
  }
  double l = 0.0;
  for (int j = 0; j < nk; ++j) {
    if (!vis[j]) continue;
    const double p = exp(s[j] - m);
    l += p;
    const uint16_t* vj = v + (size_t)j * rs + (size_t)head * d;
    for (int c = 0; c < d; ++c) out_row[c] += p * bf16_to_double(vj[c]);
  }
  for (int c = 0; c < d; ++c) out_row[c] /= l;
  if (lse) *lse = m + log(l);
}

/*
 * Brute force with an explicit mask: q [nq, H, d], k and v [nk, H, d] (bf16
 * bits), mask [nq * nk] row-major bytes (1 = query row attends key), or NULL
 * for all-visible.  out [nq, H, d] and lse [nq, H] in fp64 (lse may be NULL).
 */
int oracle_attention_explicit_mask(const uint16_t* q, const uint16_t* k, const uint16_t* v, int nq,
                                   int nk, int H, int d, const unsigned char* mask, double scale,
                                   double* out, double* lse) {
  if (nq < 0 || nk < 0 || H <= 0 || d <= 0 || !out) return -1;
  int err = 0;
#pragma omp parallel
  {
    double* s = (double*)malloc(sizeof(double) * (size_t)(nk > 0 ? nk : 1));
    unsigned char* ones = (unsigned char*)malloc((size_t)(nk > 0 ? nk : 1));
    if (!s || !ones) {
#pragma omp atomic write
      err = -2;
    } else {
      memset(ones, 1, (size_t)(nk > 0 ? nk : 1));
#pragma omp for schedule(dynamic, 4)
      for (long t = 0; t < (long)nq * H; ++t) {
        const int i = (int)(t / H), h = (int)(t % H);
        const unsigned char* vis = mask ? mask + (size_t)i * nk : ones;
        attend_one(q, k, v, i, h, nk, H, d, vis, scale, s, out + ((size_t)i * H + h) * d,
                   lse ? lse + (size_t)i * H + h : NULL);
      }
    }
    free(s);
    free(ones);
  }
  return err;
}

/*
 * One request's joint sequence [LT; X; ST; R] (Sec. 3.3 order): q, k, v are
 * [n_lt + n_x + n_st + n_r, H, d] bf16 bits.  Computes the (row, head) pairs
 * listed in pairs[2*t], pairs[2*t+1] (t < n_pairs), or every row and head when
 * pairs is NULL (then n_pairs is ignored and out is [N, H, d], lse [N, H]).
 * With a pair list, out is [n_pairs, d] and lse [n_pairs].
 */
int oracle_joint_attention(const uint16_t* q, const uint16_t* k, const uint16_t* v, int n_lt, int n_x,
                           int n_st, int n_r, int H, int d, int mode, double scale,
                           const int32_t* pairs, long n_pairs, double* out, double* lse) {
  if (n_lt < 0 || n_x < 0 || n_st < 0 || n_r < 0 || H <= 0 || d <= 0 || mode < 0 || mode > 3 || !out)
    return -1;
  const int n = n_lt + n_x + n_st + n_r;
  const int start[4] = {0, n_lt, n_lt + n_x, n_lt + n_x + n_st};
  const long total = pairs ? n_pairs : (long)n * H;
  int err = 0;
#pragma omp parallel
  {
    double* s = (double*)malloc(sizeof(double) * (size_t)(n > 0 ? n : 1));
    unsigned char* vis = (unsigned char*)malloc((size_t)(n > 0 ? n : 1));
    if (!s || !vis) {
#pragma omp atomic write
      err = -2;
    } else {
#pragma omp for schedule(dynamic, 4)
      for (long t = 0; t < total; ++t) {
        const int i = pairs ? pairs[2 * t] : (int)(t / H);
        const int h = pairs ? pairs[2 * t + 1] : (int)(t % H);
        if (i < 0 || i >= n || h < 0 || h >= H) {
#pragma omp atomic write
          err = -1;
          continue;
        }
        int qb = 3;
        while (qb > 0 && i < start[qb]) --qb;
        for (int j = 0; j < n; ++j) {
          int kb = 3;
          while (kb > 0 && j < start[kb]) --kb;
          vis[j] = orc_attends[mode][qb][kb];
        }
        attend_one(q, k, v, i, h, n, H, d, vis, scale, s, out + (size_t)t * d, lse ? lse + t : NULL);
      }
    }
    free(s);
    free(vis);
  }
  return err;
}
