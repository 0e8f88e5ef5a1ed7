/*
 * ppconv_oracle.c -- plain, slow, fp64 CPU oracle for pattern- and
 * connectivity-pruned 3x3 convolution (stride 1, pad 1, NCHW).
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product library calls, links or
 * includes this file; only the tests, the smoke check and the CPU-baseline leg
 * of the benchmark load it.  It shares no code, header or table with the CUDA
 * path.
 *
 * What it follows (Niu et al., "Towards Real-Time DNN Inference on Mobile
 * Platforms with Model Pruning and Compiler Optimization", IJCAI-20 demo):
 *   - Section 2, "Structured Model Pruning": connectivity pruning removes whole
 *     (output, input) kernels; pattern pruning keeps certain locations of each
 *     kernel.  Each kept kernel keeps 4 of its 9 taps, the 4 taps forming one
 *     pattern of a small given pattern set.
 *   - Section 3, "Sparse model storage": zeros are not stored, and indices that
 *     the structure makes redundant are dropped (a kept kernel is stored as a
 *     pattern id plus 4 weights).
 *   - Section 3, "Matrix reorder": filters (rows) are reordered so that ones with
 *     the same or similar patterns sit together, then the kept kernels of each
 *     filter are compacted (columns).
 *
 * Readings where the paper is silent (each is listed in the design notes):
 *   - pattern id of a kept kernel: the id given by the caller, else the lowest
 *     pattern whose taps contain the kernel's nonzero support;
 *   - filter order: stable sort by (kept count descending, dominant pattern
 *     ascending, filter index ascending), the dominant pattern being the most
 *     frequent pattern id of the filter's kept kernels (lowest id on ties, 0
 *     for a filter with no kept kernel);
 *   - kernel order within a filter: (pattern id ascending, input channel
 *     ascending); the 4 weights of a kernel follow the pattern's ascending taps.
 *
 * The convolution is the plain definition: every output is the bias plus the
 * sum over kept kernels and over the taps of each kernel's pattern of
 * weight * input, with zero padding, accumulated in fp64.  The error budget
 * S = |bias| + sum |weight * input| is returned beside every output.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define OR_OK 0
#define OR_INVALID_ARG 1
#define OR_BAD_PATTERN_SET 2
#define OR_TAP_NOT_IN_PATTERN 3
#define OR_PRUNED_NONZERO 4
#define OR_PATTERN_ID_MISMATCH 5

int oracle_num_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}

/* A pattern set is valid when every pattern lists 4 distinct taps in 0..8 in
 * ascending order and no two patterns are equal (Section 2: each kernel keeps
 * 4 of its 9 locations, from a small set of patterns). */
static int check_pattern_set(const uint8_t* taps, int P) {
  if (P < 1 || P > 126) return OR_BAD_PATTERN_SET;
  for (int p = 0; p < P; ++p) {
    for (int s = 0; s < 4; ++s) {
      if (taps[4 * p + s] > 8) return OR_BAD_PATTERN_SET;
      if (s > 0 && taps[4 * p + s] <= taps[4 * p + s - 1]) return OR_BAD_PATTERN_SET;
    }
    for (int q = 0; q < p; ++q) {
      int same = 1;
      for (int s = 0; s < 4; ++s)
        if (taps[4 * p + s] != taps[4 * q + s]) same = 0;
      if (same) return OR_BAD_PATTERN_SET;
    }
  }
  return OR_OK;
}

/* 1 when tap t is one of the 4 taps of pattern p. */
static int pattern_has_tap(const uint8_t* taps, int p, int t) {
  for (int s = 0; s < 4; ++s)
    if (taps[4 * p + s] == t) return 1;
  return 0;
}

/* 1 when every nonzero weight of the 9-tap kernel k sits on a tap of pattern p. */
static int support_in_pattern(const float* k, const uint8_t* taps, int p) {
  for (int t = 0; t < 9; ++t)
    if (k[t] != 0.0f && !pattern_has_tap(taps, p, t)) return 0;
  return 1;
}

/*
 * Validate a pruned layer and name the pattern of every kept kernel
 * (Section 2, connectivity and pattern pruning).
 *   w     [Co][Ci][9] fp32 weights, tap t = 3*ky + kx
 *   mask  [Co][Ci]    1 = kernel kept, 0 = kernel pruned
 *   taps  [P][4]      the pattern set
 *   given [Co][Ci]    optional caller-given pattern ids (NULL: infer)
 *   pat   [Co][Ci]    out: pattern id of each kept kernel, -1 for pruned ones
 * Returns OR_OK or the first violation found (kernels in row-major order).
 */
int oracle_pattern_ids(const float* w, const uint8_t* mask, const uint8_t* taps, int P, int Co, int Ci,
                       const uint8_t* given, int32_t* pat) {
  if (!w || !mask || !taps || !pat || Co < 1 || Ci < 1) return OR_INVALID_ARG;
  int rc = check_pattern_set(taps, P);
  if (rc != OR_OK) return rc;
  for (int o = 0; o < Co; ++o) {
    for (int i = 0; i < Ci; ++i) {
      const float* k = w + ((size_t)o * Ci + i) * 9;
      size_t oi = (size_t)o * Ci + i;
      if (!mask[oi]) {
        for (int t = 0; t < 9; ++t)
          if (k[t] != 0.0f) return OR_PRUNED_NONZERO;
        pat[oi] = -1;
        continue;
      }
      if (given) {
        if (given[oi] >= P || !support_in_pattern(k, taps, given[oi])) return OR_PATTERN_ID_MISMATCH;
        pat[oi] = given[oi];
        continue;
      }
      int found = -1;
      for (int p = 0; p < P && found < 0; ++p)
        if (support_in_pattern(k, taps, p)) found = p;
      if (found < 0) return OR_TAP_NOT_IN_PATTERN;
      pat[oi] = found;
    }
  }
  return OR_OK;
}

/* Ordering key of the filter reorder: a before b when a has more kept kernels,
 * or as many and a lower dominant pattern, or both equal and a lower index. */
static int filter_before(int a, int b, const int64_t* cnt, const int32_t* dom) {
  if (cnt[a] != cnt[b]) return cnt[a] > cnt[b];
  if (dom[a] != dom[b]) return dom[a] < dom[b];
  return a < b;
}

/*
 * The compact storage and matrix reorder of Section 3.
 *   perm [Co]       perm[j] = original index of the j-th filter after reorder
 *   kptr [Co+1]     kept kernels of filter perm[j] are entries kptr[j]..kptr[j+1]-1
 *   kidx [nk]       input channel of each stored kernel
 *   kpat [nk]       pattern id of each stored kernel
 *   kw   [nk][4]    the kernel's weights on its pattern's taps, ascending taps
 *   nk_out          number of kept kernels
 * kidx/kpat/kw must hold at least the number of kept kernels (Co*Ci is always
 * enough).  Returns OR_OK or the validation error of oracle_pattern_ids.
 */
int oracle_pack(const float* w, const uint8_t* mask, const uint8_t* taps, int P, int Co, int Ci,
                const uint8_t* given, int32_t* perm, int32_t* kptr, int32_t* kidx, uint8_t* kpat, float* kw,
                int64_t* nk_out) {
  if (!perm || !kptr || !kidx || !kpat || !kw || !nk_out) return OR_INVALID_ARG;
  int32_t* pat = (int32_t*)malloc(sizeof(int32_t) * (size_t)Co * Ci);
  int64_t* cnt = (int64_t*)calloc((size_t)Co, sizeof(int64_t));
  int32_t* dom = (int32_t*)calloc((size_t)Co, sizeof(int32_t));
  int64_t* hist = (int64_t*)calloc((size_t)P > 0 ? (size_t)P : 1, sizeof(int64_t));
  if (!pat || !cnt || !dom || !hist) {
    free(pat); free(cnt); free(dom); free(hist);
    return OR_INVALID_ARG;
  }
  int rc = oracle_pattern_ids(w, mask, taps, P, Co, Ci, given, pat);
  if (rc != OR_OK) {
    free(pat); free(cnt); free(dom); free(hist);
    return rc;
  }
  /* kept count and dominant pattern of every filter */
  for (int o = 0; o < Co; ++o) {
    memset(hist, 0, sizeof(int64_t) * (size_t)P);
    for (int i = 0; i < Ci; ++i) {
      int32_t p = pat[(size_t)o * Ci + i];
      if (p >= 0) {
        cnt[o] += 1;
        hist[p] += 1;
      }
    }
    int best = 0;
    for (int p = 1; p < P; ++p)
      if (hist[p] > hist[best]) best = p;
    dom[o] = best;
  }
  /* filter reorder: insertion sort on the key (stable by construction) */
  for (int o = 0; o < Co; ++o) perm[o] = o;
  for (int a = 1; a < Co; ++a) {
    int32_t v = perm[a];
    int b = a - 1;
    while (b >= 0 && filter_before(v, perm[b], cnt, dom)) {
      perm[b + 1] = perm[b];
      --b;
    }
    perm[b + 1] = v;
  }
  /* kernel compaction: per filter, kept kernels by (pattern, input channel) */
  int64_t e = 0;
  kptr[0] = 0;
  for (int j = 0; j < Co; ++j) {
    int o = perm[j];
    for (int p = 0; p < P; ++p) {
      for (int i = 0; i < Ci; ++i) {
        if (pat[(size_t)o * Ci + i] != p) continue;
        kidx[e] = i;
        kpat[e] = (uint8_t)p;
        for (int s = 0; s < 4; ++s) kw[4 * e + s] = w[((size_t)o * Ci + i) * 9 + taps[4 * p + s]];
        ++e;
      }
    }
    kptr[j + 1] = (int32_t)e;
  }
  *nk_out = e;
  free(pat); free(cnt); free(dom); free(hist);
  return OR_OK;
}

/* Input value at (n, i, r, c) with the zero padding of a pad-1 convolution. */
static double x_at(const float* x, int Ci, int H, int W, int n, int i, int r, int c) {
  if (r < 0 || r >= H || c < 0 || c >= W) return 0.0;
  return (double)x[(((size_t)n * Ci + i) * H + r) * W + c];
}

/* One output of the pruned layer: bias plus, over every kept kernel (o, i) and
 * every tap t of its pattern, w[o][i][t] * x[n][i][r+ky-1][c+kx-1] with
 * (ky, kx) = (t / 3, t % 3).  *s receives |bias| + sum |w * x|. */
static void one_output_pruned(const float* x, int Ci, int H, int W, const float* w, const int32_t* pat,
                              const uint8_t* taps, const float* bias, int n, int o, int r, int c, double* y,
                              double* s) {
  double acc = bias ? (double)bias[o] : 0.0;
  double mag = bias ? fabs((double)bias[o]) : 0.0;
  for (int i = 0; i < Ci; ++i) {
    int32_t p = pat[(size_t)o * Ci + i];
    if (p < 0) continue;
    for (int q = 0; q < 4; ++q) {
      int t = taps[4 * p + q];
      int ky = t / 3, kx = t % 3;
      double term = (double)w[((size_t)o * Ci + i) * 9 + t] * x_at(x, Ci, H, W, n, i, r + ky - 1, c + kx - 1);
      acc += term;
      mag += fabs(term);
    }
  }
  *y = acc;
  *s = mag;
}

/*
 * Pruned convolution over the whole output (the definition, fp64).
 *   x [N][Ci][H][W], w [Co][Ci][9], pat [Co][Ci] (from oracle_pattern_ids),
 *   bias [Co] or NULL; y, s [N][Co][H][W].
 */
void oracle_conv_pruned(const float* x, int N, int Ci, int H, int W, const float* w, const int32_t* pat,
                        const uint8_t* taps, const float* bias, int Co, double* y, double* s) {
#pragma omp parallel for collapse(2) schedule(dynamic, 1)
  for (int n = 0; n < N; ++n)
    for (int o = 0; o < Co; ++o)
      for (int r = 0; r < H; ++r)
        for (int c = 0; c < W; ++c) {
          size_t idx = (((size_t)n * Co + o) * H + r) * W + c;
          one_output_pruned(x, Ci, H, W, w, pat, taps, bias, n, o, r, c, &y[idx], &s[idx]);
        }
}

/* The same definition at a list of output points pts[k] = (n, o, r, c). */
void oracle_conv_pruned_points(const float* x, int N, int Ci, int H, int W, const float* w, const int32_t* pat,
                               const uint8_t* taps, const float* bias, int Co, int64_t npts, const int64_t* pts,
                               double* y, double* s) {
  (void)N;
  (void)Co;
#pragma omp parallel for schedule(dynamic, 64)
  for (int64_t k = 0; k < npts; ++k)
    one_output_pruned(x, Ci, H, W, w, pat, taps, bias, (int)pts[4 * k], (int)pts[4 * k + 1], (int)pts[4 * k + 2],
                      (int)pts[4 * k + 3], &y[k], &s[k]);
}

/*
 * Dense 3x3 convolution over all 9 taps of every (o, i) kernel, fp64: the
 * plain definition for an unpruned layer, and the brute-force form of a pruned
 * one when w already holds zeros outside the kept taps.
 */
void oracle_conv_dense(const float* x, int N, int Ci, int H, int W, const float* w, const float* bias, int Co,
                       double* y, double* s) {
#pragma omp parallel for collapse(2) schedule(dynamic, 1)
  for (int n = 0; n < N; ++n)
    for (int o = 0; o < Co; ++o)
      for (int r = 0; r < H; ++r)
        for (int c = 0; c < W; ++c) {
          double acc = bias ? (double)bias[o] : 0.0;
          double mag = bias ? fabs((double)bias[o]) : 0.0;
          for (int i = 0; i < Ci; ++i)
            for (int ky = 0; ky < 3; ++ky)
              for (int kx = 0; kx < 3; ++kx) {
                double term = (double)w[((size_t)o * Ci + i) * 9 + 3 * ky + kx] *
                              x_at(x, Ci, H, W, n, i, r + ky - 1, c + kx - 1);
                acc += term;
                mag += fabs(term);
              }
          size_t idx = (((size_t)n * Co + o) * H + r) * W + c;
          y[idx] = acc;
          s[idx] = mag;
        }
}

/* Dense convolution at a list of output points pts[k] = (n, o, r, c). */
void oracle_conv_dense_points(const float* x, int N, int Ci, int H, int W, const float* w, const float* bias,
                              int Co, int64_t npts, const int64_t* pts, double* y, double* s) {
  (void)N;
  (void)Co;
#pragma omp parallel for schedule(dynamic, 64)
  for (int64_t k = 0; k < npts; ++k) {
    int n = (int)pts[4 * k], o = (int)pts[4 * k + 1], r = (int)pts[4 * k + 2], c = (int)pts[4 * k + 3];
    double acc = bias ? (double)bias[o] : 0.0;
    double mag = bias ? fabs((double)bias[o]) : 0.0;
    for (int i = 0; i < Ci; ++i)
      for (int t = 0; t < 9; ++t) {
        double term = (double)w[((size_t)o * Ci + i) * 9 + t] * x_at(x, Ci, H, W, n, i, r + t / 3 - 1, c + t % 3 - 1);
        acc += term;
        mag += fabs(term);
      }
    y[k] = acc;
    s[k] = mag;
  }
}

/* Epilogue steps (Section 3 fuses convolution with its activation; the
 * residual add and the 2x2 max pool are the network-level operations of the
 * workloads).  ReLU is 1-Lipschitz, so the budget s is unchanged by it. */
void oracle_relu(double* y, int64_t n) {
  for (int64_t k = 0; k < n; ++k)
    if (y[k] < 0.0) y[k] = 0.0;
}

/* y += skip; the budget grows by |skip|. */
void oracle_add(double* y, double* s, const float* skip, int64_t n) {
  for (int64_t k = 0; k < n; ++k) {
    y[k] += (double)skip[k];
    s[k] += fabs((double)skip[k]);
  }
}

/* 2x2 max pool, stride 2 (floor), over [N*C][H][W]; the budget of a pooled
 * output is the largest budget in its window. */
void oracle_pool2(const double* y, const double* s, int64_t NC, int H, int W, double* y2, double* s2) {
  int H2 = H / 2, W2 = W / 2;
  for (int64_t m = 0; m < NC; ++m)
    for (int r = 0; r < H2; ++r)
      for (int c = 0; c < W2; ++c) {
        double best = -INFINITY, bs = 0.0;
        for (int dy = 0; dy < 2; ++dy)
          for (int dx = 0; dx < 2; ++dx) {
            size_t idx = ((size_t)m * H + 2 * r + dy) * W + 2 * c + dx;
            if (y[idx] > best) best = y[idx];
            if (s[idx] > bs) bs = s[idx];
          }
        size_t o = ((size_t)m * H2 + r) * W2 + c;
        y2[o] = best;
        s2[o] = bs;
      }
}
