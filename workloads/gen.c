/*
 * Seeded synthetic inputs for the four composite sparse expressions.
 *
 * This file holds random-number generation and sparse-structure construction
 * only (CSR / CSF index arrays and dense fp32 operand fills).  It contains none
 * of the expressions' arithmetic; both the CPU oracle and the CUDA library
 * consume what it produces.  Everything is plain C99 with fixed-width integer
 * arithmetic, so x86-64 and aarch64 hosts produce identical arrays for the same
 * seed (the only libm calls are log/cos/sqrt in the normal sampler and pow in
 * the Zipf weights; their results are rounded to fp32 or used only as sampling
 * thresholds).
 *
 * Generators (all published algorithms, restated here):
 *   splitmix64 (seeding) and xoshiro256** (stream), Vigna 2018;
 *   Lemire's multiply-shift reduction for bounded integers;
 *   Floyd's algorithm for m distinct values out of n;
 *   R-MAT recursive quadrant choice (Chakrabarti, Zhan, Faloutsos 2004);
 *   Box-Muller for N(0,1).
 * The sparse tensors mimic the paper's workloads (Sec. 6, Table 1): power-law
 * graphs in CSR, and 3-way tensors in CSF with skewed slices or fibers.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

typedef struct {
  uint64_t s[4];
} wl_rng;

static uint64_t splitmix64(uint64_t *x) {
  uint64_t z = (*x += 0x9E3779B97F4A7C15ULL);
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
  return z ^ (z >> 31);
}

void wl_seed(wl_rng *r, uint64_t seed) {
  uint64_t x = seed;
  for (int i = 0; i < 4; ++i) r->s[i] = splitmix64(&x);
}

static inline uint64_t rotl64(uint64_t x, int k) { return (x << k) | (x >> (64 - k)); }

uint64_t wl_next(wl_rng *r) {
  uint64_t *s = r->s;
  const uint64_t out = rotl64(s[1] * 5u, 7) * 9u;
  const uint64_t t = s[1] << 17;
  s[2] ^= s[0];
  s[3] ^= s[1];
  s[1] ^= s[2];
  s[0] ^= s[3];
  s[2] ^= t;
  s[3] = rotl64(s[3], 45);
  return out;
}

/* Uniform integer in [0, n). */
static inline uint64_t wl_below(wl_rng *r, uint64_t n) {
  return (uint64_t)(((unsigned __int128)wl_next(r) * (unsigned __int128)n) >> 64);
}

/* Uniform double in [0, 1) with 53 random bits. */
static inline double wl_u01(wl_rng *r) { return (double)(wl_next(r) >> 11) * 0x1.0p-53; }

/* ------------------------------------------------------------------------ */
/* sorting helpers                                                          */

/* LSD radix sort of n 64-bit keys whose values are < 2^bits. */
static void radix_sort_u64(uint64_t *a, int64_t n, int bits, uint64_t *tmp) {
  int64_t cnt[256];
  uint64_t *src = a, *dst = tmp;
  for (int shift = 0; shift < bits; shift += 8) {
    memset(cnt, 0, sizeof(cnt));
    for (int64_t i = 0; i < n; ++i) cnt[(src[i] >> shift) & 255u]++;
    int64_t run = 0;
    for (int d = 0; d < 256; ++d) {
      int64_t c = cnt[d];
      cnt[d] = run;
      run += c;
    }
    for (int64_t i = 0; i < n; ++i) dst[cnt[(src[i] >> shift) & 255u]++] = src[i];
    uint64_t *t = src;
    src = dst;
    dst = t;
  }
  if (src != a) memcpy(a, src, (size_t)n * sizeof(uint64_t));
}

static int bits_for(uint64_t maxval) {
  int b = 0;
  while (b < 64 && (maxval >> b) != 0) ++b;
  return b == 0 ? 8 : b;
}

/* Sort ascending and drop duplicates; returns the new length. */
static int64_t sort_unique_u64(uint64_t *a, int64_t n, uint64_t universe, uint64_t *tmp) {
  if (n <= 0) return 0;
  radix_sort_u64(a, n, bits_for(universe), tmp);
  int64_t m = 1;
  for (int64_t i = 1; i < n; ++i)
    if (a[i] != a[m - 1]) a[m++] = a[i];
  return m;
}

static int cmp_i32(const void *x, const void *y) {
  int32_t a = *(const int32_t *)x, b = *(const int32_t *)y;
  return (a > b) - (a < b);
}

static void sort_small_i32(int32_t *a, int64_t n) {
  if (n < 32) {
    for (int64_t i = 1; i < n; ++i) {
      int32_t v = a[i];
      int64_t j = i - 1;
      while (j >= 0 && a[j] > v) {
        a[j + 1] = a[j];
        --j;
      }
      a[j + 1] = v;
    }
  } else {
    qsort(a, (size_t)n, sizeof(int32_t), cmp_i32);
  }
}

/* n distinct uniform draws from [0, universe), returned sorted in out[0..n).
 * Draw, sort, drop duplicates and redraw the shortfall until n distinct values
 * remain.  Intended for n well below universe. */
static void draw_distinct_sorted(wl_rng *r, uint64_t universe, int64_t n, uint64_t *out,
                                 uint64_t *tmp) {
  int64_t have = 0;
  while (have < n) {
    for (int64_t i = have; i < n; ++i) out[i] = wl_below(r, universe);
    have = sort_unique_u64(out, n, universe, tmp);
  }
}

/* Floyd's algorithm: m distinct values out of [0, n), sorted ascending into
 * out.  bitmap holds n bits, all zero on entry and on exit. */
static void floyd_sorted(wl_rng *r, int32_t n, int32_t m, int32_t *out, uint64_t *bitmap) {
  int32_t k = 0;
  for (int32_t j = n - m; j < n; ++j) {
    int32_t t = (int32_t)wl_below(r, (uint64_t)j + 1u);
    int32_t pick = ((bitmap[t >> 6] >> (t & 63)) & 1u) ? j : t;
    bitmap[pick >> 6] |= 1ULL << (pick & 63);
    out[k++] = pick;
  }
  sort_small_i32(out, m);
  for (int32_t i = 0; i < m; ++i) bitmap[out[i] >> 6] &= ~(1ULL << (out[i] & 63));
}

/* ------------------------------------------------------------------------ */
/* dense operand fills                                                      */

/* U[a,b] with 24 random bits: a + (b-a) * m * 2^-24, m uniform in [0, 2^24). */
void wl_fill_uniform(wl_rng *r, int64_t n, float a, float b, float *out) {
  const double lo = a, span = (double)b - (double)a;
  for (int64_t i = 0; i < n; ++i)
    out[i] = (float)(lo + span * ((double)(wl_next(r) >> 40) * 0x1.0p-24));
}

/* N(0,1) by Box-Muller (cosine branch only), evaluated in double, rounded to fp32. */
void wl_fill_normal(wl_rng *r, int64_t n, float *out) {
  const double two_pi = 6.283185307179586476925286766559;
  for (int64_t i = 0; i < n; ++i) {
    double u1 = ((double)(wl_next(r) >> 11) + 1.0) * 0x1.0p-53; /* (0, 1] */
    double u2 = (double)(wl_next(r) >> 11) * 0x1.0p-53;          /* [0, 1) */
    out[i] = (float)(sqrt(-2.0 * log(u1)) * cos(two_pi * u2));
  }
}

void wl_fill_const(int64_t n, float v, float *out) {
  for (int64_t i = 0; i < n; ++i) out[i] = v;
}

/* ------------------------------------------------------------------------ */
/* CSR matrices                                                             */

/* Exactly per_row distinct uniform column coordinates in every row.
 * pos[nrows+1], crd[nrows*per_row].  Returns nnz or -1 on bad arguments. */
int64_t wl_uniform_csr(wl_rng *r, int32_t nrows, int32_t ncols, int32_t per_row, int32_t *pos,
                       int32_t *crd) {
  if (nrows < 0 || ncols <= 0 || per_row < 0 || per_row > ncols) return -1;
  uint64_t *bitmap = (uint64_t *)calloc(((size_t)ncols + 63) / 64, sizeof(uint64_t));
  if (!bitmap) return -1;
  pos[0] = 0;
  for (int32_t i = 0; i < nrows; ++i) {
    floyd_sorted(r, ncols, per_row, crd + (int64_t)i * per_row, bitmap);
    pos[i + 1] = (int32_t)((int64_t)(i + 1) * per_row);
  }
  free(bitmap);
  return (int64_t)nrows * per_row;
}

/* R-MAT graph with exactly nnz distinct edges on n vertices (n x n CSR).
 *
 * Each edge picks one of the four quadrants per level with probabilities
 * (a, b, c, 1-a-b-c), most significant bit first, over ceil(log2 n) levels.
 * An edge with an endpoint >= n is redrawn.  Duplicate edges are removed and
 * the shortfall is redrawn until nnz distinct edges remain.  No noise and no
 * vertex permutation: hub vertices keep the low ids.  Self loops are kept.
 * pos[n+1], crd[nnz].  Returns nnz, or -1 on bad arguments / no memory. */
int64_t wl_rmat_csr(wl_rng *r, int32_t n, int64_t nnz, double a, double b, double c,
                    int32_t *pos, int32_t *crd) {
  if (n <= 0 || nnz < 0 || (double)nnz > (double)n * (double)n) return -1;
  int scale = 0;
  while ((1LL << scale) < (int64_t)n) ++scale;
  const uint64_t ta = (uint64_t)(a * 4294967296.0);
  const uint64_t tab = (uint64_t)((a + b) * 4294967296.0);
  const uint64_t tabc = (uint64_t)((a + b + c) * 4294967296.0);
  uint64_t *keys = (uint64_t *)malloc((size_t)(nnz > 0 ? nnz : 1) * sizeof(uint64_t));
  uint64_t *tmp = (uint64_t *)malloc((size_t)(nnz > 0 ? nnz : 1) * sizeof(uint64_t));
  if (!keys || !tmp) {
    free(keys);
    free(tmp);
    return -1;
  }
  const uint64_t universe = ((uint64_t)n << 32);
  int64_t have = 0;
  while (have < nnz) {
    for (int64_t e = have; e < nnz; ++e) {
      uint64_t row, col;
      do {
        row = 0;
        col = 0;
        uint64_t x = 0;
        for (int lvl = 0; lvl < scale; ++lvl) {
          uint64_t u;
          if ((lvl & 1) == 0) {
            x = wl_next(r);
            u = x >> 32;
          } else {
            u = x & 0xFFFFFFFFULL;
          }
          uint64_t rb = 0, cb = 0;
          if (u < ta) {
          } else if (u < tab) {
            cb = 1;
          } else if (u < tabc) {
            rb = 1;
          } else {
            rb = 1;
            cb = 1;
          }
          row = (row << 1) | rb;
          col = (col << 1) | cb;
        }
      } while (row >= (uint64_t)n || col >= (uint64_t)n);
      keys[e] = (row << 32) | col;
    }
    have = sort_unique_u64(keys, nnz, universe, tmp);
  }
  int64_t p = 0;
  pos[0] = 0;
  for (int32_t i = 0; i < n; ++i) {
    while (p < nnz && (int64_t)(keys[p] >> 32) == (int64_t)i) {
      crd[p] = (int32_t)(keys[p] & 0xFFFFFFFFULL);
      ++p;
    }
    pos[i + 1] = (int32_t)p;
  }
  free(keys);
  free(tmp);
  return nnz;
}

/* ------------------------------------------------------------------------ */
/* CSF 3-tensors                                                            */
/*
 * Layout (three compressed levels, coordinates sorted within each parent):
 *   crd1[nslices]            slice coordinates i (ascending)
 *   pos2[nslices+1]          fiber range of each slice
 *   crd2[nfibers]            fiber coordinates j
 *   pos3[nfibers+1]          nonzero range of each fiber
 *   crd3[nnz]                leaf coordinates k
 */

typedef struct {
  double frac;
  int32_t rank;
} remainder_t;

static int cmp_remainder(const void *x, const void *y) {
  const remainder_t *a = (const remainder_t *)x, *b = (const remainder_t *)y;
  if (a->frac != b->frac) return a->frac < b->frac ? 1 : -1;
  return (a->rank > b->rank) - (a->rank < b->rank);
}

/* Slices with Zipf(s) rank-frequency sizes.
 *
 * Rank r (1-based, r <= d0) receives a share proportional to r^-s of the nnz,
 * rounded by the largest-remainder method, with at least one nonzero per rank
 * (taken back from rank 1) and at most d1*d2.  A seeded Fisher-Yates shuffle
 * maps ranks to slice ids.  Within each slice the (j,k) coordinates are
 * distinct and uniform over d1 x d2.  All d0 slices are non-empty.
 * Output capacities: crd1[d0], pos2[d0+1], crd2[nnz], pos3[nnz+1], crd3[nnz].
 * Returns the number of fibers, or -1 on bad arguments / no memory. */
int64_t wl_zipf_slices_csf(wl_rng *r, int32_t d0, int32_t d1, int32_t d2, int64_t nnz, double s,
                           int32_t *crd1, int32_t *pos2, int32_t *crd2, int32_t *pos3,
                           int32_t *crd3, int32_t *nslices_out) {
  if (d0 <= 0 || d1 <= 0 || d2 <= 0 || nnz < d0) return -1;
  const uint64_t plane = (uint64_t)d1 * (uint64_t)d2;
  if ((double)nnz > (double)d0 * (double)plane) return -1;
  double *w = (double *)malloc((size_t)d0 * sizeof(double));
  int64_t *cnt = (int64_t *)malloc((size_t)d0 * sizeof(int64_t));
  int32_t *order = (int32_t *)malloc((size_t)d0 * sizeof(int32_t));
  remainder_t *rem = (remainder_t *)malloc((size_t)d0 * sizeof(remainder_t));
  int32_t *perm = (int32_t *)malloc((size_t)d0 * sizeof(int32_t));
  int64_t *by_slice = (int64_t *)malloc((size_t)d0 * sizeof(int64_t));
  if (!w || !cnt || !order || !rem || !perm || !by_slice) goto fail;
  double W = 0.0;
  for (int32_t k = 0; k < d0; ++k) {
    w[k] = pow((double)(k + 1), -s);
    W += w[k];
  }
  int64_t total = 0;
  for (int32_t k = 0; k < d0; ++k) {
    double q = (double)nnz * w[k] / W;
    cnt[k] = (int64_t)floor(q);
    rem[k].frac = q - (double)cnt[k];
    rem[k].rank = k;
    total += cnt[k];
  }
  /* largest remainder: ranks by fractional part, descending (ties: lower rank) */
  qsort(rem, (size_t)d0, sizeof(rem[0]), cmp_remainder);
  for (int32_t k = 0; k < d0; ++k) order[k] = rem[k].rank;
  for (int64_t k = 0; k < nnz - total && k < d0; ++k) cnt[order[k]]++;
  for (int32_t k = 1; k < d0; ++k)
    if (cnt[k] == 0) {
      cnt[k] = 1;
      cnt[0]--;
    }
  for (int32_t k = 0; k < d0; ++k)
    if ((uint64_t)cnt[k] > plane) goto fail;
  /* rank -> slice id */
  for (int32_t k = 0; k < d0; ++k) perm[k] = k;
  for (int32_t k = d0 - 1; k > 0; --k) {
    int32_t t = (int32_t)wl_below(r, (uint64_t)k + 1u);
    int32_t x = perm[k];
    perm[k] = perm[t];
    perm[t] = x;
  }
  int64_t maxc = 0;
  for (int32_t k = 0; k < d0; ++k) {
    by_slice[perm[k]] = cnt[k];
    if (cnt[k] > maxc) maxc = cnt[k];
  }
  uint64_t *codes = (uint64_t *)malloc((size_t)maxc * sizeof(uint64_t));
  uint64_t *tmp = (uint64_t *)malloc((size_t)maxc * sizeof(uint64_t));
  if (!codes || !tmp) {
    free(codes);
    free(tmp);
    goto fail;
  }
  int64_t nf = 0, p = 0;
  pos2[0] = 0;
  pos3[0] = 0;
  for (int32_t i = 0; i < d0; ++i) {
    int64_t m = by_slice[i];
    draw_distinct_sorted(r, plane, m, codes, tmp);
    crd1[i] = i;
    int64_t prev_j = -1;
    for (int64_t e = 0; e < m; ++e) {
      int64_t j = (int64_t)(codes[e] / (uint64_t)d2);
      int64_t k = (int64_t)(codes[e] % (uint64_t)d2);
      if (j != prev_j) {
        if (prev_j >= 0) pos3[nf] = (int32_t)p;
        crd2[nf++] = (int32_t)j;
        prev_j = j;
      }
      crd3[p++] = (int32_t)k;
    }
    pos3[nf] = (int32_t)p;
    pos2[i + 1] = (int32_t)nf;
  }
  *nslices_out = d0;
  free(codes);
  free(tmp);
  free(w);
  free(cnt);
  free(order);
  free(rem);
  free(perm);
  free(by_slice);
  return nf;
fail:
  free(w);
  free(cnt);
  free(order);
  free(rem);
  free(perm);
  free(by_slice);
  return -1;
}

/* Exponent s of a Zipf law truncated to {1..max_len} whose mean is mean_len
 * (bisection; the mean decreases in s). */
double wl_zipf_exponent_for_mean(int32_t max_len, double mean_len) {
  double lo = 0.0, hi = 8.0;
  for (int it = 0; it < 200; ++it) {
    double mid = 0.5 * (lo + hi), num = 0.0, den = 0.0;
    for (int32_t k = 1; k <= max_len; ++k) {
      double pk = pow((double)k, -mid);
      num += (double)k * pk;
      den += pk;
    }
    if (num / den > mean_len)
      lo = mid;
    else
      hi = mid;
  }
  return 0.5 * (lo + hi);
}

/* Fibers with power-law lengths.
 *
 * Fiber lengths follow a Zipf law truncated to {1..max_len} whose exponent is
 * solved so that the mean is mean_len.  Lengths are drawn until their sum
 * reaches nnz (the last one is cut).  The fibers' (i,j) coordinates are
 * distinct and uniform over d0 x d1; the leaves of each fiber are distinct and
 * uniform over [0, d2).  max_len must not exceed d2.
 * Output capacities: crd1[d0], pos2[d0+1], crd2[nnz], pos3[nnz+1], crd3[nnz].
 * Returns the number of fibers, or -1 on bad arguments / no memory. */
int64_t wl_powerlaw_fibers_csf(wl_rng *r, int32_t d0, int32_t d1, int32_t d2, int64_t nnz,
                               double mean_len, int32_t max_len, int32_t *crd1, int32_t *pos2,
                               int32_t *crd2, int32_t *pos3, int32_t *crd3,
                               int32_t *nslices_out) {
  if (d0 <= 0 || d1 <= 0 || d2 <= 0 || nnz <= 0 || max_len <= 0 || max_len > d2) return -1;
  const double s = wl_zipf_exponent_for_mean(max_len, mean_len);
  double *cdf = (double *)malloc((size_t)max_len * sizeof(double));
  int32_t *len = (int32_t *)malloc((size_t)nnz * sizeof(int32_t));
  if (!cdf || !len) {
    free(cdf);
    free(len);
    return -1;
  }
  double run = 0.0;
  for (int32_t k = 1; k <= max_len; ++k) {
    run += pow((double)k, -s);
    cdf[k - 1] = run;
  }
  int64_t nf = 0, total = 0;
  while (total < nnz) {
    double u = wl_u01(r) * run;
    int32_t lo = 0, hi = max_len - 1; /* first k with cdf[k] > u */
    while (lo < hi) {
      int32_t mid = (lo + hi) >> 1;
      if (cdf[mid] > u)
        hi = mid;
      else
        lo = mid + 1;
    }
    int64_t l = (int64_t)lo + 1;
    if (total + l > nnz) l = nnz - total;
    len[nf++] = (int32_t)l;
    total += l;
  }
  free(cdf);
  const uint64_t plane = (uint64_t)d0 * (uint64_t)d1;
  if ((uint64_t)nf > plane / 2u) {
    free(len);
    return -1;
  }
  uint64_t *codes = (uint64_t *)malloc((size_t)nf * sizeof(uint64_t));
  uint64_t *tmp = (uint64_t *)malloc((size_t)nf * sizeof(uint64_t));
  uint64_t *bitmap = (uint64_t *)calloc(((size_t)d2 + 63) / 64, sizeof(uint64_t));
  if (!codes || !tmp || !bitmap) {
    free(codes);
    free(tmp);
    free(bitmap);
    free(len);
    return -1;
  }
  draw_distinct_sorted(r, plane, nf, codes, tmp);
  int64_t ns = 0, p = 0;
  int64_t prev_i = -1;
  pos3[0] = 0;
  for (int64_t f = 0; f < nf; ++f) {
    int64_t i = (int64_t)(codes[f] / (uint64_t)d1);
    int64_t j = (int64_t)(codes[f] % (uint64_t)d1);
    if (i != prev_i) {
      crd1[ns] = (int32_t)i;
      pos2[ns] = (int32_t)f;
      ++ns;
      prev_i = i;
    }
    crd2[f] = (int32_t)j;
    floyd_sorted(r, d2, len[f], crd3 + p, bitmap);
    p += len[f];
    pos3[f + 1] = (int32_t)p;
  }
  pos2[ns] = (int32_t)nf;
  *nslices_out = (int32_t)ns;
  free(codes);
  free(tmp);
  free(bitmap);
  free(len);
  return nf;
}
