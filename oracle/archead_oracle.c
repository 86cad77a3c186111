/*
 * ARCHead packed LM-head forward: plain fp64 CPU oracle.
 *
 * TEST INFRASTRUCTURE.  Only the test suite, the package smoke check and the
 * benchmark's CPU-baseline leg may load or call this library.  It shares no
 * code, header, table or helper with the CUDA path: it has its own nibble
 * unpacking, its own fp16/bf16 decoders and its own loops.
 *
 * What it computes (paper, Section 3.2, Eqs. 3, 6 and 7):
 *
 *   W_hat[n,k] = code[n,k] * s_R[n, k/g]                       (INT4 residual)
 *              + sum_j (qU[n,j] sU[j]) * (qV[k,j] sV[j])          (core A_c B_c)
 *              + sum_j (qA[n,j] sA[n]) * (qB[k,j] sB[k/g, j])     (correction A_w B_w)
 *   y[m,n]     = sum_k x[m,k] * W_hat[n,k]
 *   ce[m]      = log sum_n exp(y[m,n]) - y[m, t_m]                (Section 4, CE)
 *
 * Everything is evaluated in double precision exactly as written: a dense
 * fp64 row of W_hat is formed, then dotted with every token.  There is no
 * blocking or reordering beyond processing one vocabulary row at a time.
 *
 * Readings where the paper is silent (stated once here, used throughout):
 *  - INT4 codes are two's complement, packed along d, low nibble = even k.
 *  - All quantisers are symmetric (no zero points); scales are IEEE fp16.
 *  - A_w is quantised per row (one scale per vocabulary row) and B_w per
 *    (d-group of size g, rank column); the core factors per column.
 *
 * Two stored formats.  "int8" (format 0): INT8 core left codes and one fp16
 * scale per residual group.  "sc4" (format 1), the paper's own format
 * (Section 3.2, Eq. 3: Q_5 core left factor, SC4 residual with quantised
 * group scales; Appendix C, packed state dictionary):
 *  - core left codes are 5-bit two's complement (-16..15); row n stores its
 *    r_c codes in ceil(5 r_c / 8) bytes, code j in bits 5j..5j+4 of the row's
 *    bytes taken as one little-endian bit string;
 *  - a residual group scale is s_row[n] * (q + 1), with q a 4-bit unsigned
 *    code (two per byte, low nibble = even group) and s_row one fp16 per row.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

typedef struct {
  int64_t V, d;
  int32_t core_rank, corr_rank, group_size, format; /* format: 0 int8, 1 sc4 */
  const uint8_t *res_codes;      /* V x d/2                       */
  const uint16_t *res_scales;    /* V x d/g   fp16 bits   (int8)  */
  const int8_t *core_u;          /* V x r_c               (int8)  */
  const uint16_t *core_u_scale;  /* r_c       fp16 bits           */
  const int8_t *core_v;          /* d x r_c                       */
  const uint16_t *core_v_scale;  /* r_c       fp16 bits           */
  const int8_t *corr_a;          /* V x r_r                       */
  const uint16_t *corr_a_scale;  /* V         fp16 bits           */
  const int8_t *corr_b;          /* d x r_r                       */
  const uint16_t *corr_b_scale;  /* d/g x r_r fp16 bits           */
  const uint8_t *res_scale_codes; /* V x ceil(G/2), 4-bit codes (sc4) */
  const uint16_t *res_row_scale;  /* V         fp16 bits     (sc4) */
  const uint8_t *core_u5;         /* V x ceil(5 r_c/8)       (sc4) */
} oracle_head;

/* IEEE-754 binary16: 1 sign bit, 5 exponent bits (bias 15), 10 fraction bits. */
double oracle_fp16_value(uint16_t h) {
  int sign = (h >> 15) & 1;
  int e = (h >> 10) & 0x1F;
  int f = h & 0x3FF;
  double v;
  if (e == 0) {
    v = ldexp((double)f, -24);                 /* subnormal: f * 2^-14 * 2^-10 */
  } else if (e == 31) {
    v = f ? NAN : INFINITY;
  } else {
    v = ldexp((double)(1024 + f), e - 25);     /* (1 + f/1024) * 2^(e-15) */
  }
  return sign ? -v : v;
}

/* bfloat16: 1 sign bit, 8 exponent bits (bias 127), 7 fraction bits. */
double oracle_bf16_value(uint16_t b) {
  int sign = (b >> 15) & 1;
  int e = (b >> 7) & 0xFF;
  int f = b & 0x7F;
  double v;
  if (e == 0) {
    v = ldexp((double)f, -133);                /* f * 2^-126 * 2^-7 */
  } else if (e == 255) {
    v = f ? NAN : INFINITY;
  } else {
    v = ldexp((double)(128 + f), e - 134);     /* (1 + f/128) * 2^(e-127) */
  }
  return sign ? -v : v;
}

/* Signed INT4 code k of a packed row: byte k/2, low nibble for even k. */
int oracle_int4_code(const uint8_t *row, int64_t k) {
  int byte = row[k / 2];
  int nib = (k % 2 == 0) ? (byte & 0x0F) : ((byte >> 4) & 0x0F);
  return nib >= 8 ? nib - 16 : nib;
}

/* Signed 5-bit code j of a row of packed bytes: bits 5j..5j+4, bit b of the
 * row being bit b%8 of byte b/8; two's complement over 5 bits. */
int oracle_int5_code(const uint8_t *row, int64_t j) {
  int v = 0;
  for (int b = 0; b < 5; ++b) {
    int64_t bit = 5 * j + b;
    v |= ((row[bit / 8] >> (bit % 8)) & 1) << b;
  }
  return v >= 16 ? v - 32 : v;
}

/* 4-bit unsigned group-scale code of group grp: byte grp/2, low nibble for even grp. */
int oracle_scale_code(const uint8_t *row, int64_t grp) {
  int byte = row[grp / 2];
  return (grp % 2 == 0) ? (byte & 0x0F) : ((byte >> 4) & 0x0F);
}

/* Residual group scale s_R[n, grp] of either format. */
static double res_scale(const oracle_head *h, int64_t n, int64_t grp) {
  const int64_t G = h->d / h->group_size;
  if (h->format == 1) {
    const int64_t nb = (G + 1) / 2;
    return oracle_fp16_value(h->res_row_scale[n]) * (double)(oracle_scale_code(h->res_scale_codes + n * nb, grp) + 1);
  }
  return oracle_fp16_value(h->res_scales[n * G + grp]);
}

/* Core left code qU[n, j] of either format. */
static int core_u_code(const oracle_head *h, int64_t n, int j) {
  if (h->format == 1) return oracle_int5_code(h->core_u5 + n * ((5 * (int64_t)h->core_rank + 7) / 8), j);
  return h->core_u[n * h->core_rank + j];
}

void oracle_unpack_int5(const uint8_t *in, int64_t rows, int64_t rank, int8_t *out) {
  const int64_t nb = (5 * rank + 7) / 8;
  for (int64_t r = 0; r < rows; ++r)
    for (int64_t j = 0; j < rank; ++j) out[r * rank + j] = (int8_t)oracle_int5_code(in + r * nb, j);
}

void oracle_unpack_scale_codes(const uint8_t *in, int64_t rows, int64_t groups, int8_t *out) {
  const int64_t nb = (groups + 1) / 2;
  for (int64_t r = 0; r < rows; ++r)
    for (int64_t j = 0; j < groups; ++j) out[r * groups + j] = (int8_t)oracle_scale_code(in + r * nb, j);
}

void oracle_fp16_values(const uint16_t *in, int64_t n, double *out) {
  for (int64_t i = 0; i < n; ++i) out[i] = oracle_fp16_value(in[i]);
}

void oracle_bf16_values(const uint16_t *in, int64_t n, double *out) {
  for (int64_t i = 0; i < n; ++i) out[i] = oracle_bf16_value(in[i]);
}

void oracle_unpack_int4(const uint8_t *in, int64_t ncodes, int8_t *out) {
  for (int64_t k = 0; k < ncodes; ++k) out[k] = (int8_t)oracle_int4_code(in, k);
}

static int check_head(const oracle_head *h) {
  if (!h || h->V < 1 || h->d < 2 || h->group_size < 1) return -1;
  if (h->d % 2 != 0 || h->d % h->group_size != 0) return -1;
  if (h->core_rank < 0 || h->corr_rank < 0) return -1;
  if (h->format != 0 && h->format != 1) return -1;
  return 0;
}

/*
 * Dequantised d-side factors, decoded once per call and shared by all rows:
 *   vdq[k*r_c + j] = qV[k,j] * sV[j]          (core right factor)
 *   bdq[k*r_r + j] = qB[k,j] * sB[k/g, j]     (correction right factor)
 *   su[j]          = sU[j]                     (core left column scales)
 */
typedef struct {
  double *vdq, *bdq, *su;
} side_cache;

static void free_cache(side_cache *c) {
  free(c->vdq);
  free(c->bdq);
  free(c->su);
}

static int make_cache(const oracle_head *h, side_cache *c) {
  const int64_t d = h->d;
  const int g = h->group_size, rc = h->core_rank, rr = h->corr_rank;
  c->vdq = (double *)malloc(sizeof(double) * (size_t)(d * rc + 1));
  c->bdq = (double *)malloc(sizeof(double) * (size_t)(d * rr + 1));
  c->su = (double *)malloc(sizeof(double) * (size_t)(rc + 1));
  if (!c->vdq || !c->bdq || !c->su) {
    free_cache(c);
    return -2;
  }
  for (int j = 0; j < rc; ++j) c->su[j] = oracle_fp16_value(h->core_u_scale[j]);
  for (int64_t k = 0; k < d; ++k) {
    for (int j = 0; j < rc; ++j)
      c->vdq[k * rc + j] = (double)h->core_v[k * rc + j] * oracle_fp16_value(h->core_v_scale[j]);
    for (int j = 0; j < rr; ++j)
      c->bdq[k * rr + j] = (double)h->corr_b[k * rr + j] * oracle_fp16_value(h->corr_b_scale[(k / g) * rr + j]);
  }
  return 0;
}

/*
 * Dense fp64 row n of W_hat (Eq. 6 with W_d from Eq. 3), written to w[0..d).
 * u and a are scratch rows of r_c and r_r doubles.
 */
static void dequant_row(const oracle_head *h, const side_cache *c, int64_t n, double *w, double *u, double *a) {
  const int64_t d = h->d;
  const int g = h->group_size, rc = h->core_rank, rr = h->corr_rank;
  const uint8_t *codes = h->res_codes + n * (d / 2);
  for (int j = 0; j < rc; ++j) u[j] = (double)core_u_code(h, n, j) * c->su[j];
  double s_a = rr > 0 ? oracle_fp16_value(h->corr_a_scale[n]) : 0.0;
  for (int j = 0; j < rr; ++j) a[j] = (double)h->corr_a[n * rr + j] * s_a;
  for (int64_t k = 0; k < d; ++k) {
    double s_r = res_scale(h, n, k / g);
    double v = (double)oracle_int4_code(codes, k) * s_r;
    double core = 0.0;
    for (int j = 0; j < rc; ++j) core += u[j] * c->vdq[k * rc + j];
    double corr = 0.0;
    for (int j = 0; j < rr; ++j) corr += a[j] * c->bdq[k * rr + j];
    w[k] = v + core + corr;
  }
}

/* Per-thread scratch: one dense row plus the two left-factor rows. */
static double *row_scratch(const oracle_head *h) {
  return (double *)malloc(sizeof(double) * (size_t)(h->d + h->core_rank + h->corr_rank + 1));
}

int oracle_dequant_rows(const oracle_head *h, int64_t row0, int64_t nrows, double *out) {
  if (check_head(h) || row0 < 0 || nrows < 0 || row0 + nrows > h->V) return -1;
  side_cache c;
  if (make_cache(h, &c)) return -2;
  int failed = 0;
#pragma omp parallel
  {
    double *scr = row_scratch(h);
    if (!scr) {
#pragma omp atomic write
      failed = 1;
    }
#pragma omp for schedule(static)
    for (int64_t i = 0; i < nrows; ++i) {
      if (!scr) continue;
      double *u = scr + h->d, *a = u + h->core_rank;
      dequant_row(h, &c, row0 + i, scr, u, a);
      memcpy(out + i * h->d, scr, sizeof(double) * (size_t)h->d);
    }
    free(scr);
  }
  free_cache(&c);
  return failed ? -2 : 0;
}

/*
 * One stored component, dequantised element by element as code * scale:
 *   0: residual      [nrows x d]    code[n,k] * s_R[n,k/g]
 *   1: core left     [nrows x r_c]  qU[n,j] * sU[j]
 *   2: core right    [nrows x r_c]  qV[k,j] * sV[j]         (rows are k)
 *   3: corr left     [nrows x r_r]  qA[n,j] * sA[n]
 *   4: corr right    [nrows x r_r]  qB[k,j] * sB[k/g,j]     (rows are k)
 */
int oracle_component(const oracle_head *h, int comp, int64_t row0, int64_t nrows, double *out) {
  if (check_head(h) || row0 < 0 || nrows < 0) return -1;
  const int64_t d = h->d;
  const int g = h->group_size, rc = h->core_rank, rr = h->corr_rank;
  int64_t limit = (comp == 2 || comp == 4) ? d : h->V;
  if (comp < 0 || comp > 4 || row0 + nrows > limit) return -1;
  for (int64_t i = 0; i < nrows; ++i) {
    int64_t r = row0 + i;
    if (comp == 0) {
      for (int64_t k = 0; k < d; ++k)
        out[i * d + k] = (double)oracle_int4_code(h->res_codes + r * (d / 2), k) * res_scale(h, r, k / g);
    } else if (comp == 1) {
      for (int j = 0; j < rc; ++j)
        out[i * rc + j] = (double)core_u_code(h, r, j) * oracle_fp16_value(h->core_u_scale[j]);
    } else if (comp == 2) {
      for (int j = 0; j < rc; ++j)
        out[i * rc + j] = (double)h->core_v[r * rc + j] * oracle_fp16_value(h->core_v_scale[j]);
    } else if (comp == 3) {
      for (int j = 0; j < rr; ++j)
        out[i * rr + j] = (double)h->corr_a[r * rr + j] * oracle_fp16_value(h->corr_a_scale[r]);
    } else {
      for (int j = 0; j < rr; ++j)
        out[i * rr + j] = (double)h->corr_b[r * rr + j] *
                          oracle_fp16_value(h->corr_b_scale[(r / g) * rr + j]);
    }
  }
  return 0;
}

/*
 * Logits of vocabulary rows [row0, row0+nrows) for M tokens (Eq. 7):
 *   y[m * nrows + (n - row0)] = sum_k x[m,k] * W_hat[n,k].
 * x holds bf16 bit patterns, row-major [M x d].
 */
int oracle_logits(const oracle_head *h, const uint16_t *x_bits, int64_t M, int64_t row0,
                  int64_t nrows, double *y) {
  if (check_head(h) || M < 0 || row0 < 0 || nrows < 0 || row0 + nrows > h->V) return -1;
  const int64_t d = h->d;
  double *x = (double *)malloc(sizeof(double) * (size_t)(M * d + 1));
  if (!x) return -2;
  oracle_bf16_values(x_bits, M * d, x);
  side_cache c;
  if (make_cache(h, &c)) {
    free(x);
    return -2;
  }
  int failed = 0;
#pragma omp parallel
  {
    double *w = row_scratch(h);
    if (!w) {
#pragma omp atomic write
      failed = 1;
    }
#pragma omp for schedule(dynamic, 16)
    for (int64_t i = 0; i < nrows; ++i) {
      if (!w) continue;
      dequant_row(h, &c, row0 + i, w, w + d, w + d + h->core_rank);
      for (int64_t m = 0; m < M; ++m) {
        double acc = 0.0;
        for (int64_t k = 0; k < d; ++k) acc += x[m * d + k] * w[k];
        y[m * nrows + i] = acc;
      }
    }
    free(w);
  }
  free_cache(&c);
  free(x);
  return failed ? -2 : 0;
}

/*
 * Per-token cross entropy over the full vocabulary (natural log):
 *   ce[m] = max_n y + log sum_n exp(y[m,n] - max_n y) - y[m, t_m].
 * Also returns the argmax (lowest index among equal maxima), the gap between
 * the largest and second-largest logit, and the target logit.  A target
 * outside [0, V) yields ce = NaN and the call returns 1.
 */
int oracle_ce(const oracle_head *h, const uint16_t *x_bits, int64_t M, const int32_t *targets,
              double *ce, int64_t *argmax, double *top2_gap, double *target_logit) {
  if (check_head(h) || M < 0) return -1;
  const int64_t V = h->V;
  double *y = (double *)malloc(sizeof(double) * (size_t)(M * V + 1));
  if (!y) return -2;
  int rc = oracle_logits(h, x_bits, M, 0, V, y);
  if (rc) {
    free(y);
    return rc;
  }
  int bad_target = 0;
  for (int64_t m = 0; m < M; ++m) {
    const double *row = y + m * V;
    double mx = row[0];
    int64_t arg = 0;
    for (int64_t n = 1; n < V; ++n)
      if (row[n] > mx) { mx = row[n]; arg = n; }
    double second = -INFINITY;
    for (int64_t n = 0; n < V; ++n)
      if (n != arg && row[n] > second) second = row[n];
    double s = 0.0;
    for (int64_t n = 0; n < V; ++n) s += exp(row[n] - mx);
    double lse = mx + log(s);
    int32_t t = targets[m];
    if (t < 0 || t >= V) {
      bad_target = 1;
      ce[m] = NAN;
      if (target_logit) target_logit[m] = NAN;
    } else {
      ce[m] = lse - row[t];
      if (target_logit) target_logit[m] = row[t];
    }
    if (argmax) argmax[m] = arg;
    if (top2_gap) top2_gap[m] = V > 1 ? mx - second : INFINITY;
  }
  free(y);
  return bad_target;
}

/*
 * Persistent storage of the packed head (Section 3.3, Eq. 10): the sum of
 * numel * element_size over the stored components.  Two INT4 codes share one
 * byte; every scale is a 2-byte fp16; every factor code one byte.
 */
int64_t oracle_packed_bytes(int64_t V, int64_t d, int64_t rc, int64_t rr, int64_t g) {
  int64_t G = d / g;
  int64_t bytes = 0;
  bytes += V * d / 2;      /* residual codes        */
  bytes += V * G * 2;      /* residual group scales */
  bytes += V * rc;         /* core left codes       */
  bytes += rc * 2;         /* core left scales      */
  bytes += d * rc;         /* core right codes      */
  bytes += rc * 2;         /* core right scales     */
  bytes += V * rr;         /* correction left codes */
  if (rr > 0) bytes += V * 2; /* correction row scales (absent when r_r = 0) */
  bytes += d * rr;         /* correction right codes*/
  bytes += G * rr * 2;     /* correction group scales */
  return bytes;
}

/*
 * The same sum for the sc4 format: 4-bit group-scale codes (two per byte)
 * plus one fp16 row scale replace the fp16 group scales, and the core left
 * factor takes ceil(5 r_c / 8) bytes per row.
 */
int64_t oracle_packed_bytes_sc4(int64_t V, int64_t d, int64_t rc, int64_t rr, int64_t g) {
  int64_t G = d / g;
  int64_t bytes = 0;
  bytes += V * d / 2;            /* residual codes                  */
  bytes += V * ((G + 1) / 2);    /* residual group-scale codes      */
  bytes += V * 2;                /* residual row scales             */
  bytes += V * ((5 * rc + 7) / 8); /* core left codes, 5-bit        */
  bytes += rc * 2;               /* core left scales                */
  bytes += d * rc;               /* core right codes                */
  bytes += rc * 2;               /* core right scales               */
  bytes += V * rr;               /* correction left codes           */
  if (rr > 0) bytes += V * 2;    /* correction row scales           */
  bytes += d * rr;               /* correction right codes          */
  bytes += G * rr * 2;           /* correction group scales         */
  return bytes;
}

/* The dense BF16 head the packed module replaces: V * d * 2 bytes. */
int64_t oracle_dense_bf16_bytes(int64_t V, int64_t d) { return V * d * 2; }

int oracle_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}
