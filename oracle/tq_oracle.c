/*
 * tq_oracle.c - plain CPU oracle of the packed ternary linear layer.
 *
 * TEST INFRASTRUCTURE ONLY.  Only the tests, the smoke check of
 * __graft_entry__ and the CPU-baseline leg of bench.py may load this file's
 * library.  It shares no code, header or table with the CUDA path (it does
 * not include tq.h): every constant below is re-derived here from the paper.
 *
 * What it follows:
 *   - trit information content and the base-3 byte (paper eq. b_T,
 *     "Introduction": one ternary symbol carries log2(3) bits; five of them
 *     fit one byte since 3^5 = 243 <= 256);
 *   - lossless lattice-aware serialization of the discrete supports and
 *     their parameters (paper "Packing: From Quantization to Serialization");
 *   - reconstruction W-hat = offset + alpha0 T0 + alpha1 T1 on the salient
 *     part (paper "Model and Representation", eq. W-hat), read per group of
 *     128 along K: W = s1 T1 + off + sal s2 T2;
 *   - the weight-only A16 linear y = x W^T (paper "Model and Representation":
 *     activations stay fp16), computed here as the plain definition:
 *     dense fp64 reconstruction of one row, then a naive dot product.
 *
 * Byte layout (the paper does not print one; this is the reading the whole
 * project uses): digit d = t + 1, byte = d0 + 3 d1 + 9 d2 + 27 d3 + 81 d4,
 * first trit least significant; a 128-trit group is 25 full bytes plus one
 * tail byte holding trits 125..127 and two pad digits equal to 1; plane-1
 * rows are padded with zero bytes to a multiple of 16 bytes.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define OR_GROUP 128
#define OR_FULL_BYTES 25   /* 125 trits in 25 five-trit bytes            */
#define OR_TAIL_TRITS 3    /* 128 - 125                                   */
#define OR_GROUP_BYTES 26  /* 25 + 1 tail byte                            */

/* status bits, same meaning as the library's data-error bits */
#define OR_BAD_CODE 1u
#define OR_T2_OUTSIDE 2u
#define OR_BAD_BYTE 4u
#define OR_BAD_PAD 8u
#define OR_BAD_ROWPTR 16u

/* ---------------------------------------------------------------- sizes */

long long tqo_row_bytes(int K) {
  if (K <= 0 || K % OR_GROUP != 0) return 0;
  long long raw = (long long)(K / OR_GROUP) * OR_GROUP_BYTES;
  return ((raw + 15) / 16) * 16;
}

long long tqo_sal_words(int K) {
  if (K <= 0 || K % OR_GROUP != 0) return 0;
  return (K / OR_GROUP + 31) / 32;
}

/* --------------------------------------------------------- fp16 -> fp64 */

/* IEEE 754 binary16: 1 sign bit, 5 exponent bits (bias 15), 10 fraction
 * bits.  Every binary16 value is exactly representable in binary64. */
double tqo_half_to_double(uint16_t h) {
  int sign = (h >> 15) & 1;
  int e = (h >> 10) & 31;
  int f = h & 1023;
  double v;
  if (e == 0) {
    v = ldexp((double)f, -24); /* subnormal: f * 2^-14 * 2^-10 */
  } else if (e == 31) {
    v = f ? NAN : INFINITY;
  } else {
    v = ldexp((double)(1024 + f), e - 25); /* (1 + f/1024) * 2^(e-15) */
  }
  return sign ? -v : v;
}

/* -------------------------------------------------------------- the byte */

/* Encode up to five digits (each 0..2), least significant first. */
static int encode_digits(const int *d, int n) {
  int v = 0, p = 1;
  for (int i = 0; i < n; i++) {
    v += d[i] * p;
    p *= 3;
  }
  return v;
}

/* Decode a byte into five digits by repeated division by 3. */
static void decode_digits(int v, int *d) {
  for (int i = 0; i < 5; i++) {
    d[i] = v % 3;
    v /= 3;
  }
}

int tqo_encode_byte(const int8_t *t5) {
  int d[5];
  for (int i = 0; i < 5; i++) d[i] = t5[i] + 1;
  return encode_digits(d, 5);
}

/* returns 0 if valid, else the bad-byte bit; trits set to 0 when invalid */
int tqo_decode_byte(int v, int8_t *t5) {
  if (v < 0 || v > 242) {
    for (int i = 0; i < 5; i++) t5[i] = 0;
    return OR_BAD_BYTE;
  }
  int d[5];
  decode_digits(v, d);
  for (int i = 0; i < 5; i++) t5[i] = (int8_t)(d[i] - 1);
  return 0;
}

/* ------------------------------------------------------------- one group */

/* Pack 128 codes into 26 bytes.  Returns status bits (bad code). */
static unsigned pack_group(const int8_t *t, uint8_t *out) {
  unsigned st = 0;
  int d[5];
  for (int j = 0; j < OR_FULL_BYTES; j++) {
    for (int i = 0; i < 5; i++) {
      int c = t[5 * j + i];
      if (c < -1 || c > 1) {
        st |= OR_BAD_CODE;
        c = c < -1 ? -1 : 1;
      }
      d[i] = c + 1;
    }
    out[j] = (uint8_t)encode_digits(d, 5);
  }
  for (int i = 0; i < 5; i++) {
    if (i < OR_TAIL_TRITS) {
      int c = t[5 * OR_FULL_BYTES + i];
      if (c < -1 || c > 1) {
        st |= OR_BAD_CODE;
        c = c < -1 ? -1 : 1;
      }
      d[i] = c + 1;
    } else {
      d[i] = 1; /* pad digit: trit 0 */
    }
  }
  out[OR_FULL_BYTES] = (uint8_t)encode_digits(d, 5);
  return st;
}

/* Unpack 26 bytes into 128 codes; validates bytes and pad digits. */
static unsigned unpack_group(const uint8_t *in, int8_t *t) {
  unsigned st = 0;
  int8_t t5[5];
  for (int j = 0; j < OR_FULL_BYTES; j++) {
    st |= tqo_decode_byte(in[j], t5);
    for (int i = 0; i < 5; i++) t[5 * j + i] = t5[i];
  }
  unsigned bst = tqo_decode_byte(in[OR_FULL_BYTES], t5);
  st |= bst;
  for (int i = 0; i < OR_TAIL_TRITS; i++) t[5 * OR_FULL_BYTES + i] = t5[i];
  if (!bst && (t5[3] != 0 || t5[4] != 0)) st |= OR_BAD_PAD;
  return st;
}

static int sal_bit(const uint32_t *sal, long long words, int n, int g) {
  return (int)((sal[(long long)n * words + g / 32] >> (g % 32)) & 1u);
}

/* -------------------------------------------------------------- rowptr */

/* rowptr[n] = salient groups in rows < n.  Returns status (pad bits). */
unsigned tqo_rowptr(int N, int K, const uint32_t *sal, int32_t *rowptr) {
  int G = K / OR_GROUP;
  long long W = tqo_sal_words(K);
  unsigned st = 0;
  long long acc = 0;
  for (int n = 0; n < N; n++) {
    rowptr[n] = (int32_t)acc;
    for (int g = 0; g < G; g++) acc += sal_bit(sal, W, n, g);
    for (long long b = G; b < W * 32; b++)
      if ((sal[(long long)n * W + b / 32] >> (b % 32)) & 1u) st |= OR_BAD_PAD;
  }
  rowptr[N] = (int32_t)acc;
  return st;
}

static unsigned check_rowptr(int N, int K, const uint32_t *sal, const int32_t *rowptr) {
  int32_t *own = (int32_t *)malloc(sizeof(int32_t) * ((size_t)N + 1));
  if (!own) return OR_BAD_ROWPTR;
  tqo_rowptr(N, K, sal, own);
  unsigned st = 0;
  for (int n = 0; n <= N; n++)
    if (own[n] != rowptr[n]) st |= OR_BAD_ROWPTR;
  free(own);
  return st;
}

/* ---------------------------------------------------------- pack/unpack */

/* Pack T1 (and T2 unless NULL).  plane1: [N][row_bytes]; plane2:
 * [nnz][26] in (n, g) order.  Returns status bits. */
unsigned tqo_pack(int N, int K, const int8_t *T1, const int8_t *T2, const uint32_t *sal,
                  const int32_t *rowptr, uint8_t *plane1, uint8_t *plane2) {
  int G = K / OR_GROUP;
  long long RB = tqo_row_bytes(K), W = tqo_sal_words(K);
  unsigned st = check_rowptr(N, K, sal, rowptr);
  long long j = 0;
  for (int n = 0; n < N; n++) {
    uint8_t *row = plane1 + (long long)n * RB;
    memset(row, 0, (size_t)RB);
    for (int g = 0; g < G; g++) {
      const int8_t *t1 = T1 + (long long)n * K + (long long)g * OR_GROUP;
      st |= pack_group(t1, row + (long long)g * OR_GROUP_BYTES);
      int s = sal_bit(sal, W, n, g);
      if (T2) {
        const int8_t *t2 = T2 + (long long)n * K + (long long)g * OR_GROUP;
        if (s) {
          st |= pack_group(t2, plane2 + j * OR_GROUP_BYTES);
        } else {
          for (int k = 0; k < OR_GROUP; k++)
            if (t2[k] != 0) st |= OR_T2_OUTSIDE;
        }
      } else if (s) {
        st |= OR_T2_OUTSIDE; /* salient group but no second plane given */
      }
      j += s;
    }
  }
  return st;
}

unsigned tqo_unpack(int N, int K, const uint8_t *plane1, const uint8_t *plane2,
                    const uint32_t *sal, const int32_t *rowptr, int8_t *T1, int8_t *T2) {
  int G = K / OR_GROUP;
  long long RB = tqo_row_bytes(K), W = tqo_sal_words(K);
  unsigned st = check_rowptr(N, K, sal, rowptr);
  long long j = 0;
  for (int n = 0; n < N; n++) {
    const uint8_t *row = plane1 + (long long)n * RB;
    for (long long b = (long long)G * OR_GROUP_BYTES; b < RB; b++)
      if (row[b] != 0) st |= OR_BAD_PAD;
    for (int g = 0; g < G; g++) {
      int8_t *t1 = T1 + (long long)n * K + (long long)g * OR_GROUP;
      st |= unpack_group(row + (long long)g * OR_GROUP_BYTES, t1);
      int s = sal_bit(sal, W, n, g);
      if (T2) {
        int8_t *t2 = T2 + (long long)n * K + (long long)g * OR_GROUP;
        if (s && plane2)
          st |= unpack_group(plane2 + j * OR_GROUP_BYTES, t2);
        else
          memset(t2, 0, OR_GROUP);
      }
      j += s;
    }
  }
  return st;
}

/* ------------------------------------------------------------ the linear */

typedef struct {
  int M, N, K;
  const uint8_t *plane1, *plane2;
  const uint32_t *sal;
  const uint16_t *s1, *off, *s2;
  const uint16_t *x;
  const int32_t *rows; /* rows to compute, or NULL for all */
  int nrows;
  const long long *j0; /* per selected row: index of its first salient group */
  double *y, *a;       /* [M][nrows] */
  int tid, nthreads;
} lin_job;

/* Dense fp64 reconstruction of row n (eq. W-hat per group), from the
 * packed bytes.  j = index of the row's first salient group in plane 2. */
static void reconstruct_row(const lin_job *jb, int n, long long j, double *w) {
  int K = jb->K, G = K / OR_GROUP;
  long long RB = tqo_row_bytes(K), W = tqo_sal_words(K);
  int8_t t1[OR_GROUP], t2[OR_GROUP];
  const uint8_t *row = jb->plane1 + (long long)n * RB;
  for (int g = 0; g < G; g++) {
    unpack_group(row + (long long)g * OR_GROUP_BYTES, t1);
    double s1 = tqo_half_to_double(jb->s1[(long long)n * G + g]);
    double off = tqo_half_to_double(jb->off[(long long)n * G + g]);
    int s = sal_bit(jb->sal, W, n, g);
    double s2 = 0.0;
    if (s) {
      unpack_group(jb->plane2 + j * OR_GROUP_BYTES, t2);
      s2 = tqo_half_to_double(jb->s2[j]);
      j++;
    }
    for (int k = 0; k < OR_GROUP; k++) {
      double v = s1 * (double)t1[k] + off;
      if (s) v += s2 * (double)t2[k];
      w[g * OR_GROUP + k] = v;
    }
  }
}

static void *lin_worker(void *arg) {
  lin_job *jb = (lin_job *)arg;
  int K = jb->K;
  double *w = (double *)malloc(sizeof(double) * (size_t)K);
  if (!w) return NULL;
  for (int r = jb->tid; r < jb->nrows; r += jb->nthreads) {
    int n = jb->rows ? jb->rows[r] : r;
    reconstruct_row(jb, n, jb->j0[r], w);
    for (int m = 0; m < jb->M; m++) {
      const uint16_t *xm = jb->x + (long long)m * K;
      double acc = 0.0, aacc = 0.0;
      for (int k = 0; k < K; k++) {
        double p = w[k] * tqo_half_to_double(xm[k]);
        acc += p;
        aacc += fabs(p);
      }
      jb->y[(long long)m * jb->nrows + r] = acc;
      jb->a[(long long)m * jb->nrows + r] = aacc;
    }
  }
  free(w);
  return NULL;
}

/* y[m][r] = sum_k x[m][k] W[rows[r]][k] and a[m][r] = sum_k |x[m][k] W[rows[r]][k]|
 * in fp64, for the selected rows (rows == NULL: all N rows, nrows = N).
 * The first salient group of each row is found by counting salience bits
 * (rowptr is not trusted).  Threads split the rows. */
int tqo_linear_rows(int M, int N, int K, const uint8_t *plane1, const uint8_t *plane2,
                    const uint32_t *sal, const uint16_t *s1, const uint16_t *off,
                    const uint16_t *s2, const uint16_t *x, const int32_t *rows, int nrows,
                    double *y, double *a, int nthreads) {
  if (K <= 0 || K % OR_GROUP != 0 || N <= 0 || M <= 0) return -1;
  if (!rows) nrows = N;
  int G = K / OR_GROUP;
  long long W = tqo_sal_words(K);
  /* own running count of salient groups before each row */
  long long *before = (long long *)malloc(sizeof(long long) * (size_t)N);
  long long *j0 = (long long *)malloc(sizeof(long long) * (size_t)(nrows > 0 ? nrows : 1));
  if (!before || !j0) {
    free(before);
    free(j0);
    return -2;
  }
  long long acc = 0;
  for (int n = 0; n < N; n++) {
    before[n] = acc;
    for (int g = 0; g < G; g++) acc += sal_bit(sal, W, n, g);
  }
  for (int r = 0; r < nrows; r++) j0[r] = before[rows ? rows[r] : r];
  free(before);
  if (acc > 0 && (!plane2 || !s2)) {
    free(j0);
    return -3; /* salient groups but no second plane given */
  }
  if (nthreads < 1) nthreads = 1;
  if (nthreads > 256) nthreads = 256;
  pthread_t th[256];
  lin_job jobs[256];
  for (int t = 0; t < nthreads; t++) {
    lin_job jb = {M, N, K, plane1, plane2, sal, s1, off, s2, x, rows, nrows, j0, y, a, t, nthreads};
    jobs[t] = jb;
  }
  if (nthreads == 1) {
    lin_worker(&jobs[0]);
  } else {
    for (int t = 0; t < nthreads; t++) pthread_create(&th[t], NULL, lin_worker, &jobs[t]);
    for (int t = 0; t < nthreads; t++) pthread_join(th[t], NULL);
  }
  free(j0);
  return 0;
}
