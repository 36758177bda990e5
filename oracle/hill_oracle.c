/*
 * hill_oracle.c -- plain, slow CPU oracle for HillInfer's per-decode-step
 * token-importance evaluation (arxiv 2602.18750).
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the correctness reference for the
 * CUDA path.  Only the test suite, the smoke check and the CPU-baseline leg of
 * the benchmark may load it.  It shares no code, header, table or helper with
 * the CUDA library: it has its own descriptor-free signatures, its own
 * binary16/bfloat16 decoders and its own sort.
 *
 * Everything is computed in double precision from the exact values of the
 * 16-bit inputs.  Layouts are dense and row-major:
 *   q      [B][H][d]          16-bit floats (binary16 or bfloat16 bits)
 *   K, V   [B][Hkv][cap][d]   16-bit floats
 *   lens   [B]                int32, tokens currently cached (new token included)
 *   z      [B][H][cap]        double logits
 *   s, A   [B][cap]           double per-token importance / running sum
 *   idx    [B][max_k]         int32, ascending, -1 padded
 *   count  [B]                int32
 *   out    [B][H][d]          double attention output
 * Query head h reads KV head g = floor(h / G), G = H / Hkv (contiguous grouping
 * of query heads over KV heads, the usual GQA/MQA convention; the paper states
 * only that MHA, MQA and GQA are all handled, Sec. 5.3).
 *
 * Parity pins (what checks this file against something other than itself)
 * live in tests/test_oracle_pins.py.  No function here is "parity unpinned".
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define OR_F16 0
#define OR_BF16 1
#define OR_ATTN 0
#define OR_RAW 1

/* IEEE 754 binary16 -> double, from the format's definition:
 * 1 sign bit, 5 exponent bits (bias 15), 10 fraction bits; exponent 0 holds
 * zeros and subnormals (fraction * 2^-24), exponent 31 holds inf/NaN. */
static double or_half_to_double(uint16_t h) {
  int sign = (h >> 15) & 1;
  int e = (h >> 10) & 0x1f;
  int f = h & 0x3ff;
  double v;
  if (e == 0)
    v = ldexp((double)f, -24);
  else if (e == 31)
    v = f ? NAN : INFINITY;
  else
    v = ldexp((double)(f | 0x400), e - 25);
  return sign ? -v : v;
}

/* bfloat16 -> double: bfloat16 is the upper half of an IEEE binary32
 * (1 sign, 8 exponent bits with bias 127, 7 fraction bits). */
static double or_bf16_to_double(uint16_t h) {
  int sign = (h >> 15) & 1;
  int e = (h >> 7) & 0xff;
  int f = h & 0x7f;
  double v;
  if (e == 0)
    v = ldexp((double)f, -133);
  else if (e == 255)
    v = f ? NAN : INFINITY;
  else
    v = ldexp((double)(f | 0x80), e - 134);
  return sign ? -v : v;
}

double oracle_decode16(int dtype, uint16_t bits) {
  return dtype == OR_BF16 ? or_bf16_to_double(bits) : or_half_to_double(bits);
}

/* Decode n 16-bit values into doubles (used by the tests to see the exact
 * input values the oracle works on). */
void oracle_decode16_array(int dtype, const uint16_t* src, double* dst, int64_t n) {
  for (int64_t i = 0; i < n; ++i) dst[i] = oracle_decode16(dtype, src[i]);
}

/*
 * Step 1 -- attention logits of the current query against every cached key,
 * Eq. 1 (Sec. 2.1) before the softmax:
 *   z[b,h,j] = (sum_i q[b,h,i] * K[b,g(h),j,i]) / sqrt(d),   j < lens[b].
 * Decode reads one query token per sequence against the whole cache (Sec. 2.1,
 * "KV Cache Mechanism").  Entries j >= lens[b] are left untouched.
 */
int oracle_logits(int dtype, int B, int H, int Hkv, int d, int cap,
                  const uint16_t* q, const uint16_t* K, const int32_t* lens,
                  double* z) {
  if (B < 0 || H <= 0 || Hkv <= 0 || H % Hkv || d <= 0 || cap < 0) return 1;
  int G = H / Hkv;
  double inv_sqrt_d = 1.0 / sqrt((double)d);
  int bh;
#pragma omp parallel for schedule(dynamic)
  for (bh = 0; bh < B * H; ++bh) {
    int b = bh / H, h = bh % H, g = h / G;
    int len = lens[b] < cap ? lens[b] : cap;
    double* qv = (double*)malloc(sizeof(double) * (size_t)d);
    for (int i = 0; i < d; ++i)
      qv[i] = oracle_decode16(dtype, q[((int64_t)b * H + h) * d + i]);
    for (int j = 0; j < len; ++j) {
      const uint16_t* kr = K + (((int64_t)b * Hkv + g) * cap + j) * d;
      double acc = 0.0;
      for (int i = 0; i < d; ++i) acc += qv[i] * oracle_decode16(dtype, kr[i]);
      z[((int64_t)b * H + h) * cap + j] = acc * inv_sqrt_d;
    }
    free(qv);
  }
  return 0;
}

/*
 * CEC asymmetric precision (Sec. 4.4): the evaluation may rank tokens with
 * low-precision inner products while the attention keeps the original keys.
 * Here the keys' shadow is OCP FP8 E4M3 with one scale per (b, g, j) row and
 * the query is cast the same way per (b, h).
 * E4M3: 1 sign bit, 4 exponent bits (bias 7), 3 fraction bits; exponent 0
 * holds zero and the subnormals f * 2^-9; the largest finite magnitude is
 * 1.75 * 2^8 = 448; S.1111.111 is NaN; there is no infinity.
 */
double oracle_e4m3_decode(uint8_t c) {
  const int e = (c >> 3) & 15, f = c & 7;
  if (e == 15 && f == 7) return NAN;
  const double v = e == 0 ? ldexp((double)f, -9) : ldexp(1.0 + f / 8.0, e - 7);
  return (c & 0x80) ? -v : v;
}

/* Nearest E4M3 value of a finite float, ties to the even code, magnitudes
 * from 448 up saturating to 448. */
uint8_t oracle_e4m3_encode(float xf) {
  const double x = xf;
  const uint8_t sign = signbit(x) ? 0x80 : 0x00;
  const double a = fabs(x);
  if (a >= 448.0) return sign | 0x7e;
  if (a == 0.0) return sign;
  int ex;
  (void)frexp(a, &ex);                                   /* a = m * 2^ex, m in [0.5, 1) */
  /* spacing of the representable values around a: 2^-9 below 2^-6, else
   * 2^(floor(log2 a) - 3) */
  const double qs = a < ldexp(1.0, -6) ? ldexp(1.0, -9) : ldexp(1.0, ex - 1 - 3);
  const double n = a / qs;                               /* exact: qs is a power of two */
  long k = (long)floor(n);
  const double rem = n - (double)k;
  if (rem > 0.5 || (rem == 0.5 && (k & 1))) k += 1;
  const double v = (double)k * qs;                       /* at most 448 */
  if (v < ldexp(1.0, -6)) return sign | (uint8_t)k;      /* subnormal: code = f */
  int ev;
  (void)frexp(v, &ev);
  const int E = ev - 1 + 7;
  const int f = (int)((ldexp(v, -(ev - 1)) - 1.0) * 8.0);
  return sign | (uint8_t)(E << 3) | (uint8_t)f;
}

void oracle_e4m3_decode_array(const uint8_t* c, double* out, int64_t n) {
  for (int64_t i = 0; i < n; ++i) out[i] = oracle_e4m3_decode(c[i]);
}

void oracle_e4m3_encode_array(const float* x, uint8_t* out, int64_t n) {
  for (int64_t i = 0; i < n; ++i) out[i] = oracle_e4m3_encode(x[i]);
}

/* Quantise rows of d 16-bit values: amax = max_i |x_i| (exact), r = 448 /
 * amax and y_i = x_i * r in float32 arithmetic, code_i = e4m3(y_i), scale =
 * amax / 448 in float32 (so code_i * scale ~ x_i, the largest entry exactly
 * 448 * scale).  An all-zero row gives zero codes and scale 0.  The float32
 * steps are the ones the kernel takes, so both sides pick the same codes. */
void oracle_quantize_rows(int dtype, int64_t rows, int d, const uint16_t* x, uint8_t* codes, float* scale) {
  for (int64_t r = 0; r < rows; ++r) {
    const uint16_t* xr = x + r * d;
    float amax = 0.0f;
    for (int i = 0; i < d; ++i) {
      const float v = (float)fabs(oracle_decode16(dtype, xr[i]));
      if (v > amax) amax = v;
    }
    uint8_t* cr = codes + r * d;
    if (amax == 0.0f) {
      for (int i = 0; i < d; ++i) cr[i] = 0;
      scale[r] = 0.0f;
      continue;
    }
    const volatile float inv = 448.0f / amax;
    for (int i = 0; i < d; ++i) {
      const volatile float y = (float)oracle_decode16(dtype, xr[i]) * inv;
      cr[i] = oracle_e4m3_encode(y);
    }
    const volatile float sc = amax / 448.0f;
    scale[r] = sc;
  }
}

/*
 * Logits from the 8-bit operands: q[b,h,:] is quantised like a key row
 * (codes qc, scale sq) and
 *   z8[b,h,j] = (sum_i e4m3(qc_i) * e4m3(kc[b,g,j,i])) * sq * sk[b,g,j] / sqrt(d)
 * for j < lens[b]; kc [B][Hkv][cap][d] codes, sk [B][Hkv][cap] scales.
 */
int oracle_logits_q8(int dtype, int B, int H, int Hkv, int d, int cap, const uint16_t* q,
                     const uint8_t* kc, const float* sk, const int32_t* lens, double* z) {
  if (B < 0 || H <= 0 || Hkv <= 0 || H % Hkv || d <= 0 || cap < 0) return 1;
  const int G = H / Hkv;
  const double inv_sqrt_d = 1.0 / sqrt((double)d);
  int bh;
#pragma omp parallel for schedule(dynamic)
  for (bh = 0; bh < B * H; ++bh) {
    const int b = bh / H, h = bh % H, g = h / G;
    const int len = lens[b] < cap ? lens[b] : cap;
    uint8_t* qc = (uint8_t*)malloc((size_t)d);
    float sq;
    oracle_quantize_rows(dtype, 1, d, q + ((int64_t)b * H + h) * d, qc, &sq);
    double* qv = (double*)malloc(sizeof(double) * (size_t)d);
    for (int i = 0; i < d; ++i) qv[i] = oracle_e4m3_decode(qc[i]);
    for (int j = 0; j < len; ++j) {
      const int64_t row = ((int64_t)b * Hkv + g) * cap + j;
      const uint8_t* kr = kc + row * d;
      double acc = 0.0;
      for (int i = 0; i < d; ++i) acc += qv[i] * oracle_e4m3_decode(kr[i]);
      z[((int64_t)b * H + h) * cap + j] = acc * (double)sq * (double)sk[row] * inv_sqrt_d;
    }
    free(qv);
    free(qc);
  }
  return 0;
}

/*
 * Step 2 -- per-token importance.
 *  ATTN (the paper's definition, Sec. 4.1 "System Workflow"): a token's
 *    importance is the column-wise sum of its attention weights.  The weights
 *    are the softmax of the logits over the whole causal row j < lens[b], one
 *    softmax per (b, h); the column sum runs over every query head (so over
 *    the G query heads of each KV head and then over the KV heads):
 *      p[b,h,j] = exp(z[b,h,j] - m) / sum_j' exp(z[b,h,j'] - m),  m = max_j z
 *      s[b,j]   = sum_h p[b,h,j].
 *  RAW (Sec. 4.4 "Algorithmic Simplification"): the softmax and exponentials
 *    are dropped and tokens are ranked by the raw inner product; the stored
 *    value keeps the 1/sqrt(d) scale so both modes share the logit scale:
 *      s[b,j] = sum_h z[b,h,j].
 */
int oracle_scores(int mode, int B, int H, int cap, const int32_t* lens,
                  const double* z, double* s) {
  if (mode != OR_ATTN && mode != OR_RAW) return 1;
  for (int b = 0; b < B; ++b) {
    int len = lens[b] < cap ? lens[b] : cap;
    for (int j = 0; j < len; ++j) s[(int64_t)b * cap + j] = 0.0;
    for (int h = 0; h < H; ++h) {
      const double* zr = z + ((int64_t)b * H + h) * cap;
      if (mode == OR_RAW) {
        for (int j = 0; j < len; ++j) s[(int64_t)b * cap + j] += zr[j];
        continue;
      }
      if (len == 0) continue;
      double m = zr[0];
      for (int j = 1; j < len; ++j)
        if (zr[j] > m) m = zr[j];
      double l = 0.0;
      for (int j = 0; j < len; ++j) l += exp(zr[j] - m);
      for (int j = 0; j < len; ++j) s[(int64_t)b * cap + j] += exp(zr[j] - m) / l;
    }
  }
  return 0;
}

/*
 * Step 3 -- cumulative importance across decode steps (H2O-style running sum;
 * the paper tracks importance over the whole decoding stage, Sec. 4.2, but
 * does not spell out the rule):  A[b,j] += s[b,j] for j < lens[b].  A token
 * appended this step starts from the caller's zero.
 */
void oracle_accumulate(int B, int cap, const int32_t* lens, const double* s, double* A) {
  for (int b = 0; b < B; ++b) {
    int len = lens[b] < cap ? lens[b] : cap;
    for (int j = 0; j < len; ++j) A[(int64_t)b * cap + j] += s[(int64_t)b * cap + j];
  }
}

typedef struct {
  double key;
  int32_t j;
} or_item;

/* Order: key descending, then token index ascending; NaN keys rank last. */
static int or_cmp(const void* pa, const void* pb) {
  const or_item* a = (const or_item*)pa;
  const or_item* b = (const or_item*)pb;
  int an = isnan(a->key), bn = isnan(b->key);
  if (an != bn) return an ? 1 : -1;
  if (!an) {
    if (a->key > b->key) return -1;
    if (a->key < b->key) return 1;
  }
  return (a->j > b->j) - (a->j < b->j);
}

static int or_cmp_int(const void* pa, const void* pb) {
  int32_t a = *(const int32_t*)pa, b = *(const int32_t*)pb;
  return (a > b) - (a < b);
}

/*
 * Step 4 -- top-k critical tokens per sequence (Sec. 3.1 "Sparsity
 * Opportunity": keep the top-alpha fraction; Sec. 4.2: the global top-alpha
 * after merging all scores).  The set is the first min(k[b], lens[b]) tokens
 * of the order (key desc, index asc) -- a lower index wins a tie -- emitted in
 * ascending index order.  count[b] is also capped at max_k (the width of idx);
 * the function returns 2 if any sequence hit that cap.  idx is -1 padded.
 */
int oracle_topk(int B, int cap, const int32_t* lens, const double* key,
                const int32_t* k, int max_k, int32_t* idx, int32_t* count) {
  int rc = 0;
  for (int b = 0; b < B; ++b) {
    int len = lens[b] < cap ? lens[b] : cap;
    if (len < 0) len = 0;
    int kb = k[b] < 0 ? 0 : k[b];
    int n = kb < len ? kb : len;
    if (n > max_k) {
      n = max_k;
      rc = 2;
    }
    or_item* items = (or_item*)malloc(sizeof(or_item) * (size_t)(len > 0 ? len : 1));
    for (int j = 0; j < len; ++j) {
      items[j].key = key[(int64_t)b * cap + j];
      items[j].j = j;
    }
    qsort(items, (size_t)len, sizeof(or_item), or_cmp);
    int32_t* row = idx + (int64_t)b * max_k;
    for (int t = 0; t < n; ++t) row[t] = items[t].j;
    qsort(row, (size_t)n, sizeof(int32_t), or_cmp_int);
    for (int t = n; t < max_k; ++t) row[t] = -1;
    count[b] = n;
    free(items);
  }
  return rc;
}

/*
 * BKP bookkeeping (Sec. 4.2, "Bidirectional KV Cache Pools") as a selection
 * rule on one HBM tier: the pools become the kept set, and the two metrics
 * that decide the hot pool are applied per decode step.
 *  (1) Temporal-aware pinning: the R = min(recent, lens[b]) most recent
 *      tokens [len - R, len) are always kept.
 *  (2) The older tokens [0, len - R) are ranked as in oracle_topk (key desc,
 *      index asc) and the first min(k[b], len - R) are kept.
 *  (3) Frequency-aware tracking: the hit-rate table hits[b][j] (2 bytes per
 *      token, the table size Sec. 5.4 gives) counts the steps in which token
 *      j was kept: +1 for every kept token, saturating at 65535.  hits may
 *      be NULL.
 * The kept set is emitted in ascending order, so the pinned window comes
 * last.  If the window plus the ranked tokens exceed max_k, the window is cut
 * to its max_k most recent tokens first, the ranked part gets what is left,
 * and rc is 2.
 */
int oracle_bkp_select(int B, int cap, const int32_t* lens, const double* key, const int32_t* k,
                      int recent, int max_k, int32_t* idx, int32_t* count, uint16_t* hits) {
  int rc = 0;
  if (recent < 0) recent = 0;
  for (int b = 0; b < B; ++b) {
    int len = lens[b] < cap ? lens[b] : cap;
    if (len < 0) len = 0;
    int R = recent < len ? recent : len;
    int kb = k[b] < 0 ? 0 : k[b];
    int n = kb < len - R ? kb : len - R;
    if (R > max_k) {
      R = max_k;
      rc = 2;
    }
    if (n > max_k - R) {
      n = max_k - R;
      rc = 2;
    }
    const int older = len - (recent < len ? recent : len);   /* ranked range [0, older) */
    or_item* items = (or_item*)malloc(sizeof(or_item) * (size_t)(older > 0 ? older : 1));
    for (int j = 0; j < older; ++j) {
      items[j].key = key[(int64_t)b * cap + j];
      items[j].j = j;
    }
    qsort(items, (size_t)older, sizeof(or_item), or_cmp);
    int32_t* row = idx + (int64_t)b * max_k;
    for (int t = 0; t < n; ++t) row[t] = items[t].j;
    qsort(row, (size_t)n, sizeof(int32_t), or_cmp_int);
    for (int t = 0; t < R; ++t) row[n + t] = len - R + t;
    for (int t = n + R; t < max_k; ++t) row[t] = -1;
    count[b] = n + R;
    if (hits)
      for (int t = 0; t < n + R; ++t) {
        uint16_t* hj = hits + (int64_t)b * cap + row[t];
        if (*hj < 65535u) *hj = (uint16_t)(*hj + 1u);
      }
    free(items);
  }
  return rc;
}

/*
 * Step 5 -- attention of the current query over the selected tokens only
 * (Sec. 4.1, workflow step 6: only the critical KV is brought to the GPU for the
 * attention; Eq. 1 restricted to the selected set, the softmax renormalised
 * over that set):
 *   o[b,h,:] = sum_{t<count[b]} p_t V[b,g,idx_t,:],
 *   p_t = softmax_t( q[b,h,:] . K[b,g,idx_t,:] / sqrt(d) ).
 * count[b] == 0 gives o = 0.  Indices outside [0, cap) are an error (rc 3).
 */
int oracle_sparse_attn(int dtype, int B, int H, int Hkv, int d, int cap,
                       const uint16_t* q, const uint16_t* K, const uint16_t* V,
                       const int32_t* idx, const int32_t* count, int max_k,
                       double* out) {
  if (B < 0 || H <= 0 || Hkv <= 0 || H % Hkv || d <= 0) return 1;
  int G = H / Hkv;
  double inv_sqrt_d = 1.0 / sqrt((double)d);
  for (int b = 0; b < B; ++b)
    for (int t = 0; t < count[b] && t < max_k; ++t) {
      int32_t j = idx[(int64_t)b * max_k + t];
      if (j < 0 || j >= cap) return 3;
    }
  int bh;
#pragma omp parallel for schedule(dynamic)
  for (bh = 0; bh < B * H; ++bh) {
    int b = bh / H, h = bh % H, g = h / G;
    int n = count[b] < max_k ? count[b] : max_k;
    double* o = out + ((int64_t)b * H + h) * d;
    for (int i = 0; i < d; ++i) o[i] = 0.0;
    if (n <= 0) continue;
    double* zz = (double*)malloc(sizeof(double) * (size_t)n);
    double* qv = (double*)malloc(sizeof(double) * (size_t)d);
    for (int i = 0; i < d; ++i)
      qv[i] = oracle_decode16(dtype, q[((int64_t)b * H + h) * d + i]);
    for (int t = 0; t < n; ++t) {
      int32_t j = idx[(int64_t)b * max_k + t];
      const uint16_t* kr = K + (((int64_t)b * Hkv + g) * cap + j) * d;
      double acc = 0.0;
      for (int i = 0; i < d; ++i) acc += qv[i] * oracle_decode16(dtype, kr[i]);
      zz[t] = acc * inv_sqrt_d;
    }
    double m = zz[0];
    for (int t = 1; t < n; ++t)
      if (zz[t] > m) m = zz[t];
    double l = 0.0;
    for (int t = 0; t < n; ++t) l += exp(zz[t] - m);
    for (int t = 0; t < n; ++t) {
      int32_t j = idx[(int64_t)b * max_k + t];
      const uint16_t* vr = V + (((int64_t)b * Hkv + g) * cap + j) * d;
      double p = exp(zz[t] - m) / l;
      for (int i = 0; i < d; ++i) o[i] += p * oracle_decode16(dtype, vr[i]);
    }
    free(zz);
    free(qv);
  }
  return 0;
}

/*
 * The whole step in the paper's order: logits -> importance -> (running sum)
 * -> top-k -> sparse attention.  `accum` may be NULL (no running sum); when it
 * is given it is updated in place and ranks the tokens, otherwise s does.
 * `out` may be NULL (selection only).  z, s are caller-provided scratch/outputs
 * of sizes [B][H][cap] and [B][cap].
 */
int oracle_evict_step(int dtype, int mode, int B, int H, int Hkv, int d, int cap,
                      const uint16_t* q, const uint16_t* K, const uint16_t* V,
                      const int32_t* lens, const int32_t* k, int max_k,
                      double* z, double* s, double* accum,
                      int32_t* idx, int32_t* count, double* out) {
  int rc = oracle_logits(dtype, B, H, Hkv, d, cap, q, K, lens, z);
  if (rc) return rc;
  rc = oracle_scores(mode, B, H, cap, lens, z, s);
  if (rc) return rc;
  if (accum) oracle_accumulate(B, cap, lens, s, accum);
  rc = oracle_topk(B, cap, lens, accum ? accum : s, k, max_k, idx, count);
  if (rc) return rc;
  if (out)
    rc = oracle_sparse_attn(dtype, B, H, Hkv, d, cap, q, K, V, idx, count, max_k, out);
  return rc;
}

int oracle_num_threads(void) {
#ifdef _OPENMP
  extern int omp_get_max_threads(void);
  return omp_get_max_threads();
#else
  return 1;
#endif
}
