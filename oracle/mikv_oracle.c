/*
 * mikv_oracle.c — plain CPU oracle for the MiKV decode path (arxiv 2402.18096).
 *
 * TEST INFRASTRUCTURE ONLY: used by the tests, the smoke check and the benchmark's CPU-baseline
 * leg to check the CUDA library; the product path never calls it. It is deliberately simple:
 * one loop per formula, no blocking, no vectorisation, no reordering beyond what the formulas state.
 *
 * Build: gcc -O2 -ffp-contract=off -fno-fast-math -shared -fPIC (see oracle/__init__.py).
 *
 * Sections of the paper followed:
 *   Eq. 1  (Sec. 3.1, "Retaining Evicted KVs with Quantization"): asymmetric N-bit round-to-nearest
 *          quantizer, alpha = (max - min) / (2^N - 1), beta = min, per token.
 *   Sec. 3.2 ("Low-bit KV Quantization with Dynamic Outlier Awareness"): group size of half the
 *          head dimension; Eq. 2 channel balancer from prefill maxima; Eq. 3 keys multiplied by the
 *          balancer before the quantizer; Eq. 4 query divided by it.
 *   Fig. 4 and Sec. 3: important KV pairs kept in high precision and chosen by an accumulated
 *          attention-score (heavy-hitter) policy; the others retained in low precision.
 *   Sec. 3.4 ("Accelerating the Mixed-Precision KV Cache"): attention is permutation invariant, so
 *          the important and retained sets are stored apart and attended together.
 *   Tables 2-3 ("Cache size" columns): memory accounting.
 * Readings where the paper is silent are stated next to the code that takes them.
 */
#include "mikv_oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>

/* ---------------------------------------------------------------- number formats */

static float bf16_to_f32(uint16_t h) {
  uint32_t u = (uint32_t)h << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return f;
}

double mikv_ref_f16_to_f64(uint16_t h) {
  int sign = h >> 15, e = (h >> 10) & 31, m = h & 1023;
  double v;
  if (e == 0)
    v = ldexp((double)m, -24); /* subnormal: m * 2^-24 */
  else if (e == 31)
    v = m ? NAN : INFINITY;
  else
    v = ldexp((double)(1024 + m), e - 25); /* (1 + m/1024) * 2^(e-15) */
  return sign ? -v : v;
}

/* Encode a finite double that is exactly representable in fp16 (|v| <= 65504). */
static uint16_t encode_f16_exact(double v) {
  uint16_t sign = signbit(v) ? 0x8000 : 0;
  double a = fabs(v);
  if (a == 0.0) return sign;
  int ex;
  frexp(a, &ex);
  int E = ex - 1; /* a in [2^E, 2^(E+1)) */
  if (E < -14) return (uint16_t)(sign | (uint16_t)ldexp(a, 24));
  int mant = (int)ldexp(a, 10 - E) - 1024;
  return (uint16_t)(sign | ((E + 15) << 10) | mant);
}

/* IEEE 754 binary32 -> binary16 conversion with the given rounding direction. */
uint16_t mikv_ref_f32_to_f16(float f, int mode) {
  if (isnan(f)) return 0x7E00;
  uint16_t sign = signbit(f) ? 0x8000 : 0;
  if (isinf(f)) return sign | 0x7C00;
  double a = fabs((double)f);
  if (a == 0.0) return sign;
  int ex;
  frexp(a, &ex);
  int E = ex - 1;
  if (E > 15) { /* beyond the largest binade */
    if (mode == 0) return sign | 0x7C00;
    if (mode < 0) return sign ? 0xFC00 : 0x7BFF;
    return sign ? 0xFBFF : 0x7C00;
  }
  if (E < -14) E = -14; /* subnormal range shares the quantum 2^-24 */
  double m = ldexp((double)f, 10 - E); /* exact: f has a 24-bit significand */
  double r = mode < 0 ? floor(m) : (mode > 0 ? ceil(m) : nearbyint(m));
  double v = ldexp(r, E - 10);
  if (fabs(v) > 65504.0) return sign | 0x7C00; /* rounded past the largest finite value */
  return encode_f16_exact(v);
}

/* ---------------------------------------------------------------- Eq. 1 quantizer */

/*
 * Eq. 1 on one group. Readings (the paper gives the formula, not the storage):
 *  - beta and alpha are stored in fp16. beta16 = fp16 rounded toward -inf of min(x) and
 *    alpha16 = fp16 rounded toward +inf of fp32((max(x) - beta16) / (2^N - 1)), so that the stored
 *    grid beta16 + alpha16 * [0, 2^N - 1] covers [min, max].
 *  - the code is round-half-to-even of the fp32 quotient (x - beta16) / alpha16, clamped to
 *    [0, 2^N - 1].
 *  - a group whose values all equal an fp16 number has span 0; alpha16 is then 1.0 and every code 0.
 */
int mikv_ref_quantize_group(const float* x, int g, int bits, int32_t* codes, uint16_t* alpha16,
                            uint16_t* beta16) {
  float mn = x[0], mx = x[0];
  for (int i = 1; i < g; ++i) {
    if (x[i] < mn) mn = x[i];
    if (x[i] > mx) mx = x[i];
  }
  const int qmax = (1 << bits) - 1;
  uint16_t b16 = mikv_ref_f32_to_f16(mn, -1);
  float beta = (float)mikv_ref_f16_to_f64(b16);
  float span = mx - beta;
  uint16_t a16 = span == 0.0f ? (uint16_t)0x3C00 : mikv_ref_f32_to_f16(span / (float)qmax, +1);
  float alpha = (float)mikv_ref_f16_to_f64(a16);
  for (int i = 0; i < g; ++i) {
    float t = (x[i] - beta) / alpha;
    int c = (int)nearbyintf(t);
    if (c < 0) c = 0;
    if (c > qmax) c = qmax;
    codes[i] = c;
  }
  *alpha16 = a16;
  *beta16 = b16;
  return 0;
}

/* ---------------------------------------------------------------- bit packing */

/*
 * Packed row layout (our own definition, d = 128). Channel c is written c = 16 m + u with
 * u = c mod 16 and m = c div 16. A plane is a sequence of little-endian 16-bit units.
 *  - plane of f-bit fields, f in {2, 4, 8}: P = 16 / f codes per unit; the code of channel c sits in
 *    unit 8 * (2 * (m div P) + (u div 8)) + (u mod 8), at bits [f * (m mod P), f * (m mod P) + f).
 *  - plane of 1-bit fields: the bit of channel c sits in unit (u mod 8), at bit 2 * m + (u div 8).
 * N = 2, 4, 8: one plane of N-bit fields. N = 3: a plane of 2-bit fields holding bits 0..1 of each
 * code, then a plane of 1-bit fields holding bit 2. A row takes 16 * N bytes.
 */
static void field_position(int c, int f, int* unit, int* bit) {
  int u = c % 16, m = c / 16;
  if (f == 1) {
    *unit = u % 8;
    *bit = 2 * m + u / 8;
    return;
  }
  int P = 16 / f;
  *unit = 8 * (2 * (m / P) + u / 8) + u % 8;
  *bit = f * (m % P);
}

static int plane_count(int bits) { return bits == 3 ? 2 : 1; }
static int plane_width(int bits, int p) { return bits == 3 ? (p == 0 ? 2 : 1) : bits; }
static int plane_shift(int bits, int p) { return bits == 3 && p == 1 ? 2 : 0; }

static int valid_bits(int bits) { return bits == 2 || bits == 3 || bits == 4 || bits == 8; }

int mikv_ref_pack_row(const int32_t* codes, int d, int bits, uint8_t* packed) {
  if (!valid_bits(bits) || d != 128) return -1;
  memset(packed, 0, (size_t)d * bits / 8);
  size_t offset = 0;
  for (int p = 0; p < plane_count(bits); ++p) {
    int f = plane_width(bits, p), sh = plane_shift(bits, p);
    uint32_t mask = (1u << f) - 1;
    for (int c = 0; c < d; ++c) {
      int unit, b;
      field_position(c, f, &unit, &b);
      uint32_t v = (((uint32_t)codes[c] >> sh) & mask) << b;
      uint8_t* at = packed + offset + 2 * (size_t)unit;
      at[0] |= (uint8_t)(v & 0xFF);
      at[1] |= (uint8_t)(v >> 8);
    }
    offset += (size_t)d * f / 8;
  }
  return 0;
}

int mikv_ref_unpack_row(const uint8_t* packed, int d, int bits, int32_t* codes) {
  if (!valid_bits(bits) || d != 128) return -1;
  for (int c = 0; c < d; ++c) codes[c] = 0;
  size_t offset = 0;
  for (int p = 0; p < plane_count(bits); ++p) {
    int f = plane_width(bits, p), sh = plane_shift(bits, p);
    uint32_t mask = (1u << f) - 1;
    for (int c = 0; c < d; ++c) {
      int unit, b;
      field_position(c, f, &unit, &b);
      const uint8_t* at = packed + offset + 2 * (size_t)unit;
      uint32_t word = (uint32_t)at[0] | (uint32_t)at[1] << 8;
      codes[c] |= (int32_t)(((word >> b) & mask) << sh);
    }
    offset += (size_t)d * f / 8;
  }
  return 0;
}

/* ---------------------------------------------------------------- rows */

int mikv_ref_quantize_row(const float* x, int d, int bits, int g, uint8_t* packed, uint16_t* params) {
  if (!valid_bits(bits) || g <= 0 || d % g || d != 128) return -1;
  int32_t* codes = (int32_t*)malloc(sizeof(int32_t) * (size_t)d);
  if (!codes) return -1;
  for (int j = 0; j < d / g; ++j)
    mikv_ref_quantize_group(x + (size_t)j * g, g, bits, codes + (size_t)j * g, &params[2 * j],
                            &params[2 * j + 1]);
  mikv_ref_pack_row(codes, d, bits, packed);
  free(codes);
  return 0;
}

int mikv_ref_dequantize_row(const uint8_t* packed, const uint16_t* params, int d, int bits, int g,
                            double* x_hat) {
  if (!valid_bits(bits) || g <= 0 || d % g || d != 128) return -1;
  int32_t* codes = (int32_t*)malloc(sizeof(int32_t) * (size_t)d);
  if (!codes) return -1;
  mikv_ref_unpack_row(packed, d, bits, codes);
  for (int i = 0; i < d; ++i) {
    double alpha = mikv_ref_f16_to_f64(params[2 * (i / g)]);
    double beta = mikv_ref_f16_to_f64(params[2 * (i / g) + 1]);
    x_hat[i] = alpha * codes[i] + beta; /* Eq. 1: alpha * round((x - beta) / alpha) + beta */
  }
  free(codes);
  return 0;
}

/* ---------------------------------------------------------------- Eq. 2 balancer */

/*
 * Eq. 2. Readings: the maxima run over every batch row and prefill token (the equation has no batch
 * index); under grouped-query attention the query maximum also runs over the G query heads sharing
 * the KV head, since the balanced keys are shared by them. A zero maximum on either side gives 1.
 * fp32: sqrt(max|q| / max|k|), IEEE division and square root.
 */
int mikv_ref_balancer(int B, int Hq, int Hkv, int T, int d, const uint16_t* q_pre,
                      const uint16_t* k_pre, float* balancer) {
  if (B <= 0 || Hkv <= 0 || Hq % Hkv || T <= 0 || d <= 0) return -1;
  int G = Hq / Hkv;
  for (int h = 0; h < Hkv; ++h) {
    for (int c = 0; c < d; ++c) {
      float mq = 0.0f, mk = 0.0f;
      for (int b = 0; b < B; ++b)
        for (int t = 0; t < T; ++t) {
          for (int j = 0; j < G; ++j) {
            float v = fabsf(bf16_to_f32(q_pre[(((size_t)b * Hq + h * G + j) * T + t) * d + c]));
            if (v > mq) mq = v;
          }
          float v = fabsf(bf16_to_f32(k_pre[(((size_t)b * Hkv + h) * T + t) * d + c]));
          if (v > mk) mk = v;
        }
      balancer[(size_t)h * d + c] = (mq == 0.0f || mk == 0.0f) ? 1.0f : sqrtf(mq / mk);
    }
  }
  return 0;
}

/* ---------------------------------------------------------------- demotion (quantize + pack) */

int mikv_ref_quantize_pack(int B, int Hkv, int d, int bits, int g, int lo_cap, const uint16_t* k_src,
                           const uint16_t* v_src, const int32_t* src_tok, int n_src,
                           const int32_t* rows, int n_rows, int lo_start, const float* balancer,
                           uint8_t* k_codes, uint8_t* v_codes, uint16_t* k_params,
                           uint16_t* v_params, int32_t* lo_tok) {
  if (!valid_bits(bits) || g <= 0 || d % g || d != 128 || n_rows < 0 || lo_start < 0 ||
      lo_start + n_rows > lo_cap)
    return -1;
  size_t row_bytes = (size_t)d * bits / 8, ngroups = (size_t)(d / g);
  float* x = (float*)malloc(sizeof(float) * (size_t)d);
  if (!x) return -1;
  for (int b = 0; b < B; ++b)
    for (int h = 0; h < Hkv; ++h)
      for (int i = 0; i < n_rows; ++i) {
        size_t bh = (size_t)b * Hkv + h;
        int r = rows[bh * n_rows + i];
        if (r < 0 || r >= n_src) { free(x); return -1; }
        size_t pos = bh * lo_cap + (size_t)(lo_start + i);
        const uint16_t* krow = k_src + (bh * n_src + r) * d;
        const uint16_t* vrow = v_src + (bh * n_src + r) * d;
        for (int c = 0; c < d; ++c) /* Eq. 3: key times balancer before the quantizer */
          x[c] = bf16_to_f32(krow[c]) * (balancer ? balancer[(size_t)h * d + c] : 1.0f);
        mikv_ref_quantize_row(x, d, bits, g, k_codes + pos * row_bytes, k_params + pos * ngroups * 2);
        for (int c = 0; c < d; ++c) x[c] = bf16_to_f32(vrow[c]);
        mikv_ref_quantize_row(x, d, bits, g, v_codes + pos * row_bytes, v_params + pos * ngroups * 2);
        lo_tok[pos] = src_tok ? src_tok[bh * n_src + r] : r;
      }
  free(x);
  return 0;
}

/* ---------------------------------------------------------------- decode attention */

/*
 * softmax(s) V over the union of the important set (bf16 keys/values, attended with q) and the
 * retained set (dequantized balanced keys attended with q / balancer, Eq. 3-4; dequantized values).
 * The union is unordered (Sec. 3.4 permutation invariance). s = sm_scale * q.k.
 * Reading: important keys are stored without the balancer and attended with the plain query; in exact
 * arithmetic (q / b).(k * b) = q.k, so this is the same attention.
 */
int mikv_ref_decode_attention(int B, int Hq, int Hkv, int d, int bits, int g, int hi_cap, int lo_cap,
                              int n_lo, const uint16_t* k_hi, const uint16_t* v_hi,
                              const uint8_t* k_codes, const uint8_t* v_codes,
                              const uint16_t* k_params, const uint16_t* v_params,
                              const float* balancer, const uint16_t* q, double sm_scale,
                              double* out, double* hi_logits, double* ml) {
  if (B <= 0 || Hkv <= 0 || Hq % Hkv || !valid_bits(bits) || g <= 0 || d % g || d != 128 ||
      hi_cap < 0 || n_lo < 0 || n_lo > lo_cap || hi_cap + n_lo == 0)
    return -1;
  int G = Hq / Hkv;
  size_t row_bytes = (size_t)d * bits / 8, ngroups = (size_t)(d / g);
  int n = hi_cap + n_lo;
  double* s = (double*)malloc(sizeof(double) * (size_t)n);
  double* qv = (double*)malloc(sizeof(double) * (size_t)d);
  double* qhat = (double*)malloc(sizeof(double) * (size_t)d);
  double* xr = (double*)malloc(sizeof(double) * (size_t)d);
  if (!s || !qv || !qhat || !xr) { free(s); free(qv); free(qhat); free(xr); return -1; }
  for (int b = 0; b < B; ++b)
    for (int hq = 0; hq < Hq; ++hq) {
      int h = hq / G;
      size_t bh = (size_t)b * Hkv + h, bq = (size_t)b * Hq + hq;
      for (int c = 0; c < d; ++c) {
        qv[c] = bf16_to_f32(q[bq * d + c]);
        qhat[c] = qv[c] / (balancer ? (double)balancer[(size_t)h * d + c] : 1.0); /* Eq. 4 */
      }
      /* logits */
      for (int i = 0; i < hi_cap; ++i) {
        double acc = 0.0;
        for (int c = 0; c < d; ++c) acc += qv[c] * bf16_to_f32(k_hi[(bh * hi_cap + i) * d + c]);
        s[i] = sm_scale * acc;
      }
      for (int t = 0; t < n_lo; ++t) {
        size_t pos = bh * lo_cap + t;
        mikv_ref_dequantize_row(k_codes + pos * row_bytes, k_params + pos * ngroups * 2, d, bits, g, xr);
        double acc = 0.0;
        for (int c = 0; c < d; ++c) acc += qhat[c] * xr[c];
        s[hi_cap + t] = sm_scale * acc;
      }
      /* softmax */
      double m = -INFINITY;
      for (int i = 0; i < n; ++i)
        if (s[i] > m) m = s[i];
      double l = 0.0;
      for (int i = 0; i < n; ++i) l += exp(s[i] - m);
      /* weighted values */
      double* o = out + bq * d;
      for (int c = 0; c < d; ++c) o[c] = 0.0;
      for (int i = 0; i < hi_cap; ++i) {
        double p = exp(s[i] - m) / l;
        for (int c = 0; c < d; ++c) o[c] += p * bf16_to_f32(v_hi[(bh * hi_cap + i) * d + c]);
      }
      for (int t = 0; t < n_lo; ++t) {
        size_t pos = bh * lo_cap + t;
        double p = exp(s[hi_cap + t] - m) / l;
        mikv_ref_dequantize_row(v_codes + pos * row_bytes, v_params + pos * ngroups * 2, d, bits, g, xr);
        for (int c = 0; c < d; ++c) o[c] += p * xr[c];
      }
      if (hi_logits)
        for (int i = 0; i < hi_cap; ++i) hi_logits[bq * hi_cap + i] = s[i];
      if (ml) {
        ml[2 * bq] = m;
        ml[2 * bq + 1] = l;
      }
    }
  free(s); free(qv); free(qhat); free(xr);
  return 0;
}

/* ---------------------------------------------------------------- importance policy */

/*
 * Heavy-hitter importance (the accumulated-attention policy the paper plugs in, Fig. 4 / Sec. 3):
 * each important slot's score grows by the attention weight it receives at this step, summed over the
 * query heads that read it. Reading: retained tokens are not tracked (their high-precision values are
 * gone, so they cannot be promoted back) and no recent-token window is kept.
 */
int mikv_ref_update_importance(int B, int Hq, int Hkv, int hi_cap, const float* hi_logits,
                               const float* ml, float* acc) {
  if (B <= 0 || Hkv <= 0 || Hq % Hkv || hi_cap < 0) return -1;
  int G = Hq / Hkv;
  for (int b = 0; b < B; ++b)
    for (int h = 0; h < Hkv; ++h)
      for (int i = 0; i < hi_cap; ++i) {
        size_t bh = (size_t)b * Hkv + h;
        double add = 0.0;
        for (int j = 0; j < G; ++j) {
          size_t bq = (size_t)b * Hq + (size_t)h * G + j;
          add += exp((double)hi_logits[bq * hi_cap + i] - (double)ml[2 * bq]) / (double)ml[2 * bq + 1];
        }
        acc[bh * hi_cap + i] = (float)((double)acc[bh * hi_cap + i] + add);
      }
  return 0;
}

static int key_less(float sa, int32_t ia, float sb, int32_t ib) {
  if (sa < sb) return 1;
  if (sb < sa) return 0;
  return ia < ib;
}

/*
 * Demotion choice: the n_demote slots with the lowest (score, token id) leave the important set.
 * Reading: ties on the score go to the older (smaller id) token; results are listed by slot.
 * A slot's rank is the number of slots whose key is smaller (keys are distinct because ids are).
 */
int mikv_ref_select_demote(int B, int Hkv, int n, int n_demote, const float* scores,
                           const int32_t* ids, int32_t* demoted, int32_t* kept) {
  if (B <= 0 || Hkv <= 0 || n < 0 || n_demote < 0 || n_demote > n) return -1;
  for (int b = 0; b < B; ++b)
    for (int h = 0; h < Hkv; ++h) {
      size_t bh = (size_t)b * Hkv + h;
      const float* sc = scores + bh * n;
      int nd = 0, nk = 0;
      for (int i = 0; i < n; ++i) {
        int32_t idi = ids ? ids[bh * n + i] : i;
        int rank = 0;
        for (int j = 0; j < n; ++j) {
          int32_t idj = ids ? ids[bh * n + j] : j;
          if (j != i && key_less(sc[j], idj, sc[i], idi)) ++rank;
        }
        if (rank < n_demote)
          demoted[bh * n_demote + nd++] = i;
        else if (kept)
          kept[bh * (n - n_demote) + nk++] = i;
      }
    }
  return 0;
}

int mikv_ref_insert_token(int B, int Hkv, int d, int hi_cap, const uint16_t* k_new,
                          const uint16_t* v_new, int tok, const int32_t* slots, uint16_t* k_hi,
                          uint16_t* v_hi, int32_t* hi_tok, float* acc) {
  for (int b = 0; b < B; ++b)
    for (int h = 0; h < Hkv; ++h) {
      size_t bh = (size_t)b * Hkv + h;
      int s = slots[bh];
      if (s < 0 || s >= hi_cap) return -1;
      memcpy(k_hi + (bh * hi_cap + s) * d, k_new + bh * d, sizeof(uint16_t) * (size_t)d);
      memcpy(v_hi + (bh * hi_cap + s) * d, v_new + bh * d, sizeof(uint16_t) * (size_t)d);
      hi_tok[bh * hi_cap + s] = tok;
      acc[bh * hi_cap + s] = 0.0f;
    }
  return 0;
}

int mikv_ref_gather_hi(int B, int Hkv, int d, int hi_cap, const uint16_t* k_src,
                       const uint16_t* v_src, const int32_t* src_tok, const float* src_scores,
                       int n_src, const int32_t* rows, int n_rows, uint16_t* k_hi, uint16_t* v_hi,
                       int32_t* hi_tok, float* acc) {
  if (n_rows > hi_cap || n_rows < 0) return -1;
  for (int b = 0; b < B; ++b)
    for (int h = 0; h < Hkv; ++h)
      for (int i = 0; i < n_rows; ++i) {
        size_t bh = (size_t)b * Hkv + h;
        int r = rows[bh * n_rows + i];
        if (r < 0 || r >= n_src) return -1;
        memcpy(k_hi + (bh * hi_cap + i) * d, k_src + (bh * n_src + r) * d, sizeof(uint16_t) * (size_t)d);
        memcpy(v_hi + (bh * hi_cap + i) * d, v_src + (bh * n_src + r) * d, sizeof(uint16_t) * (size_t)d);
        hi_tok[bh * hi_cap + i] = src_tok ? src_tok[bh * n_src + r] : r;
        acc[bh * hi_cap + i] = src_scores ? src_scores[bh * n_src + r] : 0.0f;
      }
  return 0;
}

/* ---------------------------------------------------------------- reduced-precision important set */

/*
 * Sec. 3.3 / Table 3 ("Reducing the Precision of the Importance Cache"): the important rows may
 * themselves be stored as hi_bits-bit codes with fp16 (alpha, beta) per group of hg channels.
 * Readings (the paper only reports the resulting sizes and accuracies):
 *  - the important set is quantized with the same quantizer as the retained set (Eq. 1), keys
 *    multiplied by the balancer first (Eq. 3) and attended with q / balancer (Eq. 4);
 *  - a new token enters the important set already quantized (its full-precision row is not kept);
 *  - a demoted important row is re-quantized from its dequantized values: per channel the fp32 value
 *    alpha16 * c + beta16 (the product is exact in fp32, the sum rounded once), then Eq. 1 at the
 *    retained precision. Keys are already balanced and are not multiplied by the balancer again.
 * Arrays: k_hc, v_hc uint8 [B][Hkv][hi_cap][d * hi_bits / 8]; k_hp, v_hp fp16 [B][Hkv][hi_cap][d/hg][2].
 */
static void quantize_kv_row(const uint16_t* krow, const uint16_t* vrow, int d, int h, int bits, int g,
                            const float* balancer, float* x, uint8_t* kc, uint16_t* kp, uint8_t* vc,
                            uint16_t* vp) {
  for (int c = 0; c < d; ++c) /* Eq. 3 */
    x[c] = bf16_to_f32(krow[c]) * (balancer ? balancer[(size_t)h * d + c] : 1.0f);
  mikv_ref_quantize_row(x, d, bits, g, kc, kp);
  for (int c = 0; c < d; ++c) x[c] = bf16_to_f32(vrow[c]);
  mikv_ref_quantize_row(x, d, bits, g, vc, vp);
}

static int hi_args_ok(int d, int hi_bits, int hg) {
  return valid_bits(hi_bits) && hg > 0 && d == 128 && d % hg == 0;
}

int mikv_ref_dequantize_row_f32(const uint8_t* packed, const uint16_t* params, int d, int bits, int g,
                                float* x) {
  if (!valid_bits(bits) || g <= 0 || d % g || d != 128) return -1;
  int32_t* codes = (int32_t*)malloc(sizeof(int32_t) * (size_t)d);
  if (!codes) return -1;
  mikv_ref_unpack_row(packed, d, bits, codes);
  for (int i = 0; i < d; ++i) {
    float alpha = (float)mikv_ref_f16_to_f64(params[2 * (i / g)]);
    float beta = (float)mikv_ref_f16_to_f64(params[2 * (i / g) + 1]);
    float prod = alpha * (float)codes[i]; /* exact: 11-bit alpha times an 8-bit code */
    x[i] = prod + beta;                   /* one rounding */
  }
  free(codes);
  return 0;
}

int mikv_ref_gather_hi_q(int B, int Hkv, int d, int hi_cap, int hi_bits, int hg, const uint16_t* k_src,
                         const uint16_t* v_src, const int32_t* src_tok, const float* src_scores, int n_src,
                         const int32_t* rows, int n_rows, const float* balancer, uint8_t* k_hc, uint8_t* v_hc,
                         uint16_t* k_hp, uint16_t* v_hp, int32_t* hi_tok, float* acc) {
  if (!hi_args_ok(d, hi_bits, hg) || n_rows > hi_cap || n_rows < 0) return -1;
  size_t rb = (size_t)d * hi_bits / 8, np = (size_t)(d / hg) * 2;
  float* x = (float*)malloc(sizeof(float) * (size_t)d);
  if (!x) return -1;
  for (int b = 0; b < B; ++b)
    for (int h = 0; h < Hkv; ++h)
      for (int i = 0; i < n_rows; ++i) {
        size_t bh = (size_t)b * Hkv + h, slot = bh * hi_cap + i;
        int r = rows[bh * n_rows + i];
        if (r < 0 || r >= n_src) { free(x); return -1; }
        quantize_kv_row(k_src + (bh * n_src + r) * d, v_src + (bh * n_src + r) * d, d, h, hi_bits, hg, balancer,
                        x, k_hc + slot * rb, k_hp + slot * np, v_hc + slot * rb, v_hp + slot * np);
        hi_tok[slot] = src_tok ? src_tok[bh * n_src + r] : r;
        acc[slot] = src_scores ? src_scores[bh * n_src + r] : 0.0f;
      }
  free(x);
  return 0;
}

int mikv_ref_insert_token_q(int B, int Hkv, int d, int hi_cap, int hi_bits, int hg, const uint16_t* k_new,
                            const uint16_t* v_new, int tok, const int32_t* slots, const float* balancer,
                            uint8_t* k_hc, uint8_t* v_hc, uint16_t* k_hp, uint16_t* v_hp, int32_t* hi_tok,
                            float* acc) {
  if (!hi_args_ok(d, hi_bits, hg)) return -1;
  size_t rb = (size_t)d * hi_bits / 8, np = (size_t)(d / hg) * 2;
  float* x = (float*)malloc(sizeof(float) * (size_t)d);
  if (!x) return -1;
  for (int b = 0; b < B; ++b)
    for (int h = 0; h < Hkv; ++h) {
      size_t bh = (size_t)b * Hkv + h;
      int s = slots[bh];
      if (s < 0 || s >= hi_cap) { free(x); return -1; }
      size_t slot = bh * hi_cap + s;
      quantize_kv_row(k_new + bh * d, v_new + bh * d, d, h, hi_bits, hg, balancer, x, k_hc + slot * rb,
                      k_hp + slot * np, v_hc + slot * rb, v_hp + slot * np);
      hi_tok[slot] = tok;
      acc[slot] = 0.0f;
    }
  free(x);
  return 0;
}

/*
 * Decode attention with a reduced-precision important set: like mikv_ref_decode_attention, except
 * that the important keys are dequantized balanced keys attended with q / balancer (Eq. 3-4) and the
 * important values are dequantized values.
 */
int mikv_ref_decode_attention_q(int B, int Hq, int Hkv, int d, int hi_bits, int hg, int bits, int g, int hi_cap,
                                int lo_cap, int n_lo, const uint8_t* k_hc, const uint8_t* v_hc,
                                const uint16_t* k_hp, const uint16_t* v_hp, const uint8_t* k_codes,
                                const uint8_t* v_codes, const uint16_t* k_params, const uint16_t* v_params,
                                const float* balancer, const uint16_t* q, double sm_scale, double* out,
                                double* hi_logits, double* ml) {
  if (B <= 0 || Hkv <= 0 || Hq % Hkv || !valid_bits(bits) || g <= 0 || d % g || d != 128 ||
      !hi_args_ok(d, hi_bits, hg) || hi_cap < 0 || n_lo < 0 || n_lo > lo_cap || hi_cap + n_lo == 0)
    return -1;
  int G = Hq / Hkv;
  size_t rb = (size_t)d * bits / 8, np = (size_t)(d / g) * 2;
  size_t hrb = (size_t)d * hi_bits / 8, hnp = (size_t)(d / hg) * 2;
  int n = hi_cap + n_lo;
  double* s = (double*)malloc(sizeof(double) * (size_t)n);
  double* qhat = (double*)malloc(sizeof(double) * (size_t)d);
  double* xr = (double*)malloc(sizeof(double) * (size_t)d);
  if (!s || !qhat || !xr) { free(s); free(qhat); free(xr); return -1; }
  for (int b = 0; b < B; ++b)
    for (int hq = 0; hq < Hq; ++hq) {
      int h = hq / G;
      size_t bh = (size_t)b * Hkv + h, bq = (size_t)b * Hq + hq;
      for (int c = 0; c < d; ++c) /* Eq. 4 */
        qhat[c] = bf16_to_f32(q[bq * d + c]) / (balancer ? (double)balancer[(size_t)h * d + c] : 1.0);
      for (int i = 0; i < n; ++i) {
        if (i < hi_cap) {
          size_t slot = bh * hi_cap + i;
          mikv_ref_dequantize_row(k_hc + slot * hrb, k_hp + slot * hnp, d, hi_bits, hg, xr);
        } else {
          size_t pos = bh * lo_cap + (i - hi_cap);
          mikv_ref_dequantize_row(k_codes + pos * rb, k_params + pos * np, d, bits, g, xr);
        }
        double acc = 0.0;
        for (int c = 0; c < d; ++c) acc += qhat[c] * xr[c];
        s[i] = sm_scale * acc;
      }
      double m = -INFINITY;
      for (int i = 0; i < n; ++i)
        if (s[i] > m) m = s[i];
      double l = 0.0;
      for (int i = 0; i < n; ++i) l += exp(s[i] - m);
      double* o = out + bq * d;
      for (int c = 0; c < d; ++c) o[c] = 0.0;
      for (int i = 0; i < n; ++i) {
        if (i < hi_cap) {
          size_t slot = bh * hi_cap + i;
          mikv_ref_dequantize_row(v_hc + slot * hrb, v_hp + slot * hnp, d, hi_bits, hg, xr);
        } else {
          size_t pos = bh * lo_cap + (i - hi_cap);
          mikv_ref_dequantize_row(v_codes + pos * rb, v_params + pos * np, d, bits, g, xr);
        }
        double p = exp(s[i] - m) / l;
        for (int c = 0; c < d; ++c) o[c] += p * xr[c];
      }
      if (hi_logits)
        for (int i = 0; i < hi_cap; ++i) hi_logits[bq * hi_cap + i] = s[i];
      if (ml) {
        ml[2 * bq] = m;
        ml[2 * bq + 1] = l;
      }
    }
  free(s); free(qhat); free(xr);
  return 0;
}

int mikv_ref_demote_hi_q(int B, int Hkv, int d, int hi_cap, int hi_bits, int hg, int bits, int g, int lo_cap,
                         const int32_t* slots, int lo_pos, const uint8_t* k_hc, const uint8_t* v_hc,
                         const uint16_t* k_hp, const uint16_t* v_hp, const int32_t* hi_tok, uint8_t* k_codes,
                         uint8_t* v_codes, uint16_t* k_params, uint16_t* v_params, int32_t* lo_tok) {
  if (!hi_args_ok(d, hi_bits, hg) || !valid_bits(bits) || g <= 0 || d % g || lo_pos < 0 || lo_pos >= lo_cap)
    return -1;
  size_t hrb = (size_t)d * hi_bits / 8, hnp = (size_t)(d / hg) * 2;
  size_t rb = (size_t)d * bits / 8, np = (size_t)(d / g) * 2;
  float* x = (float*)malloc(sizeof(float) * (size_t)d);
  if (!x) return -1;
  for (int b = 0; b < B; ++b)
    for (int h = 0; h < Hkv; ++h) {
      size_t bh = (size_t)b * Hkv + h;
      int s = slots[bh];
      if (s < 0 || s >= hi_cap) { free(x); return -1; }
      size_t slot = bh * hi_cap + s, pos = bh * lo_cap + lo_pos;
      mikv_ref_dequantize_row_f32(k_hc + slot * hrb, k_hp + slot * hnp, d, hi_bits, hg, x);
      mikv_ref_quantize_row(x, d, bits, g, k_codes + pos * rb, k_params + pos * np);
      mikv_ref_dequantize_row_f32(v_hc + slot * hrb, v_hp + slot * hnp, d, hi_bits, hg, x);
      mikv_ref_quantize_row(x, d, bits, g, v_codes + pos * rb, v_params + pos * np);
      lo_tok[pos] = hi_tok[slot];
    }
  free(x);
  return 0;
}

/* ---------------------------------------------------------------- per-channel keys (App. C) */

/*
 * App. C ("Experiments on Per-Channel Quantization of Keys"): keys quantized per channel, over groups of
 * 64 consecutive retained tokens, with incoming tokens buffered until a group is complete. Readings:
 *  - Eq. 1 with its rounding rules (R2, R3) applied to each channel's 64 values of a token group: one
 *    (alpha16, beta16) per (group, channel); each token's codes are packed in the usual row layout;
 *  - no balancer on per-channel keys (per-channel scales isolate the outlier channels themselves);
 *    values stay per-token (Eq. 1 with group g);
 *  - demoted tokens wait in bf16 in a staging buffer, which here is important-set rows hi_cap ..
 *    hi_cap + 63 (attended like important rows, never scored); when a group of 64 completes it is
 *    quantized into retained rows 64 j .. 64 j + 63 and the buffer starts over.
 * Key parameters: k_params fp16 [B][Hkv][lo_cap / 64][d][2].
 */
#define MIKV_REF_KCH_GROUP 64

int mikv_ref_quantize_channel_group(const float* x, int d, int bits, uint8_t* packed, uint16_t* params) {
  const int n = MIKV_REF_KCH_GROUP;
  if (!valid_bits(bits) || d != 128) return -1;
  float* col = (float*)malloc(sizeof(float) * n);
  int32_t* codes = (int32_t*)malloc(sizeof(int32_t) * (size_t)n * d);
  int32_t* ccol = (int32_t*)malloc(sizeof(int32_t) * n);
  if (!col || !codes || !ccol) { free(col); free(codes); free(ccol); return -1; }
  for (int c = 0; c < d; ++c) {
    for (int t = 0; t < n; ++t) col[t] = x[(size_t)t * d + c];
    mikv_ref_quantize_group(col, n, bits, ccol, &params[2 * c], &params[2 * c + 1]);
    for (int t = 0; t < n; ++t) codes[(size_t)t * d + c] = ccol[t];
  }
  for (int t = 0; t < n; ++t) mikv_ref_pack_row(codes + (size_t)t * d, d, bits, packed + (size_t)t * d * bits / 8);
  free(col); free(codes); free(ccol);
  return 0;
}

/*
 * Append n_rows source rows (k_src/v_src bf16 [B][Hkv][n_src][d], rows [B][Hkv][n_rows], token ids src_tok or
 * the row index) to the retained set at positions n_lo .. n_lo + n_rows - 1 of every (b, h): a position
 * whose group completes is quantized with its group (keys per channel from the staged rows and the new
 * ones, values per token at group g), the others go to staging row hi_cap + (position mod 64) of the
 * important arrays (k_hi/v_hi bf16 [B][Hkv][hi_rows][d], hi_tok [B][Hkv][hi_rows], hi_rows >= hi_cap + 64).
 */
int mikv_ref_append_retained_kch(int B, int Hkv, int d, int bits, int g, int hi_cap, int hi_rows, int lo_cap,
                                 int n_lo, const uint16_t* k_src, const uint16_t* v_src, const int32_t* src_tok,
                                 int n_src, const int32_t* rows, int n_rows, uint16_t* k_hi, uint16_t* v_hi,
                                 int32_t* hi_tok, uint8_t* k_codes, uint8_t* v_codes, uint16_t* k_params,
                                 uint16_t* v_params, int32_t* lo_tok) {
  const int n = MIKV_REF_KCH_GROUP;
  if (!valid_bits(bits) || g <= 0 || d % g || d != 128 || hi_rows < hi_cap + n || lo_cap % n || n_lo < 0 ||
      n_rows < 0 || n_lo + n_rows > lo_cap)
    return -1;
  size_t rb = (size_t)d * bits / 8, np = (size_t)(d / g) * 2;
  float* x = (float*)malloc(sizeof(float) * (size_t)n * d);
  float* xr = (float*)malloc(sizeof(float) * (size_t)d);
  if (!x || !xr) { free(x); free(xr); return -1; }
  for (int b = 0; b < B; ++b)
    for (int h = 0; h < Hkv; ++h) {
      size_t bh = (size_t)b * Hkv + h;
      for (int i = 0; i < n_rows; ++i) {
        int r = rows[bh * n_rows + i];
        if (r < 0 || r >= n_src) { free(x); free(xr); return -1; }
        int p = n_lo + i, slot = hi_cap + p % n;
        /* stage the row (bf16 copy, unbalanced key) */
        memcpy(k_hi + (bh * hi_rows + slot) * d, k_src + (bh * n_src + r) * d, sizeof(uint16_t) * (size_t)d);
        memcpy(v_hi + (bh * hi_rows + slot) * d, v_src + (bh * n_src + r) * d, sizeof(uint16_t) * (size_t)d);
        hi_tok[bh * hi_rows + slot] = src_tok ? src_tok[bh * n_src + r] : r;
        if (p % n != n - 1) continue;
        /* the group of positions p - 63 .. p is complete: quantize it from the staging rows */
        int grp = p / n;
        for (int t = 0; t < n; ++t)
          for (int c = 0; c < d; ++c) x[(size_t)t * d + c] = bf16_to_f32(k_hi[(bh * hi_rows + hi_cap + t) * d + c]);
        mikv_ref_quantize_channel_group(x, d, bits, k_codes + (bh * lo_cap + (size_t)grp * n) * rb,
                                        k_params + ((bh * (lo_cap / n)) + grp) * (size_t)d * 2);
        for (int t = 0; t < n; ++t) {
          size_t pos = bh * lo_cap + (size_t)grp * n + t;
          for (int c = 0; c < d; ++c) xr[c] = bf16_to_f32(v_hi[(bh * hi_rows + hi_cap + t) * d + c]);
          mikv_ref_quantize_row(xr, d, bits, g, v_codes + pos * rb, v_params + pos * np);
          lo_tok[pos] = hi_tok[bh * hi_rows + hi_cap + t];
        }
      }
    }
  free(x); free(xr);
  return 0;
}

/*
 * Decode attention with per-channel retained keys: like mikv_ref_decode_attention, except that the
 * important set holds n_hi bf16 rows (hi_cap slots plus the staged retained tokens) of arrays with
 * hi_rows rows per head, the retained rows are the n_lo_q = 64 * complete-group rows, and a retained key
 * is alpha16[group][c] * code + beta16[group][c] attended with the plain query (no balancer).
 */
int mikv_ref_decode_attention_kch(int B, int Hq, int Hkv, int d, int bits, int g, int hi_rows, int n_hi, int lo_cap,
                                  int n_lo_q, const uint16_t* k_hi, const uint16_t* v_hi, const uint8_t* k_codes,
                                  const uint8_t* v_codes, const uint16_t* k_params, const uint16_t* v_params,
                                  const uint16_t* q, double sm_scale, double* out, double* hi_logits, double* ml) {
  const int n = MIKV_REF_KCH_GROUP;
  if (B <= 0 || Hkv <= 0 || Hq % Hkv || !valid_bits(bits) || g <= 0 || d % g || d != 128 || n_hi < 0 ||
      n_hi > hi_rows || n_lo_q < 0 || n_lo_q % n || n_lo_q > lo_cap || n_hi + n_lo_q == 0)
    return -1;
  int G = Hq / Hkv, tot = n_hi + n_lo_q;
  size_t rb = (size_t)d * bits / 8, np = (size_t)(d / g) * 2;
  double* s = (double*)malloc(sizeof(double) * (size_t)tot);
  double* qv = (double*)malloc(sizeof(double) * (size_t)d);
  double* xr = (double*)malloc(sizeof(double) * (size_t)d);
  int32_t* codes = (int32_t*)malloc(sizeof(int32_t) * (size_t)d);
  if (!s || !qv || !xr || !codes) { free(s); free(qv); free(xr); free(codes); return -1; }
  for (int b = 0; b < B; ++b)
    for (int hq = 0; hq < Hq; ++hq) {
      int h = hq / G;
      size_t bh = (size_t)b * Hkv + h, bq = (size_t)b * Hq + hq;
      for (int c = 0; c < d; ++c) qv[c] = bf16_to_f32(q[bq * d + c]);
      for (int i = 0; i < tot; ++i) {
        double acc = 0.0;
        if (i < n_hi) {
          for (int c = 0; c < d; ++c) acc += qv[c] * bf16_to_f32(k_hi[(bh * hi_rows + i) * d + c]);
        } else {
          int t = i - n_hi;
          const uint16_t* kp = k_params + ((bh * (lo_cap / n)) + t / n) * (size_t)d * 2;
          mikv_ref_unpack_row(k_codes + (bh * lo_cap + t) * rb, d, bits, codes);
          for (int c = 0; c < d; ++c)
            acc += qv[c] * (mikv_ref_f16_to_f64(kp[2 * c]) * codes[c] + mikv_ref_f16_to_f64(kp[2 * c + 1]));
        }
        s[i] = sm_scale * acc;
      }
      double m = -INFINITY;
      for (int i = 0; i < tot; ++i)
        if (s[i] > m) m = s[i];
      double l = 0.0;
      for (int i = 0; i < tot; ++i) l += exp(s[i] - m);
      double* o = out + bq * d;
      for (int c = 0; c < d; ++c) o[c] = 0.0;
      for (int i = 0; i < tot; ++i) {
        double p = exp(s[i] - m) / l;
        if (i < n_hi) {
          for (int c = 0; c < d; ++c) o[c] += p * bf16_to_f32(v_hi[(bh * hi_rows + i) * d + c]);
        } else {
          size_t pos = bh * lo_cap + (i - n_hi);
          mikv_ref_dequantize_row(v_codes + pos * rb, v_params + pos * np, d, bits, g, xr);
          for (int c = 0; c < d; ++c) o[c] += p * xr[c];
        }
      }
      if (hi_logits)
        for (int i = 0; i < n_hi; ++i) hi_logits[bq * n_hi + i] = s[i];
      if (ml) {
        ml[2 * bq] = m;
        ml[2 * bq + 1] = l;
      }
    }
  free(s); free(qv); free(xr); free(codes);
  return 0;
}

/* ---------------------------------------------------------------- prefill importance */

/*
 * Initial importance of every prefill token: the accumulated attention it receives from the prefill's
 * causal attention (H2O's heavy-hitter score, the policy MiKV plugs in, Fig. 4 / Sec. 3): for KV head h,
 * scores[t] = sum over the G query heads j of h and over queries i >= t of the causal softmax weight
 * softmax_{t' <= i}(sm_scale * q_i . k_t') at t' = t. Reading: the same accumulation as the decode-time
 * update (R9) applied to the prefill queries; fp64 throughout.
 * q_pre bf16 [B][Hq][T][d], k_pre bf16 [B][Hkv][T][d], scores fp64 [B][Hkv][T].
 */
int mikv_ref_prefill_scores(int B, int Hq, int Hkv, int T, int d, const uint16_t* q_pre, const uint16_t* k_pre,
                            double sm_scale, double* scores) {
  if (B <= 0 || Hkv <= 0 || Hq % Hkv || T <= 0 || d <= 0) return -1;
  int G = Hq / Hkv;
  double* s = (double*)malloc(sizeof(double) * (size_t)T);
  if (!s) return -1;
  for (size_t x = 0; x < (size_t)B * Hkv * T; ++x) scores[x] = 0.0;
  for (int b = 0; b < B; ++b)
    for (int hq = 0; hq < Hq; ++hq) {
      int h = hq / G;
      const uint16_t* qh = q_pre + ((size_t)b * Hq + hq) * T * d;
      const uint16_t* kh = k_pre + ((size_t)b * Hkv + h) * T * d;
      double* out = scores + ((size_t)b * Hkv + h) * T;
      for (int i = 0; i < T; ++i) {
        double m = -INFINITY;
        for (int t = 0; t <= i; ++t) {
          double acc = 0.0;
          for (int c = 0; c < d; ++c) acc += (double)bf16_to_f32(qh[(size_t)i * d + c]) * bf16_to_f32(kh[(size_t)t * d + c]);
          s[t] = sm_scale * acc;
          if (s[t] > m) m = s[t];
        }
        double l = 0.0;
        for (int t = 0; t <= i; ++t) l += exp(s[t] - m);
        for (int t = 0; t <= i; ++t) out[t] += exp(s[t] - m) / l;
      }
    }
  free(s);
  return 0;
}

/* ---------------------------------------------------------------- memory accounting */

/*
 * Cache size relative to fp16 for every token (the "Cache size" columns of Tables 2-3): a token in
 * the important set costs hi_bits per element (plus 32/g bits of fp16 alpha and beta when it is itself
 * quantized), a retained token bits + 32/g. Returned as a fraction.
 */
double mikv_ref_cache_fraction(int bits, int g, double ratio, int hi_bits) {
  double hi = hi_bits >= 16 ? 1.0 : (hi_bits + 32.0 / g) / 16.0;
  double lo = (bits + 32.0 / g) / 16.0;
  return ratio * hi + (1.0 - ratio) * lo;
}

/* ---------------------------------------------------------------- importance budget */

/*
 * Tables 1-3 state the important set as a ratio of the tokens; the count is the ratio times the context
 * length rounded to the nearest integer, a half rounded up (reading R10). Written as: take the whole part
 * of the product, then add one when the remaining fraction is at least one half.
 */
int mikv_ref_budget(int T, double ratio) {
  if (T < 0 || ratio != ratio || ratio < 0.0 || ratio > 1.0) return -1;
  double x = ratio * (double)T;
  int whole = (int)x; /* x >= 0: truncation is the floor */
  if (x - (double)whole >= 0.5) whole += 1;
  return whole;
}
