/*
 * qwm_oracle.c -- plain, slow CPU oracle for the QuantWM per-chunk KV-cache path.
 *
 * TEST INFRASTRUCTURE ONLY.  Only the test suite, the smoke check and the
 * benchmark's CPU-baseline leg may load this library.  The product path (the
 * CUDA library under paper_2609_26425_gb300/) shares no code, header, table or
 * helper with this file and never calls it.
 *
 * Everything here follows the paper "QuantWM: Temporally Consistent 2-Bit KV
 * Cache Quantization for Video World Models" step by step, in the paper's
 * order and notation.  Equation numbers count the displayed equations of the
 * paper in order of appearance (Eq. 1-2 affine quantization, Eq. 3-4
 * centroid-residual form, Eq. 5 logits, Eq. 9 Query-aware distance, Eq. 10
 * group range, Eq. 12 QSAC score, Eq. 13 PSAC error, Eq. 16 coefficients,
 * Eq. 17 compensated logits).
 *
 * Arithmetic: scalar fp32 in a fixed, sequential order for every quantity that
 * decides an integer (centroid ids, INT2 codes, fp16 scales, INT8 PSAC codes).
 * The sums of products that the paper writes as exact inner products (the
 * Query-aware distance, the PSAC projection and the two error sums of the
 * keep rule) take one fused multiply-add (fmaf, a single rounding) per term,
 * in channel order; every other multiply and add is rounded on its own, so
 * the library is compiled with -ffp-contract=off and fuses nothing else.
 * Reconstruction and attention are evaluated in fp64.
 *
 * Readings of the paper where it is silent (rounding, zero-point range, scale
 * storage, INT8 coefficient scheme, keep rule, k-means initialisation) are
 * stated at each function.
 *
 * Parity pins: every function here is pinned by tests under tests/ against
 * closed forms, library routines or brute force (see test_oracle_*.py).
 */
#include <float.h>
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define ORC_OK 0
#define ORC_EINVAL 1

/* ------------------------------------------------------------------------ */
/* Number formats, written from the IEEE-754 / bfloat16 definitions.        */
/* ------------------------------------------------------------------------ */

/* bfloat16 -> fp32: bf16 is the upper half of an fp32 bit pattern. */
float oracle_bf16_to_f32(uint16_t b) {
  uint32_t u = (uint32_t)b << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return f;
}

/* fp32 -> bfloat16, round to nearest, ties to even (by the definition:
 * compare the discarded 16 bits with one half of the kept ulp). */
uint16_t oracle_f32_to_bf16(float f) {
  uint32_t u;
  memcpy(&u, &f, sizeof u);
  if (isnan(f)) return (uint16_t)((u >> 16) | 0x0040u); /* quiet NaN */
  uint32_t kept = u >> 16;
  uint32_t rest = u & 0xFFFFu;
  if (rest > 0x8000u || (rest == 0x8000u && (kept & 1u))) kept += 1u; /* carries into exponent */
  return (uint16_t)kept;
}

/* IEEE binary16 bits -> fp32 value, decoded field by field. */
float oracle_f16_to_f32(uint16_t h) {
  int sign = (h >> 15) & 1;
  int e = (h >> 10) & 0x1F;
  int m = h & 0x3FF;
  double v;
  if (e == 0) v = ldexp((double)m, -24);               /* subnormal: m * 2^-24 */
  else if (e == 31) v = m ? NAN : INFINITY;
  else v = ldexp((double)(1024 + m), e - 25);          /* (1 + m/1024) * 2^(e-15) */
  return (float)(sign ? -v : v);
}

/* Encode a value that is exactly representable in binary16 (non-negative). */
static uint16_t f16_encode_exact(double v) {
  if (v == 0.0) return 0;
  if (isinf(v) || v > 65504.0) return 0x7C00u;
  if (v < ldexp(1.0, -14)) return (uint16_t)(v / ldexp(1.0, -24)); /* subnormal */
  int e;
  double fr = frexp(v, &e);          /* v = fr * 2^e, fr in [0.5, 1) */
  int exp16 = e - 1 + 15;            /* v = (2 fr) * 2^(e-1) */
  int mant = (int)((2.0 * fr - 1.0) * 1024.0);
  return (uint16_t)((exp16 << 10) | mant);
}

/* fp32 (x >= 0) -> binary16 rounded toward +infinity: the smallest binary16
 * value that is >= x.  Used for group scales and the PSAC row scale so that
 * the stored scale never shrinks the range it has to cover. */
uint16_t oracle_f32_to_f16_ru(float x) {
  double v = (double)x;
  if (!(v > 0.0)) return 0; /* zero (and -0) */
  if (v > 65504.0) return 0x7C00u;
  double ulp;
  if (v < ldexp(1.0, -14)) {
    ulp = ldexp(1.0, -24);
  } else {
    int e;
    frexp(v, &e);               /* 2^(e-1) <= v < 2^e */
    ulp = ldexp(1.0, e - 1 - 10);
  }
  double k = ceil(v / ulp);     /* exact: v/ulp is a scaled fp32 value */
  return f16_encode_exact(k * ulp);
}

/* Bit position of channel c's 2-bit code inside a token's packed codes
 * (App. D.1 packs four INT2 codes per byte; the order inside is a reading):
 * every 16 channels form one little-endian 32-bit word; inside it the even
 * channel 2k sits at bits 2k and the odd channel 2k+1 at bits 16 + 2k.  Each
 * byte still holds four codes (byte 0: channels 0,2,4,6; byte 1: 8..14 even;
 * byte 2: 1,3,5,7; byte 3: 9..15 odd). */
static int code_bit(int c) {
  int j = c % 16;
  return 32 * (c / 16) + 16 * (j & 1) + 2 * (j >> 1);
}

/* Round half to even (Eq. 1 rounding operator, reading: ties to even). */
static float rint_even(float x) { return nearbyintf(x); }

/* ------------------------------------------------------------------------ */
/* k-means centroid fitting (Sec. 2, QVG convention: Lloyd iterations).      */
/* ------------------------------------------------------------------------ */
/*
 * Per head h, on the chunk's own tokens x[N][H][d] (bf16):
 *   init: centroid j = token floor(j*N/C) (deterministic; the paper does not
 *         state an initialisation);
 *   repeat iters times:
 *     assign: j* = argmin_j sum_c (x_c - mu_jc)^2, summed over c in order in
 *             fp32 (subtract, square, add); ties go to the lowest j;
 *     update: mu_j = (sum of members, fp64) / count, rounded to fp32;
 *             a cluster with no members keeps its previous centroid;
 *   output: the fp32 centroids rounded to bf16 (the paper keeps centroids in
 *           BF16).
 * objective[it*H + h] receives sum_i min_j dist (fp64 sum of the fp32
 * distances) of assignment step it; assign (optional) receives the final
 * assignment [N][H].
 */
int oracle_fit_centroids(int H, int d, int C, int iters, const uint16_t* x, int64_t N,
                         uint16_t* out, float* cent_f32, int32_t* assign, double* objective,
                         int nthreads) {
  if (H <= 0 || d <= 0 || C <= 0 || C > 65536 || N <= 0 || iters < 0 || !x || !out) return ORC_EINVAL;
#ifdef _OPENMP
  if (nthreads > 0) omp_set_num_threads(nthreads);
#pragma omp parallel for schedule(dynamic, 1)
#endif
  for (int h = 0; h < H; ++h) {
    float* mu = (float*)malloc(sizeof(float) * (size_t)C * d);
    double* sum = (double*)malloc(sizeof(double) * (size_t)C * d);
    int64_t* cnt = (int64_t*)malloc(sizeof(int64_t) * (size_t)C);
    int32_t* lab = (int32_t*)malloc(sizeof(int32_t) * (size_t)N);
    for (int j = 0; j < C; ++j) {
      int64_t src = ((int64_t)j * N) / C;
      for (int c = 0; c < d; ++c) mu[(size_t)j * d + c] = oracle_bf16_to_f32(x[((size_t)src * H + h) * d + c]);
    }
    for (int it = 0; it < iters; ++it) {
      double obj = 0.0;
      for (int64_t i = 0; i < N; ++i) {
        const uint16_t* xi = x + ((size_t)i * H + h) * d;
        float best = 0.0f;
        int bj = -1;
        for (int j = 0; j < C; ++j) {
          float acc = 0.0f;
          for (int c = 0; c < d; ++c) {
            float t = oracle_bf16_to_f32(xi[c]) - mu[(size_t)j * d + c];
            float t2 = t * t;
            acc = acc + t2;
          }
          if (bj < 0 || acc < best) { best = acc; bj = j; }
        }
        lab[i] = bj;
        obj += (double)best;
      }
      if (objective) objective[(size_t)it * H + h] = obj;
      memset(sum, 0, sizeof(double) * (size_t)C * d);
      memset(cnt, 0, sizeof(int64_t) * (size_t)C);
      for (int64_t i = 0; i < N; ++i) {
        const uint16_t* xi = x + ((size_t)i * H + h) * d;
        int j = lab[i];
        cnt[j] += 1;
        for (int c = 0; c < d; ++c) sum[(size_t)j * d + c] += (double)oracle_bf16_to_f32(xi[c]);
      }
      for (int j = 0; j < C; ++j) {
        if (cnt[j] == 0) continue;
        for (int c = 0; c < d; ++c) mu[(size_t)j * d + c] = (float)(sum[(size_t)j * d + c] / (double)cnt[j]);
      }
    }
    if (assign) {
      /* final assignment against the final fp32 centroids */
      for (int64_t i = 0; i < N; ++i) {
        const uint16_t* xi = x + ((size_t)i * H + h) * d;
        float best = 0.0f;
        int bj = -1;
        for (int j = 0; j < C; ++j) {
          float acc = 0.0f;
          for (int c = 0; c < d; ++c) {
            float t = oracle_bf16_to_f32(xi[c]) - mu[(size_t)j * d + c];
            float t2 = t * t;
            acc = acc + t2;
          }
          if (bj < 0 || acc < best) { best = acc; bj = j; }
        }
        assign[(size_t)i * H + h] = bj;
      }
    }
    for (int j = 0; j < C; ++j)
      for (int c = 0; c < d; ++c) {
        float v = mu[(size_t)j * d + c];
        out[((size_t)h * C + j) * d + c] = oracle_f32_to_bf16(v);
        if (cent_f32) cent_f32[((size_t)h * C + j) * d + c] = v;
      }
    free(mu); free(sum); free(cnt); free(lab);
  }
  return ORC_OK;
}

/* ------------------------------------------------------------------------ */
/* Quantize-on-append: QSAC assignment, INT2 residual quantization, PSAC.   */
/* ------------------------------------------------------------------------ */

/* Relative gap between two non-negative decision values. */
static float rel_gap(float a, float b) {
  float m = fabsf(a) > fabsf(b) ? fabsf(a) : fabsf(b);
  if (m == 0.0f) return 0.0f;
  return fabsf(a - b) / m;
}

/*
 * INT2 quantization of one residual group (Eq. 1-2 with b = 2, q in {0..3}).
 * Readings: the range is widened to include 0 (lo = min(min x, 0),
 * hi = max(max x, 0)) so that the zero-point always fits in two bits and the
 * error stays within half a step; s = (hi - lo) / 3 is stored as binary16
 * rounded up, and its stored value is used from then on; X / s is evaluated as
 * x * (1/s); rounding is half to even; an all-zero range gives s = 0, z = 0,
 * codes 0.
 */
/* The zero-inclusive range of a group over 3 (the scale before storage). */
static float group_s32(const float* xg, int G) {
  float lo = 0.0f, hi = 0.0f;
  for (int c = 0; c < G; ++c) {
    if (xg[c] < lo) lo = xg[c];
    if (xg[c] > hi) hi = xg[c];
  }
  return (hi - lo) / 3.0f;
}

/* Codes and zero-point of one group for a given stored scale s (>= the
 * group's (hi - lo) / 3, so the three steps still span the range). */
static void int2_group_with(const float* xg, int G, float s, int* z_out, uint8_t* q_out);

static void int2_group(const float* xg, int G, uint16_t* s_bits, int* z_out, uint8_t* q_out) {
  float s32 = group_s32(xg, G);
  uint16_t sb = oracle_f32_to_f16_ru(s32);
  float s = oracle_f16_to_f32(sb);
  *s_bits = sb;
  int2_group_with(xg, G, s, z_out, q_out);
}

static void int2_group_with(const float* xg, int G, float s, int* z_out, uint8_t* q_out) {
  float lo = 0.0f;
  for (int c = 0; c < G; ++c)
    if (xg[c] < lo) lo = xg[c];
  if (s == 0.0f) {
    *z_out = 0;
    for (int c = 0; c < G; ++c) q_out[c] = 0;
    return;
  }
  float inv = 1.0f / s;
  float zf = rint_even(-lo * inv);        /* z = round(q_min - X_min / s), q_min = 0 */
  int z = (int)zf;
  if (z < 0) z = 0;
  if (z > 3) z = 3;
  *z_out = z;
  for (int c = 0; c < G; ++c) {
    int q = (int)rint_even(xg[c] * inv) + z; /* clip(round(X/s) + z, 0, 3) */
    if (q < 0) q = 0;
    if (q > 3) q = 3;
    q_out[c] = (uint8_t)q;
  }
}

/*
 * Two-level group scales (App. D.1: "group scales use INT8 codes with a
 * shared FP16 secondary scale").  Readings: the secondary scale is shared by
 * the d/G groups of one token-head; s2 = binary16 round-up of
 * max_g s32_g / 255 with s32_g = (hi_g - lo_g) / 3 (reading 2's range); each
 * group's code is the smallest integer c in [0, 255] with c * s2 >= s32_g (an
 * unsigned byte: scales are never negative); the stored scale c * s2 (exact
 * in fp32) then quantizes the group, so the step still covers the range.
 */
static void two_level_scales(const float* res, int d, int G, uint8_t* code, uint16_t* s2_bits, float* s_eff) {
  const int ng = d / G;
  float mx = 0.0f;
  float s32[64];
  for (int g = 0; g < ng; ++g) {
    s32[g] = group_s32(res + g * G, G);
    if (s32[g] > mx) mx = s32[g];
  }
  uint16_t sb = oracle_f32_to_f16_ru(mx / 255.0f);
  float s2 = oracle_f16_to_f32(sb);
  if (mx > 0.0f && 255.0f * s2 < mx) {   /* mx / 255 rounded down in fp32: one binary16 step up */
    sb = (uint16_t)(sb + 1);
    s2 = oracle_f16_to_f32(sb);
  }
  *s2_bits = sb;
  for (int g = 0; g < ng; ++g) {
    int c = 0;
    if (s2 > 0.0f) {
      c = (int)ceilf(s32[g] / s2);
      if (c > 0 && (float)(c - 1) * s2 >= s32[g]) c -= 1;   /* smallest covering code */
      if ((float)c * s2 < s32[g]) c += 1;
      if (c > 255) c = 255;
    }
    code[g] = (uint8_t)c;
    s_eff[g] = (float)c * s2;
  }
}

/*
 * oracle_quantize: one chunk of new Key (is_key = 1) or Value (is_key = 0)
 * tokens x[N][H][d] (bf16) against the chunk's centroids cent[H][C][d] (bf16).
 *
 * Per token i and head h:
 *  1. Query-aware distance (Sec. 4.1, Eq. 9): dQ_j = sum_c w_c (k_c - mu_jc)^2,
 *     summed over c in order, acc = fma(w_c, t * t, acc).  w = NULL means w = 1
 *     (the cold-start rule of App. C.3); Values always use w = 1.
 *  2. Candidates: the M smallest (dQ_j, j) in lexicographic order (ties to the
 *     lower index); M >= C means every centroid (App. C.5).
 *  3. QSAC score (Sec. 4.1, Eq. 10 and 12): for each candidate,
 *     r = k - mu_j, R_g = max_{c in g} r_c - min_{c in g} r_c (plain range, as
 *     written), S_j = sum_g W_g R_g^2 with W_g = sum_{c in g} w_c (both sums in
 *     order); id = argmin over (S_j, j).
 *  4. INT2 residual quantization of x = k - mu_id per group of G channels
 *     (Sec. 2, Eq. 1-2, see int2_group) and k0_c = mu_id,c + s (q_c - z).
 *  5. PSAC (Sec. 4.2, Eq. 13 and 16), Keys only, when U is given and r > 0:
 *     E = k - k0; c_j = sum_c E_c U_cj (in order, one fma per term);
 *     a = max_j |c_j|;
 *     sigma = fp16 round-up of a / 127; t_j = clip(round(c_j * (1/sigma)),
 *     -127, 127) (reading: symmetric absmax INT8, App. D.1 gives INT8 codes
 *     with one FP16 scale per row); chat_j = t_j sigma; e'_c = E_c -
 *     sum_j U_cj chat_j (fma per term); the row is kept only when
 *     sum_c w_c e'_c^2 is strictly below sum_c w_c E_c^2 (both fma per term
 *     on the rounded squares; App. D.1: keep a correction only when it
 *     lowers the approximated Query-weighted error; reading: the diagonal-w
 *     form of Eq. 8); otherwise codes and sigma are zero.
 *
 * Packing (App. D.1, four INT2 codes per byte): channel c's code sits at bit
 * code_bit(c) of the token's d/4 code bytes (see code_bit; d must be a
 * multiple of 16); group g's zero-point goes to byte g/4, bits 2*(g%4).
 *
 * Outputs ([N][H][...] token-major; pointers marked optional may be NULL):
 *   ids[N][H] u8, codes[N][H][d/4] u8, scales[N][H][d/G] fp16 bits,
 *   zeros[N][H][zb] u8 with zb = ceil(2*(d/G)/8),
 *   coef[N][H][r] i8, sigma[N][H] fp16 bits, kept[N][H] u8   (Keys with PSAC)
 *   khat0[N][H][d] fp32 (optional), cand[N][H][M'] i32 with M' = min(M, C)
 *   (optional), margins (optional, relative gaps at the decisions):
 *     m_topm  : between the M-th and (M+1)-th smallest dQ (1 if M >= C)
 *     m_sel   : between the best and second-best S among the candidates
 *     m_psac  : smallest relative distance of a PSAC pre-rounding value
 *               (c_j/sigma, a/127 on the fp16 grid) to a rounding boundary,
 *               and of the keep test (1 when PSAC is off)
 *   dq_out[N][H][C] (optional): every Query-aware distance dQ_j;
 *   s_out[N][H][M'] (optional): the QSAC score of each candidate, in the
 *   order of cand.
 * force_ids (optional) skips steps 1-3 and uses the given ids.
 */
int oracle_quantize(int H, int d, int C, int G, int r, int M, int is_key,
                    const uint16_t* x, int64_t N, const uint16_t* cent, const float* w,
                    const uint16_t* U, const uint8_t* force_ids,
                    uint8_t* ids, uint8_t* codes, uint16_t* scales, uint8_t* zeros,
                    int8_t* coef, uint16_t* sigma, uint8_t* kept,
                    float* khat0, int32_t* cand, float* m_topm, float* m_sel, float* m_psac,
                    float* dq_out, float* s_out, int nthreads,
                    int scale_mode, uint8_t* scode, uint16_t* s2, const float* Mfull) {
  if (H <= 0 || d <= 0 || d > 256 || C <= 0 || C > 256 || G <= 0 || d % G || d % 16 || r < 0 || M <= 0 || N < 0)
    return ORC_EINVAL;
  if (!x || !cent || !ids || !codes || !scales || !zeros) return ORC_EINVAL;
  if (scale_mode != 0 && (scale_mode != 1 || !scode || !s2 || d / G > 64)) return ORC_EINVAL;
  const int ng = d / G;
  const int zb = (2 * ng + 7) / 8;
  const int Mc = M < C ? M : C;
  const int psac = is_key && U && r > 0;
  if (psac && (!coef || !sigma || !kept)) return ORC_EINVAL;
#ifdef _OPENMP
  if (nthreads > 0) omp_set_num_threads(nthreads);
#pragma omp parallel for schedule(dynamic, 64)
#endif
  for (int64_t ih = 0; ih < N * (int64_t)H; ++ih) {
    int64_t i = ih / H;
    int h = (int)(ih % H);
    float* k = (float*)malloc(sizeof(float) * d * 4 + sizeof(float) * C + sizeof(int) * C + sizeof(float) * (r + 1) * 2);
    float* wv = k + d;
    float* res = wv + d;
    float* E = res + d;
    float* dq = E + d;
    int* chosen = (int*)(dq + C);
    float* cj = (float*)(chosen + C);
    float* chat = cj + (r + 1);
    const uint16_t* xi = x + ((size_t)i * H + h) * d;
    const uint16_t* mu_h = cent + (size_t)h * C * d;
    for (int c = 0; c < d; ++c) {
      k[c] = oracle_bf16_to_f32(xi[c]);
      wv[c] = (is_key && w) ? w[(size_t)h * d + c] : 1.0f;
    }
    int id;
    if (force_ids) {
      id = force_ids[(size_t)i * H + h];
      if (m_topm) m_topm[(size_t)i * H + h] = 1.0f;
      if (m_sel) m_sel[(size_t)i * H + h] = 1.0f;
    } else {
      /* 1. Query-aware distance (Eq. 9), or with Mfull the full quadratic
       * form of the ablation in App. C.4: e = k - mu_j (each difference
       * rounded), t = M e (t_c = sum_c' M_cc' e_c', one fma per term in c'
       * order), d = sum_c e_c t_c (one fma per term in c order). */
      for (int j = 0; j < C; ++j) {
        const uint16_t* mu = mu_h + (size_t)j * d;
        float acc = 0.0f;
        if (Mfull && is_key) {
          const float* Mh = Mfull + (size_t)h * d * d;
          for (int c = 0; c < d; ++c) res[c] = k[c] - oracle_bf16_to_f32(mu[c]);
          for (int c = 0; c < d; ++c) {
            float tc = 0.0f;
            for (int c2 = 0; c2 < d; ++c2) tc = fmaf(Mh[(size_t)c * d + c2], res[c2], tc);
            acc = fmaf(res[c], tc, acc);
          }
        } else {
          for (int c = 0; c < d; ++c) {
            float t = k[c] - oracle_bf16_to_f32(mu[c]);
            float t2 = t * t;
            acc = fmaf(wv[c], t2, acc); /* one fused multiply-add per term */
          }
        }
        dq[j] = acc;
        chosen[j] = 0;
        if (dq_out) dq_out[((size_t)i * H + h) * C + j] = acc;
      }
      /* 2. top-M candidates, lexicographic (dQ, j) */
      int* candl = (int*)malloc(sizeof(int) * Mc);
      float lastd = 0.0f;
      for (int m = 0; m < Mc; ++m) {
        int bj = -1;
        for (int j = 0; j < C; ++j) {
          if (chosen[j]) continue;
          if (bj < 0 || dq[j] < dq[bj]) bj = j;
        }
        chosen[bj] = 1;
        candl[m] = bj;
        lastd = dq[bj];
      }
      if (m_topm) {
        float g = 1.0f;
        if (Mc < C) {
          int nj = -1;
          for (int j = 0; j < C; ++j) {
            if (chosen[j]) continue;
            if (nj < 0 || dq[j] < dq[nj]) nj = j;
          }
          g = rel_gap(lastd, dq[nj]);
        }
        m_topm[(size_t)i * H + h] = g;
      }
      /* 3. QSAC score (Eq. 10, 12) */
      float bestS = 0.0f, secondS = INFINITY;
      int bestj = -1;
      for (int m = 0; m < Mc; ++m) {
        int j = candl[m];
        const uint16_t* mu = mu_h + (size_t)j * d;
        float S = 0.0f;
        for (int g = 0; g < ng; ++g) {
          float Wg = 0.0f, mx = 0.0f, mn = 0.0f;
          for (int c = g * G; c < (g + 1) * G; ++c) {
            float rc = k[c] - oracle_bf16_to_f32(mu[c]);
            if (c == g * G) { mx = rc; mn = rc; }
            if (rc > mx) mx = rc;
            if (rc < mn) mn = rc;
            Wg = Wg + wv[c];
          }
          float R = mx - mn;
          float R2 = R * R;
          float t = Wg * R2;
          S = S + t;
        }
        if (bestj < 0 || S < bestS || (S == bestS && j < bestj)) {
          if (bestj >= 0) secondS = bestS < secondS ? bestS : secondS;
          bestS = S;
          bestj = j;
        } else if (S < secondS) {
          secondS = S;
        }
        if (cand) cand[((size_t)i * H + h) * Mc + m] = j;
        if (s_out) s_out[((size_t)i * H + h) * Mc + m] = S;
      }
      if (m_sel) m_sel[(size_t)i * H + h] = (Mc > 1) ? rel_gap(bestS, secondS) : 1.0f;
      id = bestj;
      free(candl);
    }
    ids[(size_t)i * H + h] = (uint8_t)id;
    /* 4. INT2 residual quantization (Eq. 1-2) and k0 = mu + Q_b(r) (Eq. 4) */
    const uint16_t* mu = mu_h + (size_t)id * d;
    uint8_t* cd = codes + ((size_t)i * H + h) * (d / 4);
    uint8_t* zz = zeros + ((size_t)i * H + h) * zb;
    uint16_t* sc = scales + ((size_t)i * H + h) * ng;
    memset(cd, 0, d / 4);
    memset(zz, 0, zb);
    uint8_t qv[256];
    for (int c = 0; c < d; ++c) res[c] = k[c] - oracle_bf16_to_f32(mu[c]);
    float* k0 = E; /* reuse: holds k0 first, then E */
    float s_eff[64];
    if (scale_mode == 1)
      two_level_scales(res, d, G, scode + ((size_t)i * H + h) * ng, s2 + (size_t)i * H + h, s_eff);
    for (int g = 0; g < ng; ++g) {
      uint16_t sb = 0;
      int z;
      float s;
      if (scale_mode == 1) {
        s = s_eff[g];
        int2_group_with(res + g * G, G, s, &z, qv);
      } else {
        int2_group(res + g * G, G, &sb, &z, qv);
        s = oracle_f16_to_f32(sb);
      }
      sc[g] = sb;
      zz[g / 4] |= (uint8_t)(z << (2 * (g % 4)));
      for (int c = g * G; c < (g + 1) * G; ++c) {
        int q = qv[c - g * G];
        int bit = code_bit(c);
        cd[bit / 8] |= (uint8_t)(q << (bit % 8));
        float deq = (float)(q - z) * s;
        k0[c] = oracle_bf16_to_f32(mu[c]) + deq;
      }
    }
    if (khat0)
      for (int c = 0; c < d; ++c) khat0[((size_t)i * H + h) * d + c] = k0[c];
    float mps = 1.0f;
    /* 5. PSAC (Eq. 13, 16) */
    if (psac) {
      const uint16_t* Uh = U + (size_t)h * d * r; /* [d][r] */
      for (int c = 0; c < d; ++c) E[c] = k[c] - k0[c];
      float a = 0.0f;
      for (int j = 0; j < r; ++j) {
        float acc = 0.0f;
        for (int c = 0; c < d; ++c) {
          acc = fmaf(E[c], oracle_bf16_to_f32(Uh[(size_t)c * r + j]), acc);
        }
        cj[j] = acc;
        float ab = fabsf(acc);
        if (ab > a) a = ab;
      }
      float a127 = a / 127.0f;
      uint16_t sgb = oracle_f32_to_f16_ru(a127);
      float sg = oracle_f16_to_f32(sgb);
      int8_t* t = coef + ((size_t)i * H + h) * r;
      if (a127 > 0.0f) {
        /* distance of a/127 to the nearest binary16 value, relative */
        float lower = sg;
        uint16_t lb = sgb;
        if (sg != a127 && sgb > 0) { lb = (uint16_t)(sgb - 1); lower = oracle_f16_to_f32(lb); }
        float gu = rel_gap(a127, sg), gl = rel_gap(a127, lower);
        float gmin = gu < gl ? gu : gl;
        if (gmin < mps) mps = gmin;
      }
      if (sg == 0.0f) {
        for (int j = 0; j < r; ++j) { t[j] = 0; chat[j] = 0.0f; }
      } else {
        float inv = 1.0f / sg;
        for (int j = 0; j < r; ++j) {
          float y = cj[j] * inv;
          float qq = rint_even(y);
          if (qq > 127.0f) qq = 127.0f;
          if (qq < -127.0f) qq = -127.0f;
          t[j] = (int8_t)qq;
          chat[j] = qq * sg;
          float b = floorf(y) + 0.5f; /* nearest rounding boundary */
          float gb = fabsf(y) > 0.0f ? fabsf(y - b) / fabsf(y) : 1.0f;
          if (fabsf(y) <= 127.5f && gb < mps) mps = gb;
        }
      }
      float errq = 0.0f, err0 = 0.0f;
      for (int c = 0; c < d; ++c) {
        float u = 0.0f;
        for (int j = 0; j < r; ++j) u = fmaf(oracle_bf16_to_f32(Uh[(size_t)c * r + j]), chat[j], u);
        float ep = E[c] - u;
        float e2 = ep * ep;
        errq = fmaf(wv[c], e2, errq);
        float E2 = E[c] * E[c];
        err0 = fmaf(wv[c], E2, err0);
      }
      int keep = errq < err0;
      float gk = rel_gap(errq, err0);
      if (gk < mps) mps = gk;
      kept[(size_t)i * H + h] = (uint8_t)keep;
      sigma[(size_t)i * H + h] = keep ? sgb : (uint16_t)0;
      if (!keep)
        for (int j = 0; j < r; ++j) t[j] = 0;
    } else if (is_key && r > 0 && coef && sigma && kept) {
      memset(coef + ((size_t)i * H + h) * r, 0, r);
      sigma[(size_t)i * H + h] = 0;
      kept[(size_t)i * H + h] = 0;
    }
    if (m_psac) m_psac[(size_t)i * H + h] = mps;
    free(k);
  }
  return ORC_OK;
}

/* ------------------------------------------------------------------------ */
/* Reconstruction (Sec. 2 Eq. 4; Sec. 4.2 Eq. 17), fp64.                      */
/* ------------------------------------------------------------------------ */
/*
 * khat[i][h][c] = mu_id,c + s_g (q_c - z_g) + sum_j (t_j sigma) U_cj
 * (the PSAC term only when coef/sigma/U are given and r > 0).  Values use the
 * same path without PSAC (App. D.1).
 */
int oracle_dequant(int H, int d, int C, int G, int r, int64_t N, const uint16_t* cent,
                   const uint8_t* ids, const uint8_t* codes, const uint16_t* scales,
                   const uint8_t* zeros, const int8_t* coef, const uint16_t* sigma,
                   const uint16_t* U, double* out, const uint8_t* scode, const uint16_t* s2) {
  if (H <= 0 || d <= 0 || C <= 0 || G <= 0 || d % G || N < 0 || !out) return ORC_EINVAL;
  const int ng = d / G;
  const int zb = (2 * ng + 7) / 8;
  const int psac = coef && sigma && U && r > 0;
  for (int64_t i = 0; i < N; ++i)
    for (int h = 0; h < H; ++h) {
      size_t th = (size_t)i * H + h;
      int id = ids[th];
      if (id >= C) return ORC_EINVAL;
      const uint16_t* mu = cent + ((size_t)h * C + id) * d;
      for (int c = 0; c < d; ++c) {
        int g = c / G;
        int bit = code_bit(c);
        int q = (codes[th * (d / 4) + bit / 8] >> (bit % 8)) & 3;
        int z = (zeros[th * zb + g / 4] >> (2 * (g % 4))) & 3;
        double s = scode ? (double)scode[th * ng + g] * (double)oracle_f16_to_f32(s2[th])
                         : (double)oracle_f16_to_f32(scales[th * ng + g]);
        double v = (double)oracle_bf16_to_f32(mu[c]) + s * (double)(q - z);
        if (psac) {
          double sg = (double)oracle_f16_to_f32(sigma[th]);
          const uint16_t* Uh = U + (size_t)h * d * r;
          for (int j = 0; j < r; ++j)
            v += (double)coef[th * r + j] * sg * (double)oracle_bf16_to_f32(Uh[(size_t)c * r + j]);
        }
        out[th * d + c] = v;
      }
    }
  return ORC_OK;
}

/* ------------------------------------------------------------------------ */
/* Attention over the reconstructed cache (Sec. 3.3 Eq. 5), fp64.            */
/* ------------------------------------------------------------------------ */
/*
 * For each selected query row i (rows = NULL: all Nq rows) and head h:
 *   l_j = scale * sum_c q_ic k_jc  over every key j (cached chunks followed by
 *   the active chunk, no mask: cached chunks are strictly in the past);
 *   p_j = exp(l_j - max_j l_j); o = sum_j p_j v_j / sum_j p_j;
 *   lse = max_j l_j + log(sum_j p_j).
 * q is bf16 [Nq][H][d]; k, v are fp64 [Nk][H][d]; out is fp64 [n][H][d];
 * lse (optional) is fp64 [H][n] with n = number of selected rows.
 */
int oracle_attend(int H, int d, int64_t Nq, int64_t Nk, const uint16_t* q, const double* k,
                  const double* v, double scale, const int64_t* rows, int64_t n_rows,
                  double* out, double* lse, int nthreads) {
  if (H <= 0 || d <= 0 || Nk <= 0 || !q || !k || !v || !out) return ORC_EINVAL;
  int64_t n = rows ? n_rows : Nq;
#ifdef _OPENMP
  if (nthreads > 0) omp_set_num_threads(nthreads);
#pragma omp parallel for schedule(dynamic, 1)
#endif
  for (int64_t rh = 0; rh < n * (int64_t)H; ++rh) {
    int64_t ri = rh / H;
    int h = (int)(rh % H);
    int64_t i = rows ? rows[ri] : ri;
    double* lg = (double*)malloc(sizeof(double) * (size_t)Nk);
    double* qi = (double*)malloc(sizeof(double) * (size_t)d);
    for (int c = 0; c < d; ++c) qi[c] = (double)oracle_bf16_to_f32(q[((size_t)i * H + h) * d + c]);
    double mx = -INFINITY;
    for (int64_t j = 0; j < Nk; ++j) {
      const double* kj = k + ((size_t)j * H + h) * d;
      double acc = 0.0;
      for (int c = 0; c < d; ++c) acc += qi[c] * kj[c];
      lg[j] = acc * scale;
      if (lg[j] > mx) mx = lg[j];
    }
    double l = 0.0;
    double* o = out + ((size_t)ri * H + h) * d;
    for (int c = 0; c < d; ++c) o[c] = 0.0;
    for (int64_t j = 0; j < Nk; ++j) {
      double p = exp(lg[j] - mx);
      l += p;
      const double* vj = v + ((size_t)j * H + h) * d;
      for (int c = 0; c < d; ++c) o[c] += p * vj[c];
    }
    for (int c = 0; c < d; ++c) o[c] /= l;
    if (lse) lse[(size_t)h * n + ri] = mx + log(l);
    free(lg);
    free(qi);
  }
  return ORC_OK;
}

/* Number of OpenMP threads the oracle uses by default (1 without OpenMP). */
int oracle_max_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}
