/*
 * jq_oracle.c -- plain, slow, obviously-correct CPU oracle for the naive
 * W4A4 linear layer of JustQuant (arxiv 2609.33601).
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path may link, load or
 * call this file: only tests/, __graft_entry__.smoke() and the cpu_baseline /
 * reference leg of bench.py use it.  It shares no code, header, table or
 * constant with the CUDA library (paper_2609_33601_gb300/csrc).
 *
 * What the paper fixes (and what this file computes):
 *   - The deployed graph is a "plain low-bit operator graph": quantise, pack,
 *     low-bit GEMM, with no smoothing, rotation, normalisation or SVD branch
 *     (Sec. 1 contributions; Appendix FAQ Q7).
 *   - Transformer-block linears run INT4 weights and INT4 activations with
 *     group-wise scales: group128 for DiT-XL/2 and ELF-B (Appendix tables
 *     "DiT-XL/2 experimental details", "ELF-B and LLaDA-8B experimental
 *     details"), group64 for FLUX (Sec. 4.2 "FLUX"; Appendix table "FLUX
 *     experimental details").
 *   - The paper prints no quantiser formula.  The reading used here (and in
 *     the GPU path) is the symmetric INT4 rule: for each row and each run of
 *     G consecutive reduction-axis elements,
 *         amax = max |x|,  s = fl32(amax / 7),
 *         q = clamp(rint(fl32(x / s)), -8, 7)      (round half to even)
 *     with s = 0 and q = 0 when amax == 0.  Codes are packed two per byte,
 *     element 2j in the low nibble, 4-bit two's complement.
 *   - The linear layer: acc[m,n,g] = sum_{k in g} qa[m,k]*qw[n,k] (exact
 *     integers), y[m,n] = sum_g acc*s_a[m,g]*s_w[n,g] + bias[n], evaluated
 *     here in fp64 and rounded once to bf16 (round to nearest even).
 *   - Two further settings, each defined where its section begins below: the
 *     ternary weights of W1.58A4 (absmean rule, 2-bit packing) and the NVFP4
 *     format of the LLaDA-8B rows (E2M1 elements, E4M3 block scales).
 *   - The training side: fake quantisation with the straight-through
 *     estimator (last section).
 *
 * Every function here is pinned by tests/test_oracle_pins.py,
 * tests/test_oracle_nvfp4_pins.py or tests/test_oracle_fakequant_pins.py
 * against hand-worked examples, exact rational evaluations, enumerations and
 * invariants; none is unpinned.
 *
 * Floating point: compile with -O2 -ffp-contract=off and without fast-math,
 * so float division is the IEEE-754 single-precision correctly-rounded one
 * and rintf rounds half to even (default rounding mode).  OpenMP only splits
 * independent rows across threads; it never changes any arithmetic.
 */
#include <math.h>
#include <omp.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#include "jq_oracle.h"

/* Thread control for the timed CPU baseline (no effect on any result: every parallel loop
 * here splits independent rows, each computed in one fixed order). */
void oracle_set_threads(int n) { omp_set_num_threads(n > 0 ? n : 1); }
int oracle_max_threads(void) { return omp_get_max_threads(); }

/* ---- bf16 helpers ------------------------------------------------------ */

/* bf16 -> fp32 is exact: a bf16 is the top half of an fp32. */
static float bf16_bits_to_float(uint16_t b) {
  uint32_t u = ((uint32_t)b) << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return f;
}

/*
 * Round an fp64 value to the nearest bf16 (ties to even), by exact scaling:
 * find the bf16 quantum (ulp) of |v|, round |v|/ulp to an integer with rint
 * (fp64, ties to even), scale back.  bf16 has 8 significant bits, normal
 * exponents down to 2^-126 and subnormals in steps of 2^-133.
 */
uint16_t oracle_bf16_rne(double v) {
  if (isnan(v)) return 0x7FC0;
  const int neg = signbit(v) ? 1 : 0;
  double a = fabs(v);
  double r;
  if (a == 0.0) {
    r = 0.0;
  } else if (isinf(a)) {
    r = INFINITY;
  } else {
    int e;
    (void)frexp(a, &e);           /* a = f * 2^e, f in [0.5, 1) -> a in [2^(e-1), 2^e) */
    int ulp_exp = (e - 1) - 7;    /* 8 significant bits */
    if (ulp_exp < -133) ulp_exp = -133;  /* subnormal quantum */
    double q = ldexp(a, -ulp_exp);       /* exact */
    double n = rint(q);                  /* ties to even */
    r = ldexp(n, ulp_exp);
    /* largest finite bf16 is (2 - 2^-7) * 2^127; anything rounding above it is inf */
    if (r > ldexp(255.0, 120)) r = INFINITY;
  }
  float f = (float)r; /* exact: r is representable in bf16, hence in fp32 */
  uint32_t u;
  memcpy(&u, &f, sizeof u);
  uint16_t b = (uint16_t)(u >> 16);
  if (neg) b |= 0x8000;
  return b;
}

/* ---- quantiser (one group) --------------------------------------------- */

/*
 * Symmetric INT4 quantisation of one group of G consecutive values already
 * widened to fp32 (the rule in the file header).  Writes G codes and returns
 * the group scale.
 */
static float quantize_group(const float* xf, int64_t G, int8_t* q) {
  float amax = 0.0f;
  for (int64_t k = 0; k < G; ++k) {
    float a = fabsf(xf[k]);
    if (a > amax) amax = a;
  }
  if (amax == 0.0f) {
    for (int64_t k = 0; k < G; ++k) q[k] = 0;
    return 0.0f;
  }
  const float s = amax / 7.0f;            /* IEEE single division */
  for (int64_t k = 0; k < G; ++k) {
    float t = xf[k] / s;                  /* IEEE single division */
    float r = rintf(t);                   /* half to even */
    if (r > 7.0f) r = 7.0f;
    if (r < -8.0f) r = -8.0f;
    q[k] = (int8_t)r;
  }
  return s;
}

/* Activations: bf16 [M, K] with row stride ldx (elements) -> codes [M, K] and
 * scales [M, K/G] (row-major, one scale per token and K-group). */
void oracle_quantize_bf16(const uint16_t* x, int64_t M, int64_t K, int64_t ldx,
                          int64_t G, int8_t* codes, float* scales) {
  const int64_t ng = K / G;
#pragma omp parallel for schedule(static)
  for (int64_t m = 0; m < M; ++m) {
    float* xf = (float*)malloc((size_t)K * sizeof(float));
    for (int64_t k = 0; k < K; ++k) xf[k] = bf16_bits_to_float(x[m * ldx + k]);
    for (int64_t g = 0; g < ng; ++g)
      scales[m * ng + g] = quantize_group(xf + g * G, G, codes + m * K + g * G);
    free(xf);
  }
}

/* Weights: fp32 [N, K] row-major -> codes [N, K] and scales [N, K/G] (one
 * scale per output channel and K-group). */
void oracle_quantize_f32(const float* w, int64_t N, int64_t K, int64_t G,
                         int8_t* codes, float* scales) {
  const int64_t ng = K / G;
#pragma omp parallel for schedule(static)
  for (int64_t n = 0; n < N; ++n) {
    for (int64_t g = 0; g < ng; ++g) {
      scales[n * ng + g] = quantize_group(w + n * K + g * G, G, codes + n * K + g * G);
    }
  }
}

/* ---- packing ------------------------------------------------------------ */

/* codes [rows, K] -> bytes [rows, K/2]: element 2j in the low nibble, 2j+1 in
 * the high nibble, each as 4-bit two's complement. */
void oracle_pack(const int8_t* codes, int64_t rows, int64_t K, uint8_t* packed) {
  for (int64_t r = 0; r < rows; ++r)
    for (int64_t j = 0; j < K / 2; ++j) {
      uint8_t lo = (uint8_t)(codes[r * K + 2 * j] & 0x0F);
      uint8_t hi = (uint8_t)(codes[r * K + 2 * j + 1] & 0x0F);
      packed[r * (K / 2) + j] = (uint8_t)(lo | (hi << 4));
    }
}

/* Inverse of oracle_pack: sign-extend each nibble. */
void oracle_unpack(const uint8_t* packed, int64_t rows, int64_t K, int8_t* codes) {
  for (int64_t r = 0; r < rows; ++r)
    for (int64_t j = 0; j < K / 2; ++j) {
      uint8_t b = packed[r * (K / 2) + j];
      int lo = b & 0x0F, hi = (b >> 4) & 0x0F;
      codes[r * K + 2 * j] = (int8_t)(lo >= 8 ? lo - 16 : lo);
      codes[r * K + 2 * j + 1] = (int8_t)(hi >= 8 ? hi - 16 : hi);
    }
}

/* ---- ternary weights (W1.58A4) ----------------------------------------- */

/*
 * The W1.58A4 setting of the paper runs ternary weights with INT4 activations,
 * group128 (Appendix table "DiT-XL/2 experimental details": "Ternary weights,
 * INT4 activations, group128"; the ELF-B table likewise).  The paper prints no
 * ternary rule.  The reading used here is the absmean rule of 1.58-bit weight
 * quantisation, applied per row and per group of G consecutive reduction-axis
 * elements (the group the paper names):
 *     s = fl32(mean |w|)     -- the mean taken in fp64, summing the group in
 *                               index order, then one division by G
 *     q = clamp(rint(fl32(w / s)), -1, 1)        (round half to even)
 * with s = 0 and q = 0 for an all-zero group.  A ternary code is an INT4 code,
 * so the W1.58A4 linear layer is oracle_linear with these weight codes.
 */
void oracle_quantize_ternary_f32(const float* w, int64_t N, int64_t K, int64_t G, int8_t* codes,
                                 float* scales) {
#pragma omp parallel for schedule(static)
  for (int64_t n = 0; n < N; ++n) {
    for (int64_t g = 0; g < K / G; ++g) {
      const float* wg = w + n * K + g * G;
      double sum = 0.0;
      for (int64_t k = 0; k < G; ++k) sum += fabs((double)wg[k]);
      const float s = (float)(sum / (double)G);
      scales[n * (K / G) + g] = s;
      for (int64_t k = 0; k < G; ++k) {
        int q = 0;
        if (s != 0.0f) {
          const float t = wg[k] / s;        /* IEEE single division */
          const float r = rintf(t);         /* ties to even */
          q = r > 1.0f ? 1 : (r < -1.0f ? -1 : (int)r);
        }
        codes[n * K + g * G + k] = (int8_t)q;
      }
    }
  }
}

/*
 * 2-bit packing of ternary codes: the code q is stored as q + 1 in {0, 1, 2}.
 * Every 16 consecutive elements of a row fill 4 bytes; byte j (j = 0..3) holds
 * elements 2j, 2j+1, 8+2j and 9+2j in its bits 0-1, 2-3, 4-5 and 6-7.  (Read
 * as a little-endian 32-bit word, the four 2-bit fields at bit offsets 2i of
 * every byte, i = 0..3, then collect elements {2j}, {2j+1}, {8+2j}, {9+2j}.)
 */
static int64_t ternary_bit(int64_t e) { /* bit offset of element e (0..15) within its 32-bit word */
  const int64_t half = e / 8, r = e % 8;
  return 8 * (r / 2) + 2 * (r % 2) + 4 * half;
}

void oracle_pack_ternary(const int8_t* codes, int64_t rows, int64_t K, uint8_t* packed) {
  for (int64_t r = 0; r < rows; ++r)
    for (int64_t w0 = 0; w0 < K; w0 += 16) {
      uint32_t word = 0;
      for (int64_t e = 0; e < 16; ++e)
        word |= (uint32_t)(codes[r * K + w0 + e] + 1) << ternary_bit(e);
      for (int64_t b = 0; b < 4; ++b) packed[r * (K / 4) + w0 / 4 + b] = (uint8_t)(word >> (8 * b));
    }
}

void oracle_unpack_ternary(const uint8_t* packed, int64_t rows, int64_t K, int8_t* codes) {
  for (int64_t r = 0; r < rows; ++r)
    for (int64_t w0 = 0; w0 < K; w0 += 16) {
      uint32_t word = 0;
      for (int64_t b = 0; b < 4; ++b) word |= (uint32_t)packed[r * (K / 4) + w0 / 4 + b] << (8 * b);
      for (int64_t e = 0; e < 16; ++e) codes[r * K + w0 + e] = (int8_t)((int)((word >> ternary_bit(e)) & 3u) - 1);
    }
}

/* ---- NVFP4 (the LLaDA-8B W4A4 format) ---------------------------------- */

/*
 * The paper runs LLaDA-8B as "NVFP4 W4A4" (Appendix table "ELF-B and LLaDA-8B experimental
 * details") and prints no definition of the format.  The reading used here is the published
 * NVFP4 format: elements in FP4 E2M1 (magnitudes 0, 0.5, 1, 1.5, 2, 3, 4, 6), one FP8 E4M3 scale
 * per block of 16 consecutive reduction-axis elements of a row, and one fp32 scale g per
 * tensor.  For weights g = fl32(amax |w| / 2688) (2688 = 6 * 448: the block holding the tensor's
 * largest magnitude gets the largest E4M3 scale); for activations g is a calibrated constant the
 * caller supplies.  Per block b of a row:
 *     s_b = e4m3(fl32(amax_b / fl32(6 * g)))   (nearest, ties to even mantissa, saturating at 448)
 *     S_b = fl32(s_b * g)
 *     q   = e2m1(fl32(x / S_b))               (nearest, ties to even mantissa, saturating at 6)
 * and q = 0 wherever g == 0 or S_b == 0.  The codes are kept here as 2q (integers in [-12, 12]).
 * The linear layer: y = sum_b (sum_{k in b} qa * qw) * sa_b * sw_b * ga * gw + bias, in fp64.
 */

/* Nearest E2M1 magnitude to a (finite, >= 0), ties to the even mantissa, saturating at 6;
 * returned doubled (an integer in {0, 1, 2, 3, 4, 6, 8, 12}). */
static int e2m1_twice(double a) {
  static const double grid[8] = {0.0, 0.5, 1.0, 1.5, 2.0, 3.0, 4.0, 6.0};
  static const int even[8] = {1, 0, 1, 0, 1, 0, 1, 0}; /* mantissa bit 0 */
  if (a >= 6.0) return 12;
  for (int i = 0; i < 7; ++i) {
    if (a <= grid[i + 1]) {
      const double dlo = a - grid[i], dhi = grid[i + 1] - a; /* exact: a is an fp32 value */
      const int pick = dlo < dhi ? i : (dhi < dlo ? i + 1 : (even[i] ? i : i + 1));
      return (int)(2.0 * grid[pick]);
    }
  }
  return 12;
}

/* Nearest E4M3 value to a (finite, >= 0): 3 mantissa bits, exponent bias 7, normals down to
 * 2^-6, subnormals in steps of 2^-9, ties to even, saturating at the largest finite 448. */
static float e4m3_round(float a) {
  if (a == 0.0f) return 0.0f;
  int e;
  (void)frexp((double)a, &e);     /* a in [2^(e-1), 2^e) */
  int q_exp = (e - 1) - 3;        /* 3 mantissa bits */
  if (q_exp < -9) q_exp = -9;     /* subnormal quantum */
  const double n = rint(ldexp((double)a, -q_exp)); /* exact scaling; ties to even */
  double r = ldexp(n, q_exp);
  if (r > 448.0) r = 448.0;
  return (float)r;
}

float oracle_nvfp4_tensor_scale(const float* x, int64_t n) {
  float amax = 0.0f;
  for (int64_t i = 0; i < n; ++i) {
    const float a = fabsf(x[i]);
    if (a > amax) amax = a;
  }
  return amax / 2688.0f;
}

void oracle_quantize_nvfp4(const float* x, int64_t rows, int64_t K, float g, int8_t* codes2,
                           float* block_scales) {
  const int64_t nb = K / 16;
#pragma omp parallel for schedule(static)
  for (int64_t r = 0; r < rows; ++r) {
    for (int64_t b = 0; b < nb; ++b) {
      const float* xb = x + r * K + b * 16;
      float amax = 0.0f;
      for (int k = 0; k < 16; ++k) {
        const float a = fabsf(xb[k]);
        if (a > amax) amax = a;
      }
      float s = 0.0f, S = 0.0f;
      if (g != 0.0f) {
        const float six_g = 6.0f * g;
        s = e4m3_round(amax / six_g);
        S = s * g;
      }
      block_scales[r * nb + b] = s;
      for (int k = 0; k < 16; ++k) {
        int q2 = 0;
        if (S != 0.0f) {
          const float t = xb[k] / S;  /* IEEE single division */
          q2 = e2m1_twice(fabs((double)t));
          if (t < 0.0f) q2 = -q2;
        }
        codes2[r * K + b * 16 + k] = (int8_t)q2;
      }
    }
  }
}

/* Packing: E2M1 codes (bit 3 sign, bits 1-2 exponent, bit 0 mantissa), two per byte, element 2j
 * in the low nibble of byte j.  Magnitude codes: 0 -> 0, 0.5 -> 1, 1 -> 2, 1.5 -> 3, 2 -> 4,
 * 3 -> 5, 4 -> 6, 6 -> 7 (the code is the magnitude's index in that list). */
static int e2m1_code(int q2) {
  static const int twice[8] = {0, 1, 2, 3, 4, 6, 8, 12};
  const int m = q2 < 0 ? -q2 : q2;
  for (int i = 0; i < 8; ++i)
    if (twice[i] == m) return (q2 < 0 ? 8 : 0) | i;
  return -1;
}

void oracle_pack_nvfp4(const int8_t* codes2, int64_t rows, int64_t K, uint8_t* packed) {
  for (int64_t r = 0; r < rows; ++r)
    for (int64_t j = 0; j < K / 2; ++j)
      packed[r * (K / 2) + j] =
          (uint8_t)(e2m1_code(codes2[r * K + 2 * j]) | (e2m1_code(codes2[r * K + 2 * j + 1]) << 4));
}

void oracle_unpack_nvfp4(const uint8_t* packed, int64_t rows, int64_t K, int8_t* codes2) {
  static const int twice[8] = {0, 1, 2, 3, 4, 6, 8, 12};
  for (int64_t r = 0; r < rows; ++r)
    for (int64_t j = 0; j < K / 2; ++j) {
      const int b = packed[r * (K / 2) + j];
      const int lo = b & 15, hi = b >> 4;
      codes2[r * K + 2 * j] = (int8_t)((lo & 8) ? -twice[lo & 7] : twice[lo & 7]);
      codes2[r * K + 2 * j + 1] = (int8_t)((hi & 8) ? -twice[hi & 7] : twice[hi & 7]);
    }
}

/* y64[m, n] = sum_b acc4[m,n,b] / 4 * sa[m,b] * sw[n,b] * ga * gw + bias[n], in fp64, with
 * acc4 = sum over the block of (2 qa) * (2 qw), an exact integer; ybf16 = its bf16 rounding. */
void oracle_linear_nvfp4(const int8_t* qa2, const float* sa, float ga, const int8_t* qw2, const float* sw,
                         float gw, const float* bias, int64_t M, int64_t N, int64_t K, double* y64,
                         uint16_t* ybf16) {
  const int64_t nb = K / 16;
#pragma omp parallel for schedule(static)
  for (int64_t m = 0; m < M; ++m)
    for (int64_t n = 0; n < N; ++n) {
      double y = 0.0;
      for (int64_t b = 0; b < nb; ++b) {
        int32_t acc4 = 0;
        for (int k = 0; k < 16; ++k)
          acc4 += (int32_t)qa2[m * K + b * 16 + k] * (int32_t)qw2[n * K + b * 16 + k];
        y += (double)acc4 / 4.0 * (double)sa[m * nb + b] * (double)sw[n * nb + b];
      }
      y = y * (double)ga * (double)gw + (bias ? (double)bias[n] : 0.0);
      y64[m * N + n] = y;
      ybf16[m * N + n] = oracle_bf16_rne(y);
    }
}

/* ---- integer GEMM and the dequantising epilogue ------------------------- */

/* acc[m, n, g] = sum over the G elements of group g of qa[m,k] * qw[n,k]. */
void oracle_group_partials(const int8_t* qa, const int8_t* qw, int64_t M, int64_t N,
                           int64_t K, int64_t G, int32_t* acc) {
  const int64_t ng = K / G;
#pragma omp parallel for schedule(static)
  for (int64_t m = 0; m < M; ++m)
    for (int64_t n = 0; n < N; ++n)
      for (int64_t g = 0; g < ng; ++g) {
        int32_t s = 0;
        for (int64_t k = g * G; k < (g + 1) * G; ++k) s += (int32_t)qa[m * K + k] * (int32_t)qw[n * K + k];
        acc[(m * N + n) * ng + g] = s;
      }
}

/*
 * y64[m, n] = sum_g acc[m,n,g] * s_a[m,g] * s_w[n,g] + bias[n]   (fp64)
 * ybf16     = bf16_rne(y64)
 * s_a is [M, K/G], s_w is [N, K/G] (per output channel), bias is [N] or NULL.
 * The partial sums are recomputed here, one group at a time, from the codes.
 * Either output pointer may be NULL.
 */
void oracle_linear(const int8_t* qa, const float* s_a, const int8_t* qw, const float* s_w,
                   const float* bias, int64_t M, int64_t N, int64_t K, int64_t G,
                   double* y64, uint16_t* ybf16) {
  const int64_t ng = K / G;
#pragma omp parallel for schedule(static)
  for (int64_t m = 0; m < M; ++m)
    for (int64_t n = 0; n < N; ++n) {
      double y = 0.0;
      for (int64_t g = 0; g < ng; ++g) {
        int32_t s = 0;
        for (int64_t k = g * G; k < (g + 1) * G; ++k) s += (int32_t)qa[m * K + k] * (int32_t)qw[n * K + k];
        y += ((double)s * (double)s_a[m * ng + g]) * (double)s_w[n * ng + g];
      }
      if (bias) y += (double)bias[n];
      if (y64) y64[m * N + n] = y;
      if (ybf16) ybf16[m * N + n] = oracle_bf16_rne(y);
    }
}

/* ---- training side: fake quantisation and the straight-through estimator ----------------
 *
 * Stage 1 of Theseus QAD (Sec. 3, Algorithm 1) updates the student's parameters by gradient
 * descent through its quantised blocks, and the paper names the straight-through estimator
 * (STE) as the gradient rule that 4-bit activations pass through (Sec. 3, "Why QAT fails";
 * Fig. "STE instability").  It prints neither the forward nor the backward rule.  The reading
 * computed here:
 *   forward   xhat = q * s for every element, where q = clamp(rint(fl32(x / s)), -8, 7) is the
 *             deployed quantiser's code and s is the group's scale: amax/7 of the group as in
 *             the file header, or a positive finite scale the caller gives (a learned one);
 *             q * s is formed exactly (fp64) and rounded once to the input's type (bf16 or fp32,
 *             nearest even);
 *   backward  dL/dx = dL/dxhat where the unclamped code rint(fl32(x / s)) lies in [-8, 7], and
 *             +0 where the clamp acted; the scale is held constant (no gradient reaches s).
 * With the amax scale every |x / s| is at most about 7, so no code reaches the clamp and the
 * mask is all ones; a group whose amax is 0 has s = 0, xhat = 0 and mask 1.  A zero code gives
 * xhat = +0 whatever the sign of x (the code, an integer, has none).
 */

/* One group of G fp32 values.  s_given: NULL for the amax rule, else the scale to use.
 * Writes the exact products q*s (fp64) and the pass-through mask; returns the scale used. */
static float fake_quant_group(const float* xf, int64_t G, const float* s_given, double* xhat,
                              uint8_t* mask) {
  float s;
  if (s_given) {
    s = *s_given;
  } else {
    float amax = 0.0f;
    for (int64_t k = 0; k < G; ++k) {
      float a = fabsf(xf[k]);
      if (a > amax) amax = a;
    }
    if (amax == 0.0f) {
      for (int64_t k = 0; k < G; ++k) {
        xhat[k] = 0.0;
        mask[k] = 1;
      }
      return 0.0f;
    }
    s = amax / 7.0f;                       /* IEEE single division */
  }
  for (int64_t k = 0; k < G; ++k) {
    float r = rintf(xf[k] / s);            /* IEEE single division, then half to even */
    mask[k] = (r >= -8.0f && r <= 7.0f) ? 1 : 0;
    if (r > 7.0f) r = 7.0f;
    if (r < -8.0f) r = -8.0f;
    const int q = (int)r;                  /* the code is an integer: code 0 gives +0, never -0 */
    xhat[k] = (double)q * (double)s;       /* exact: a 4-bit integer times a 24-bit significand */
  }
  return s;
}

/* Activations: bf16 [M, K] (dense rows) -> xhat bf16 [M, K], mask u8 [M, K] and the scales used
 * [M, K/G].  s_in: NULL (amax rule) or [M, K/G] positive finite scales. */
void oracle_fake_quant_bf16(const uint16_t* x, int64_t M, int64_t K, int64_t G, const float* s_in,
                            uint16_t* xhat, uint8_t* mask, float* s_out) {
  const int64_t ng = K / G;
#pragma omp parallel for schedule(static)
  for (int64_t m = 0; m < M; ++m) {
    float* xf = (float*)malloc((size_t)G * sizeof(float));
    double* e = (double*)malloc((size_t)G * sizeof(double));
    for (int64_t g = 0; g < ng; ++g) {
      const int64_t o = m * K + g * G;
      for (int64_t k = 0; k < G; ++k) xf[k] = bf16_bits_to_float(x[o + k]);
      s_out[m * ng + g] = fake_quant_group(xf, G, s_in ? s_in + m * ng + g : NULL, e, mask + o);
      for (int64_t k = 0; k < G; ++k) xhat[o + k] = oracle_bf16_rne(e[k]);
    }
    free(e);
    free(xf);
  }
}

/* Weights: fp32 [N, K] -> xhat fp32 [N, K] (the exact product rounded once to fp32), mask and
 * scales as above. */
void oracle_fake_quant_f32(const float* w, int64_t N, int64_t K, int64_t G, const float* s_in,
                           float* what, uint8_t* mask, float* s_out) {
  const int64_t ng = K / G;
#pragma omp parallel for schedule(static)
  for (int64_t n = 0; n < N; ++n) {
    double* e = (double*)malloc((size_t)G * sizeof(double));
    for (int64_t g = 0; g < ng; ++g) {
      const int64_t o = n * K + g * G;
      s_out[n * ng + g] = fake_quant_group(w + o, G, s_in ? s_in + n * ng + g : NULL, e, mask + o);
      for (int64_t k = 0; k < G; ++k) what[o + k] = (float)e[k];  /* round to nearest even */
    }
    free(e);
  }
}

/* STE backward on bf16 gradients: grad_x = grad where mask is 1, +0 where it is 0. */
void oracle_ste_backward_bf16(const uint16_t* grad, const uint8_t* mask, int64_t n, uint16_t* grad_x) {
  for (int64_t i = 0; i < n; ++i) grad_x[i] = mask[i] ? grad[i] : (uint16_t)0;
}

/* ---- DiT-XL/2 neighbour operations fused with the activation quantiser ---
 *
 * In a DiT-XL/2 block (the 0.6B model of the paper's Sec. 1 deployment remark
 * and of its W4A4 / W1.58A4 group128 experiments, Appendix table "DiT-XL/2
 * experimental details") the inputs of the block linears come from small
 * elementwise operations: the adaLN modulation x (1 + scale) + shift of the
 * normalised tokens feeds the attention's QKV projection and the MLP's first
 * linear, and the MLP's GELU (tanh approximation) feeds its second linear.
 * The paper prints neither operation; these are the readings:
 *   - modulation: per token m of sample b = m / T (T tokens per sample) and
 *     channel k, the bf16 value the linear layer receives is
 *         z = bf16( fl32( fl32( x * fl32(1 + scale[b,k]) ) + shift[b,k] ) ),
 *     each step an IEEE single operation (no fused multiply-add), rounded
 *     once to bf16 (nearest even);
 *   - GELU: the tanh approximation 0.5 h (1 + tanh(sqrt(2/pi) (h + 0.044715 h^3)))
 *     evaluated in fp32 by a fully specified sequence of IEEE single operations
 *     (oracle_gelu_tanh_f32: 1 + tanh(u) as 2 sigma(2u), the logistic through
 *     an exponential of Cody and Waite's reduction and a degree-8 Taylor
 *     polynomial), then rounded to bf16, as a bf16 model evaluates it (in fp32,
 *     then stored in bf16).  The kernels execute the same operations, so the
 *     two agree bit for bit; the fp32 value is within a few ulps of the exact
 *     GELU where h >= -9 (below that the logistic underflows: |GELU| < 2^-105).
 * Then z is quantised by the activation rule of the file header.  The
 * functions also return z, so that the two steps can be checked apart.
 */

static uint16_t modulate_bf16(float x, float shift, float scale) {
  const float one_plus = 1.0f + scale; /* IEEE single */
  const float t = x * one_plus;        /* IEEE single */
  const float z = t + shift;           /* IEEE single */
  return oracle_bf16_rne((double)z);   /* exact widening, one rounding to bf16 */
}

/* 2^n as an fp32 (n in [-126, 127]), built from its bit pattern. */
static float pow2_f32(int n) {
  const uint32_t u = (uint32_t)(n + 127) << 23;
  float f;
  memcpy(&f, &u, sizeof f);
  return f;
}

/* e^x for x <= 0 in fp32 steps.  Cody and Waite's argument reduction: n = rint(x log2 e),
 * r = x - n ln2 with ln2 split into a 15-bit high part (whose product with n is exact for
 * |n| <= 150) and a low part, each subtracted by one fused multiply-add; e^r by its Taylor
 * polynomial to degree 8 in Horner form with fused multiply-adds (|r| <= 0.35, the truncation
 * below 2^-32); then e^x = 2^n e^r, the power of two applied by one product, or by two where
 * 2^n is below the normal range (each product one IEEE rounding).  Below x = -104, e^x rounds
 * to 0 in fp32 and 0 is returned. */
static float exp_neg_f32(float x) {
  if (x < -104.0f) return 0.0f;
  const float n = rintf(x * 0x1.715476p+0f);
  float r = fmaf(-n, 0x1.62e4p-1f, x);
  r = fmaf(-n, 0x1.7f7d1cp-20f, r);
  float p = 0x1.a01a02p-16f;        /* 1/8! */
  p = fmaf(p, r, 0x1.a01a02p-13f);  /* 1/7! */
  p = fmaf(p, r, 0x1.6c16c2p-10f);  /* 1/6! */
  p = fmaf(p, r, 0x1.111112p-7f);   /* 1/5! */
  p = fmaf(p, r, 0x1.555556p-5f);   /* 1/4! */
  p = fmaf(p, r, 0x1.555556p-3f);   /* 1/3! */
  p = fmaf(p, r, 0x1p-1f);          /* 1/2! */
  p = fmaf(p, r, 1.0f);
  p = fmaf(p, r, 1.0f);
  const int ni = (int)n;
  if (ni >= -126) return p * pow2_f32(ni);
  return (p * pow2_f32(ni + 64)) * 0x1p-64f;
}

/* The tanh GELU of one value in fp32 steps (the reading in the section header):
 * u = fl32(0.7978846 * fl32(h + fl32(0.044715 * fl32(fl32(h * h) * h)))), sigma(2u) as
 * 1 / (1 + e^{-2u}) for u >= 0 and e^{2u} / (1 + e^{2u}) for u < 0 (exp_neg_f32), and
 * g = fl32(h * sigma); +-0 gives +-0. */
float oracle_gelu_tanh_f32(float h) {
  if (h == 0.0f) return h;
  const float h3 = (h * h) * h;
  const float p = h + 0x1.6e4e26p-5f * h3;
  const float u = 0x1.988454p-1f * p;
  float sig;
  if (u >= 0.0f) {
    sig = 1.0f / (1.0f + exp_neg_f32(-2.0f * u));
  } else {
    const float e = exp_neg_f32(2.0f * u);
    sig = e / (1.0f + e);
  }
  return h * sig;
}

void oracle_modulate_quantize_bf16(const uint16_t* x, int64_t M, int64_t K, int64_t ldx, const float* shift,
                                   const float* scale, int64_t tokens_per_sample, int64_t G, uint16_t* z,
                                   int8_t* codes, float* scales) {
  const int64_t ng = K / G;
#pragma omp parallel for schedule(static)
  for (int64_t m = 0; m < M; ++m) {
    const int64_t b = m / tokens_per_sample;
    float* zf = (float*)malloc((size_t)K * sizeof(float));
    for (int64_t k = 0; k < K; ++k) {
      const uint16_t zb = modulate_bf16(bf16_bits_to_float(x[m * ldx + k]), shift[b * K + k], scale[b * K + k]);
      z[m * K + k] = zb;
      zf[k] = bf16_bits_to_float(zb);
    }
    for (int64_t g = 0; g < ng; ++g)
      scales[m * ng + g] = quantize_group(zf + g * G, G, codes + m * K + g * G);
    free(zf);
  }
}

void oracle_gelu_quantize_bf16(const uint16_t* h, int64_t M, int64_t K, int64_t ldh, int64_t G, uint16_t* z,
                               int8_t* codes, float* scales) {
  const int64_t ng = K / G;
#pragma omp parallel for schedule(static)
  for (int64_t m = 0; m < M; ++m) {
    float* zf = (float*)malloc((size_t)K * sizeof(float));
    for (int64_t k = 0; k < K; ++k) {
      const uint16_t zb = oracle_bf16_rne((double)oracle_gelu_tanh_f32(bf16_bits_to_float(h[m * ldh + k])));
      z[m * K + k] = zb;
      zf[k] = bf16_bits_to_float(zb);
    }
    for (int64_t g = 0; g < ng; ++g)
      scales[m * ng + g] = quantize_group(zf + g * G, G, codes + m * K + g * G);
    free(zf);
  }
}
