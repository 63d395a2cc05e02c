/*
 * hscale_oracle.c -- CPU oracle for the H-Scale hot path.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is a plain, slow, fp64 restatement of
 * what the paper "H-Scale: Hessian-Guided Scale Refinement for NVFP4 Sub-Byte
 * LLM Inference" defines.  Only the tests, the smoke check and the benchmark's
 * CPU-baseline leg may load it; the CUDA library never does.  It shares no
 * code, header, table or constant generator with the CUDA library: every format
 * is decoded here from its bit fields and every rounding decision is taken by
 * exact fp64 comparison.
 *
 * Equation numbers follow the paper's order: Eq. 1 effective scale s = s_g*l,
 * Eq. 2 quantizer s*Clip(Round(w/s)), Eq. 3 layer-output objective, Eq. 4
 * h = diag(X^T X), Eq. 5 decoupled weighted loss, Eq. 6 group objective, Eq. 7
 * l_init = Q_fp8(s_init/s_g), Eq. 8 E4M3 ladder, Eq. 9 shift set, Eq. 10 clipped
 * walk, Eq. 11 candidate set, Eq. 12 FP4 projection, Eq. 13 argmin.
 *
 * What each function follows:
 *   oracle_hessian_accumulate   h += diag(X^T X) over a token chunk      (Sec. 3.2, Eq. 4)
 *   oracle_global_scale         s_g = amax|W| / (6*448); the paper names a tensor-level
 *                               FP32 global scale (Sec. 3.1, Eq. 1) but prints no
 *                               formula: this is the standard NVFP4 choice that puts
 *                               the largest group exactly on the top E4M3 code
 *   oracle_rtn_codes            l_init = Q_fp8(s_init / s_g), s_init = amax_group / 6
 *                               (Sec. 3.3 "Initialization", Eq. 7)
 *   oracle_refine               Algorithm 1 (HScaleGroupQuantize): clipped walk on the
 *                               E4M3 ladder (Eqs. 8-10), candidate set (Eq. 11), FP4
 *                               projection (Eq. 12), argmin of the diagonal-Hessian
 *                               weighted error (Eqs. 6 and 13), final re-quantization
 *   oracle_refine_f64           Algorithm 1 on fp64 weights: the local quantizer of
 *                               Algorithm 3 (GPTQ + H-Scale), whose running weights are fp64
 *   oracle_hessian_full         H += X^T X, the GPTQ Hessian of Algorithm 3
 *   oracle_fourover6_codes      Algorithm 2's initialization: the better of the anchors
 *                               m/4 and m/6 by plain MSE (Sec. 3.5, Algorithm 2)
 *   oracle_pack                 final FP4 quantization with given local scales (Sec. 3.3
 *                               "Final re-quantization"; quantizer of Eq. 2)
 *   oracle_quantize_at_scale    Eq. 2 at a real scale s (calibration microcase, App. A.1)
 *   oracle_dequant_residual     dW = W - W_hat of the packed NVFP4 weights (the dW of Eq. 3;
 *                               W_hat = s_g * E4M3(code) * E2M1(nibble), Eqs. 1-2)
 *   oracle_output_error         ||X dW^T||_F^2 (Eq. 3)
 *
 * Parity unpinned: the paper does not fix these conventions, so no pin can check
 * them, and they are readings: the order among exactly equal errors, the sign
 * nibble of a code that rounds to zero, the nibble order inside a byte, s_g when W
 * is all zero, the clamp of a code-0 RTN scale to code 1, the rounding mode of
 * Q_fp8 (round-to-nearest-even, saturating), and that w/s is the exact real quotient.
 *
 * Built with -ffp-contract=off so that no multiply-add is fused behind our back.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <stddef.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* ------------------------------------------------------------------ */
/* threading (only affects speed: every output is computed by the same */
/* sequential fp64 arithmetic whatever the thread count)               */
/* ------------------------------------------------------------------ */
void oracle_set_threads(int n) {
#ifdef _OPENMP
  if (n > 0) omp_set_num_threads(n);
#else
  (void)n;
#endif
}

int oracle_max_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}

/* ------------------------------------------------------------------ */
/* formats                                                             */
/* ------------------------------------------------------------------ */

/* bfloat16 bit pattern -> its exact value (bf16 is the top half of an IEEE binary32). */
static double bf16_value(uint16_t bits) {
  uint32_t u = (uint32_t)bits << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return (double)f;
}

static int bf16_sign(uint16_t bits) { return (bits >> 15) & 1; }

/* OCP FP8 E4M3 ("E4M3FN"): 1 sign, 4 exponent bits (bias 7), 3 mantissa bits,
 * no infinities, S.1111.111 is NaN.  Decoded from the bit fields.
 * The sorted positive finite values are the ladder L+ of Eq. 8 (M = 126 values,
 * bytes 0x01..0x7E), and the byte is the index iota of Algorithm 1. */
double oracle_e4m3_decode(uint8_t byte) {
  int s = byte >> 7, e = (byte >> 3) & 15, m = byte & 7;
  double v;
  if (e == 15 && m == 7) return NAN;
  if (e == 0)
    v = ldexp((double)m, -9);            /* subnormal: m/8 * 2^(1-7) */
  else
    v = ldexp((double)(8 + m), e - 10);  /* (1 + m/8) * 2^(e-7) */
  return s ? -v : v;
}

/* FP4 E2M1: 1 sign, 2 exponent bits (bias 1), 1 mantissa bit; magnitudes
 * {0, 0.5, 1, 1.5, 2, 3, 4, 6}.  Decoded from the bit fields. */
double oracle_e2m1_decode(uint8_t nibble) {
  int s = (nibble >> 3) & 1, e = (nibble >> 1) & 3, m = nibble & 1;
  double v = (e == 0) ? 0.5 * m : ldexp(1.0 + 0.5 * m, e - 1);
  return s ? -v : v;
}

#define E4M3_MAX_CODE 126 /* M of Eq. 8: index of 448 */
#define E2M1_MAX_CODE 7   /* magnitude code of 6.0 */

/* Round-to-nearest-even with saturation onto the E4M3 ladder (code 0 = value 0
 * included) of the real number  num / (k * s_g).  Decided by exact comparisons of
 * num against k * mu * s_g for each midpoint mu of consecutive ladder values:
 * mu has <= 5 significant bits, k <= 2 bits, s_g 24 bits, so k*mu*s_g has <= 31
 * bits and is exact in fp64.  Ties go to the code with an even last mantissa bit
 * (the even code).  Values above the last midpoint saturate to 448 (code 126). */
static int e4m3_rne_sat_quotient(double num, double k, double s_g) {
  int c = 0;
  for (int i = 1; i <= E4M3_MAX_CODE; ++i) {
    double mu = 0.5 * (oracle_e4m3_decode((uint8_t)(i - 1)) + oracle_e4m3_decode((uint8_t)i));
    double t = k * mu * s_g;
    if (num > t) {
      c = i;
    } else {
      if (num == t) c = (i % 2 == 0) ? i : i - 1;
      break;
    }
  }
  return c;
}

/* Round-to-nearest-even with saturation onto the E2M1 magnitude grid of the real
 * number a / scale (Round and Clip of Eq. 2; Clip bounds to [-6, 6]).  Exact
 * comparisons of a against mid * scale: for an effective scale s_g * l (28 bits)
 * the product has <= 31 bits.  Ties go to the even code. */
static int e2m1_rne_sat_quotient(double a, double scale) {
  int c = 0;
  for (int i = 1; i <= E2M1_MAX_CODE; ++i) {
    double mid = 0.5 * (oracle_e2m1_decode((uint8_t)(i - 1)) + oracle_e2m1_decode((uint8_t)i));
    double t = mid * scale;
    if (a > t) {
      c = i;
    } else {
      if (a == t) c = (i % 2 == 0) ? i : i - 1;
      break;
    }
  }
  return c;
}

/* ------------------------------------------------------------------ */
/* Hessian diagonal: h_j += sum_t x_tj^2  (Sec. 3.2, Eq. 4)               */
/* ------------------------------------------------------------------ */
void oracle_hessian_accumulate(const uint16_t* x, int64_t tokens, int64_t n, int64_t ld,
                               double* h) {
  if (tokens <= 0 || n <= 0) return;
  const int64_t block = 64;
  const int64_t nblocks = (n + block - 1) / block;
#pragma omp parallel for schedule(static)
  for (int64_t b = 0; b < nblocks; ++b) {
    int64_t j0 = b * block, j1 = j0 + block < n ? j0 + block : n;
    for (int64_t t = 0; t < tokens; ++t) {
      const uint16_t* row = x + t * ld;
      for (int64_t j = j0; j < j1; ++j) {
        double v = bf16_value(row[j]);
        h[j] += v * v;
      }
    }
  }
}

/* ------------------------------------------------------------------ */
/* global scale                                                        */
/* ------------------------------------------------------------------ */
/* s_g = fl32(amax|W| / (6 * 448)).  The fp64 quotient rounded to fp32 equals the
 * correctly rounded fp32 quotient (53 >= 2*24 + 2).  amax = 0 gives s_g = 1. */
float oracle_global_scale(const uint16_t* w, int64_t count, double* amax_out) {
  double amax = 0.0;
  for (int64_t i = 0; i < count; ++i) {
    double a = fabs(bf16_value(w[i]));
    if (a > amax) amax = a;
  }
  if (amax_out) *amax_out = amax;
  if (amax == 0.0) return 1.0f;
  return (float)(amax / (6.0 * 448.0));
}

/* ------------------------------------------------------------------ */
/* RTN local-scale code of one group (Sec. 3.3 "Initialization", Eq. 7) */
/* ------------------------------------------------------------------ */
/* s_init = amax_group / 6 (max-abs scale), l_init = Q_fp8(s_init / s_g): the E4M3
 * round-to-nearest-even (saturating) of amax_group / (6 s_g).  A result of code 0
 * (value 0, not on the ladder L+) is clamped to code 1, as the walk of Eq. 10 clips
 * indices to [1, M]. */
static int rtn_code_of_values(const double* v, double s_g) {
  double amax = 0.0;
  for (int j = 0; j < 16; ++j) {
    double a = fabs(v[j]);
    if (a > amax) amax = a;
  }
  int c = e4m3_rne_sat_quotient(amax, 6.0, s_g);
  return c < 1 ? 1 : c;
}

/* the 16 values of a bf16 group (exact in fp64) */
static void group_values(const uint16_t* g, double* v) {
  for (int j = 0; j < 16; ++j) v[j] = bf16_value(g[j]);
}

static int rtn_code_of_group(const uint16_t* g, double s_g) {
  double v[16];
  group_values(g, v);
  return rtn_code_of_values(v, s_g);
}

void oracle_rtn_codes(const uint16_t* w, int64_t m, int64_t n, float s_g, uint8_t* codes) {
  const int64_t ng = n / 16;
#pragma omp parallel for schedule(static)
  for (int64_t r = 0; r < m; ++r)
    for (int64_t i = 0; i < ng; ++i)
      codes[r * ng + i] = (uint8_t)rtn_code_of_group(w + r * n + i * 16, (double)s_g);
}

/* ------------------------------------------------------------------ */
/* one group under one candidate local scale                           */
/* ------------------------------------------------------------------ */
/* E(s) = sum_j h_j (w_j - s q_j)^2 with s = s_g * lambda_c (Eqs. 6, 12, 13).
 * s (<= 28 bits), q_j * s (<= 30 bits) and the residual are exact in fp64; only the
 * squares and the sum round (relative error ~1e-16).  Returns E; writes the magnitude
 * codes if q != NULL. */
static double group_error_values(const double* v, const float* h, double s_g, int code, uint8_t* q) {
  const double scale = s_g * oracle_e4m3_decode((uint8_t)code);
  double e = 0.0;
  for (int j = 0; j < 16; ++j) {
    double a = fabs(v[j]);
    int k = e2m1_rne_sat_quotient(a, scale);
    double d = a - oracle_e2m1_decode((uint8_t)k) * scale;
    double hj = h ? (double)h[j] : 1.0;
    e += hj * d * d;
    if (q) q[j] = (uint8_t)k;
  }
  return e;
}

static double group_error(const uint16_t* g, const float* h, double s_g, int code, uint8_t* q) {
  double v[16];
  group_values(g, v);
  return group_error_values(v, h, s_g, code, q);
}

/* nibble = sign(w) << 3 | magnitude code (E2M1 bit layout S.EE.M); the sign bit is
 * the sign bit of w, so a negative weight that rounds to 0 gives 0x8.  Element 2j
 * goes to the low nibble of byte j, element 2j+1 to the high nibble. */
static void pack_group(const uint16_t* g, const uint8_t* q, uint8_t* out8) {
  for (int j = 0; j < 8; ++j) {
    uint8_t lo = (uint8_t)((bf16_sign(g[2 * j]) << 3) | q[2 * j]);
    uint8_t hi = (uint8_t)((bf16_sign(g[2 * j + 1]) << 3) | q[2 * j + 1]);
    out8[j] = (uint8_t)(lo | (hi << 4));
  }
}

/* ------------------------------------------------------------------ */
/* Algorithm 1, HScaleGroupQuantize                                    */
/* ------------------------------------------------------------------ */
/* For every row-group pair:
 *   c <- iota(l_init) (given init code, or the RTN code of the group)
 *   for delta = -D..U:  l(delta) = lambda_clip(c + delta, 1, M)          (Eq. 10)
 *   S = { s_g * l }                                                     (Eq. 11)
 *   E(s) = || (w - Q_fp4(w/s) s) (.) sqrt(h) ||^2                       (Eqs. 12, 13)
 *   s* = argmin E; store Q_fp4(w/s*) and the code of s*.
 * Tie rule (the paper only says argmin): smallest E, then smallest |shift|, then the
 * smaller shift, where the shift is the realised code minus c; codes repeated by the
 * clip are one candidate.  Diagnostics per group (any pointer may be NULL):
 *   near_tie: 1 iff the best and the runner-up among distinct codes satisfy
 *             E2 - E1 <= 1e-6 * E2 (both zero counts as a tie); 0 with one code.
 *   delta:    chosen code - c;  e_best, e_init (shift 0), e_second (runner-up or -1). */
/* Algorithm 1 on one group of values (see above); returns the chosen code and writes the
 * magnitude codes of the final quantization and the diagnostics. */
static int refine_group(const double* v, const float* hg, double s_g, int c, int down, int up, uint8_t* q,
                        uint8_t* near_tie, int16_t* delta_out, double* e_best, double* e_init,
                        double* e_second) {
  /* errors by code; a code repeated by the clip is evaluated once */
  double err[E4M3_MAX_CODE + 1];
  for (int k = 0; k <= E4M3_MAX_CODE; ++k) err[k] = -1.0;
  int best = -1, best_shift = 0;
  double best_e = 0.0;
  for (int d = -down; d <= up; ++d) {
    int cc = c + d;
    if (cc < 1) cc = 1;
    if (cc > E4M3_MAX_CODE) cc = E4M3_MAX_CODE;
    if (err[cc] < 0.0) err[cc] = group_error_values(v, hg, s_g, cc, NULL);
    double e = err[cc];
    int shift = cc - c;
    int better = 0;
    if (best < 0 || e < best_e) better = 1;
    else if (e == best_e && cc != best) {
      int as = shift < 0 ? -shift : shift, ab = best_shift < 0 ? -best_shift : best_shift;
      if (as < ab || (as == ab && shift < best_shift)) better = 1;
    }
    if (better) { best = cc; best_e = e; best_shift = shift; }
  }
  const double e0 = err[c];
  /* runner-up over the distinct codes other than the winner */
  double second = -1.0;
  for (int cc = 1; cc <= E4M3_MAX_CODE; ++cc)
    if (cc != best && err[cc] >= 0.0 && (second < 0.0 || err[cc] < second)) second = err[cc];
  group_error_values(v, hg, s_g, best, q);
  if (near_tie) *near_tie = (uint8_t)(second >= 0.0 && (second - best_e) <= 1e-6 * second);
  if (delta_out) *delta_out = (int16_t)best_shift;
  if (e_best) *e_best = best_e;
  if (e_init) *e_init = e0;
  if (e_second) *e_second = second;
  return best;
}

void oracle_refine(const uint16_t* w, const float* h, int64_t m, int64_t n, float s_g_f,
                   const uint8_t* init_codes, int down, int up, uint8_t* codes_out,
                   uint8_t* packed_out, uint8_t* near_tie, int16_t* delta_out, double* e_best,
                   double* e_init, double* e_second) {
  const int64_t ng = n / 16;
  const double s_g = (double)s_g_f;
#pragma omp parallel for schedule(static)
  for (int64_t r = 0; r < m; ++r) {
    for (int64_t i = 0; i < ng; ++i) {
      const int64_t gi = r * ng + i;
      const uint16_t* g = w + r * n + i * 16;
      const float* hg = h ? h + i * 16 : NULL;
      double v[16];
      group_values(g, v);
      int c;
      if (init_codes) {
        c = init_codes[gi] & 0x7F;
        if (c < 1) c = 1;
        if (c > E4M3_MAX_CODE) c = E4M3_MAX_CODE;
      } else {
        c = rtn_code_of_values(v, s_g);
      }
      uint8_t q[16];
      const int best = refine_group(v, hg, s_g, c, down, up, q, near_tie ? near_tie + gi : NULL,
                                    delta_out ? delta_out + gi : NULL, e_best ? e_best + gi : NULL,
                                    e_init ? e_init + gi : NULL, e_second ? e_second + gi : NULL);
      if (codes_out) codes_out[gi] = (uint8_t)best;
      if (packed_out) pack_group(g, q, packed_out + gi * 8);
    }
  }
}

/* Algorithm 1 on real-valued (fp64) weights W [m, n] with the RTN initial codes of Eq. 7,
 * the local quantizer inside GPTQ (Algorithm 3), where the running weights are no longer
 * bf16.  Rounding decisions stay exact: |w| is compared with mid * s (<= 31 bits, exact)
 * in fp64.  Writes the codes [m, n/16], the signed dequantized values
 * W_hat = sign(w) s q [m, n], the packed nibbles [m, n/2] and the near-tie flags
 * [m, n/16] (any output may be NULL). */
void oracle_refine_f64(const double* w, const float* h, int64_t m, int64_t n, float s_g_f, int down, int up,
                       uint8_t* codes_out, double* w_hat, uint8_t* packed_out, uint8_t* near_tie) {
  const int64_t ng = n / 16;
  const double s_g = (double)s_g_f;
#pragma omp parallel for schedule(static)
  for (int64_t r = 0; r < m; ++r) {
    for (int64_t i = 0; i < ng; ++i) {
      const int64_t gi = r * ng + i;
      const double* v = w + r * n + i * 16;
      const float* hg = h ? h + i * 16 : NULL;
      uint8_t q[16];
      const int best = refine_group(v, hg, s_g, rtn_code_of_values(v, s_g), down, up, q,
                                    near_tie ? near_tie + gi : NULL, NULL, NULL, NULL, NULL);
      if (codes_out) codes_out[gi] = (uint8_t)best;
      const double scale = s_g * oracle_e4m3_decode((uint8_t)best);
      for (int j = 0; j < 16; ++j) {
        const double mag = oracle_e2m1_decode(q[j]) * scale;
        if (w_hat) w_hat[r * n + i * 16 + j] = signbit(v[j]) ? -mag : mag;
      }
      if (packed_out)
        for (int j = 0; j < 8; ++j) {
          uint8_t lo = (uint8_t)(((signbit(v[2 * j]) ? 1 : 0) << 3) | q[2 * j]);
          uint8_t hi = (uint8_t)(((signbit(v[2 * j + 1]) ? 1 : 0) << 3) | q[2 * j + 1]);
          packed_out[gi * 8 + j] = (uint8_t)(lo | (hi << 4));
        }
    }
  }
}

/* Full Hessian H += X^T X over a token chunk (the GPTQ Hessian of Algorithm 3; its
 * diagonal is the h of Eq. 4): plain fp64 sums in token order. */
void oracle_hessian_full(const uint16_t* x, int64_t tokens, int64_t n, int64_t ld, double* H) {
#pragma omp parallel for schedule(static)
  for (int64_t i = 0; i < n; ++i)
    for (int64_t t = 0; t < tokens; ++t) {
      const double xi = bf16_value(x[t * ld + i]);
      if (xi == 0.0) continue;
      for (int64_t j = 0; j < n; ++j) H[i * n + j] += xi * bf16_value(x[t * ld + j]);
    }
}

/* All candidate errors of one group over an explicit code list (tests: full-grid and
 * brute-force comparisons).  err[k] = E(codes[k]). */
void oracle_group_errors(const uint16_t* g16, const float* h16, float s_g, const uint8_t* codes,
                         int count, double* err) {
  for (int k = 0; k < count; ++k) err[k] = group_error(g16, h16, (double)s_g, codes[k], NULL);
}

/* ------------------------------------------------------------------ */
/* Algorithm 2, 4over6 initialization (the part before HScaleGroupQuantize) */
/* ------------------------------------------------------------------ */
/* For every group: m = max|w|; for each anchor c in C = {4, 6}, in that order,
 *   l_c = Q_fp8(m / (c s_g))   (round-to-nearest-even, saturating; code 0 clamps to 1,
 *                               the same reading as Eq. 7)
 *   L(c) = || w - Q_fp4(w / (s_g l_c)) s_g l_c ||^2      (plain weight MSE)
 * and the initial code is the code of argmin_c L(c); the first anchor in the order of C
 * wins an exact tie (a reading: the paper writes argmin over C without a tie rule).
 * near_tie (may be NULL): 1 iff the two anchors give different codes whose errors are
 * within 1e-6 relative of each other. */
void oracle_fourover6_codes(const uint16_t* w, int64_t m, int64_t n, float s_g_f,
                            uint8_t* codes_out, uint8_t* near_tie) {
  const int64_t ng = n / 16;
  const double s_g = (double)s_g_f;
#pragma omp parallel for schedule(static)
  for (int64_t r = 0; r < m; ++r) {
    for (int64_t i = 0; i < ng; ++i) {
      const uint16_t* g = w + r * n + i * 16;
      double mx = 0.0;
      for (int j = 0; j < 16; ++j) {
        double a = fabs(bf16_value(g[j]));
        if (a > mx) mx = a;
      }
      const double anchors[2] = {4.0, 6.0};
      int code[2];
      double err[2];
      for (int k = 0; k < 2; ++k) {
        int c = e4m3_rne_sat_quotient(mx, anchors[k], s_g);
        code[k] = c < 1 ? 1 : c;
        err[k] = group_error(g, NULL, s_g, code[k], NULL);
      }
      const int pick = err[1] < err[0] ? 1 : 0;
      codes_out[r * ng + i] = (uint8_t)code[pick];
      if (near_tie) {
        const double hi = err[0] > err[1] ? err[0] : err[1];
        const double lo = err[0] > err[1] ? err[1] : err[0];
        near_tie[r * ng + i] = (uint8_t)(code[0] != code[1] && hi - lo <= 1e-6 * hi);
      }
    }
  }
}

/* ------------------------------------------------------------------ */
/* final FP4 quantization with given local-scale codes                 */
/* ------------------------------------------------------------------ */
void oracle_pack(const uint16_t* w, int64_t m, int64_t n, float s_g, const uint8_t* codes,
                 uint8_t* packed_out) {
  const int64_t ng = n / 16;
#pragma omp parallel for schedule(static)
  for (int64_t r = 0; r < m; ++r) {
    for (int64_t i = 0; i < ng; ++i) {
      const int64_t gi = r * ng + i;
      uint8_t q[16];
      int c = codes[gi] & 0x7F;  /* a code off the ladder is read as its clipped index (Eq. 10) */
      if (c < 1) c = 1;
      if (c > E4M3_MAX_CODE) c = E4M3_MAX_CODE;
      group_error(w + r * n + i * 16, NULL, (double)s_g, c, q);
      pack_group(w + r * n + i * 16, q, packed_out + gi * 8);
    }
  }
}

/* ------------------------------------------------------------------ */
/* Eq. 2 quantizer at an arbitrary real scale (Appendix A.1 microcase)    */
/* ------------------------------------------------------------------ */
/* w_hat_j = s * sign(w_j) * Clip(Round(|w_j| / s)); codes_out gets the signed grid
 * value index as sign * magnitude-code.  Comparisons are a > mid * s in fp64. */
void oracle_quantize_at_scale(const double* w, int64_t len, double s, double* w_hat,
                              int8_t* codes_out) {
  for (int64_t j = 0; j < len; ++j) {
    double a = fabs(w[j]);
    int k = e2m1_rne_sat_quotient(a, s);
    double v = oracle_e2m1_decode((uint8_t)k) * s;
    w_hat[j] = (w[j] < 0 || (w[j] == 0 && signbit(w[j]))) ? -v : v;
    if (codes_out) codes_out[j] = (int8_t)((w[j] < 0) ? -k : k);
  }
}

/* ||X dW^T||_F^2 = sum_r sum_t (sum_j X_tj dW_rj)^2 (Eq. 3); X is [N, n], dW is [m, n],
 * both row-major fp64. */
double oracle_output_error(const double* X, int64_t N, int64_t n, const double* dW, int64_t m) {
  /* one fp64 partial per output row, summed in row order afterwards, so the result does
   * not depend on the thread count */
  double* row_total = (double*)malloc((size_t)(m > 0 ? m : 1) * sizeof(double));
  if (row_total == NULL) return NAN;
#pragma omp parallel for schedule(static)
  for (int64_t r = 0; r < m; ++r) {
    double rt = 0.0;
    for (int64_t t = 0; t < N; ++t) {
      double acc = 0.0;
      for (int64_t j = 0; j < n; ++j) acc += X[t * n + j] * dW[r * n + j];
      rt += acc * acc;
    }
    row_total[r] = rt;
  }
  double total = 0.0;
  for (int64_t r = 0; r < m; ++r) total += row_total[r];
  free(row_total);
  return total;
}

/* ------------------------------------------------------------------ */
/* quantization residual dW = W - W_hat (the dW of Eq. 3)               */
/* ------------------------------------------------------------------ */
/* W_hat_j = sign(nibble_j) * s_g * E4M3(code of the group) * E2M1(magnitude of nibble_j),
 * the value the packed NVFP4 format encodes (Eq. 1 scale times the Eq. 2 grid value).  A
 * code off the ladder is read as its clipped index, as in oracle_pack.  s_g * l * q has at
 * most 24 + 4 + 2 significant bits, so W_hat is exact in fp64; dW is the fp64 rounding of
 * w - W_hat. */
void oracle_dequant_residual(const uint16_t* w, int64_t m, int64_t n, float s_g_f,
                             const uint8_t* codes, const uint8_t* packed, double* dw_out) {
  const double s_g = (double)s_g_f;
  const int64_t ng = n / 16;
#pragma omp parallel for schedule(static)
  for (int64_t r = 0; r < m; ++r) {
    for (int64_t i = 0; i < ng; ++i) {
      const int64_t gi = r * ng + i;
      int c = codes[gi] & 0x7F;
      if (c < 1) c = 1;
      if (c > E4M3_MAX_CODE) c = E4M3_MAX_CODE;
      const double s = s_g * oracle_e4m3_decode((uint8_t)c);
      for (int j = 0; j < 16; ++j) {
        const uint8_t nib = (uint8_t)((packed[gi * 8 + j / 2] >> (4 * (j & 1))) & 0xF);
        const double mag = s * oracle_e2m1_decode((uint8_t)(nib & 0x7));
        const double w_hat = (nib & 0x8) ? -mag : mag;
        const int64_t e = r * n + i * 16 + j;
        dw_out[e] = bf16_value(w[e]) - w_hat;
      }
    }
  }
}
