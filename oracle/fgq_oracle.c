/*
 * fgq_oracle.c -- CPU oracle for Fine-Grained Quantization (FGQ),
 * "Ternary Neural Networks with Fine-Grained Quantization" (arXiv 1705.01462).
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the plain, slow, obviously-correct statement
 * of what the FGQ hot path computes.  It is used by the test-suite, by the smoke check
 * and by the benchmark's CPU-baseline leg; nothing in the product library calls, links
 * or includes it, and it shares no code with the CUDA kernels.
 *
 * Arithmetic: exact integers (int64 / unsigned __int128) for every decision and every
 * group sum, fp64 for the fp32-output contraction.  Single threaded.
 *
 * Contents
 *   oracle_round_ratio_f32      exact round-to-nearest-even of S*2^u/k to fp32
 *   oracle_ternarize_group      Eq. 5 (and Eq. 4) for one group, exact
 *   oracle_ternarize_group_f64  the same rule in plain fp64 over a sort (any group size)
 *   oracle_ternarize            Eq. 2: independent groups of G along the reduction axis
 *   oracle_pack_codes           2-bit code words (encoding defined by this library)
 *   oracle_dfp_exponent         dynamic-fixed-point shared exponent (Section 4)
 *   oracle_quantize             DFP quantisation to 8/4-bit codes (Section 4)
 *   oracle_pack_act             8-bit bytes / 4-bit nibble packing
 *   oracle_conv2d               grouped contraction over explicit im2col (Eq. 2, Section 4)
 *   oracle_conv2d_at            the same at a list of output positions
 *   oracle_gemm                 grouped contraction for a [P][Kred] activation matrix
 *   oracle_group_sums           the int32-accumulator group sums s[m][g][p]
 *   oracle_conv2d_group_sums    the same sums of a convolution, at listed output positions
 *   oracle_conv2d_w8            dense 8-bit-weight convolution (first layer, Section 4)
 *   oracle_ternarize_threshold  ternarization at an analytical threshold (Section 3, Lemma 1),
 *                               per group or with one threshold and one alpha per layer
 *   oracle_ternary_error        per-group ternary error ||w - alpha t||^2 (Section 3)
 *   oracle_quantize_alpha       8/4-bit fixed-point alphas, one DFP exponent per filter
 *                               (Section 4)
 *
 * Readings of the paper that this file fixes (where the paper is silent):
 *   - Ties between candidate thresholds with exactly equal objective are broken towards
 *     the larger threshold (fewest kept weights).
 *   - alpha is the fp32 value nearest (ties to even) to the exact mean of the kept |w|.
 *   - DFP scale is a power of two 2^E, E the smallest integer with max|x|*2^-E <= qmax,
 *     clamped to [-149, 127] so that 2^E is an fp32 number; rounding is half-to-even;
 *     negative inputs of unsigned types saturate to 0.
 */
#include <math.h>
#include <stddef.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORACLE_OK 0
#define ORACLE_ERR_ARG 1
#define ORACLE_ERR_NONFINITE 4

#define ORACLE_U8 0
#define ORACLE_S8 1
#define ORACLE_U4 2
#define ORACLE_S4 3

#define ORACLE_MAX_G 128

typedef unsigned __int128 u128;

static uint32_t f32_bits(float x) {
  uint32_t b;
  memcpy(&b, &x, sizeof b);
  return b;
}

static int bitlen_u128(u128 v) {
  int n = 0;
  while (v) {
    v >>= 1;
    n++;
  }
  return n;
}

int oracle_abi_version(void) { return 1; }

/*
 * Exact fp32 rounding (nearest, ties to even, subnormals included) of the positive
 * rational S * 2^u / k, for 1 <= S < 2^63, 1 <= k <= 2^16.
 */
float oracle_round_ratio_f32(uint64_t S, uint32_t k, int u) {
  if (S == 0 || k == 0) return 0.0f;
  u128 num = ((u128)S) << 64;
  u128 q = num / k;
  int sticky = (num % k) != 0;
  int nb = bitlen_u128(q);          /* q >= 2^48, so nb >= 49 and drop >= 25 */
  int lead_exp = nb - 1 + u - 64;   /* binary exponent of the leading bit of the value */
  int lsb_exp = lead_exp >= -126 ? lead_exp - 23 : -149;
  int drop = lsb_exp - (u - 64);    /* low bits of q that fall below the fp32 lsb */
  u128 mant, rem, half;
  if (drop <= 0) {                  /* cannot happen for the callers in this file */
    return (float)ldexp((double)(uint64_t)q, u - 64);
  }
  mant = q >> drop;
  rem = q & ((((u128)1) << drop) - 1);
  half = ((u128)1) << (drop - 1);
  if (rem > half || (rem == half && (sticky || (mant & 1)))) mant += 1;
  return (float)ldexp((double)(uint64_t)mant, lsb_exp);
}

/*
 * Ternarize one group of G <= 128 fp32 weights (Section 3.1, Eq. 5; Eq. 4 reaches the
 * same optimum): choose the threshold Delta maximising (sum_{|w|>Delta} |w|)^2 /
 * |{|w|>Delta}|, then alpha = mean of the kept |w| and t_i = sign(w_i) for kept i.
 *
 * The distinct kept sets I_Delta are exactly {i : |w_i| >= tau} for tau running over
 * the non-zero magnitudes of the group, so the candidates are enumerated that way, each
 * with its own count k and sum S recomputed from scratch (O(G^2), no sorting).
 *
 * Exact arithmetic.  Let F = max(biased exponent of max|w|, 1).  Every magnitude whose
 * exponent is at least F-8 is an integer multiple of 2^(F-158) below 2^32, so sums of up
 * to 128 of them are exact in uint64 and S_a^2*k_b vs S_b^2*k_a is exact in 128 bits.
 * Thresholds below 2^(F-8-127) never win: at the optimum (kept count kopt, sum S) the
 * objective does not grow when its smallest kept magnitude a is dropped, which needs
 * a >= S_{kopt-1} (sqrt(kopt / (kopt-1)) - 1) > max|w| / (2 kopt - 1) >= max|w| / 255;
 * so such thresholds are skipped (a magnitude below every candidate is never kept).
 *
 * Returns ORACLE_OK, or ORACLE_ERR_NONFINITE (then t = 0 and alpha = 0).
 */
int oracle_ternarize_group(const float* w, int G, int8_t* t, float* alpha) {
  uint32_t mag[ORACLE_MAX_G];
  uint64_t A[ORACLE_MAX_G];
  int inwin[ORACLE_MAX_G];
  uint32_t mmax = 0;
  int i, c;
  if (G < 1 || G > ORACLE_MAX_G) return ORACLE_ERR_ARG;
  for (i = 0; i < G; i++) {
    mag[i] = f32_bits(w[i]) & 0x7fffffffu;
    if (mag[i] >= 0x7f800000u) {
      for (c = 0; c < G; c++) t[c] = 0;
      *alpha = 0.0f;
      return ORACLE_ERR_NONFINITE;
    }
    if (mag[i] > mmax) mmax = mag[i];
  }
  for (i = 0; i < G; i++) t[i] = 0;
  *alpha = 0.0f;
  if (mmax == 0) return ORACLE_OK;  /* all-zero group: alpha = 0, all codes 0 */

  {
    int F = (int)(mmax >> 23);
    if (F < 1) F = 1;
    for (i = 0; i < G; i++) {
      int f = (int)(mag[i] >> 23);
      uint64_t sig = f ? ((mag[i] & 0x7fffffu) | 0x800000u) : (mag[i] & 0x7fffffu);
      int fe = f ? f : 1;
      inwin[i] = mag[i] != 0 && fe >= F - 8;
      A[i] = inwin[i] ? (sig << (fe - F + 8)) : 0;
    }

    {
      uint64_t best_S = 0;
      uint64_t best_k = 0;
      uint32_t best_tau = 0;
      for (c = 0; c < G; c++) {
        uint32_t tau;
        uint64_t k = 0, S = 0;
        if (!inwin[c]) continue;
        tau = mag[c];
        for (i = 0; i < G; i++) {
          if (mag[i] >= tau) {
            k += 1;
            S += A[i];
          }
        }
        if (best_k == 0) {
          best_S = S;
          best_k = k;
          best_tau = tau;
        } else {
          u128 lhs = (u128)S * S * best_k;       /* J(candidate) * k * best_k */
          u128 rhs = (u128)best_S * best_S * k;  /* J(best)      * k * best_k */
          if (lhs > rhs || (lhs == rhs && k < best_k)) {
            best_S = S;
            best_k = k;
            best_tau = tau;
          }
        }
      }
      *alpha = oracle_round_ratio_f32(best_S, (uint32_t)best_k, F - 158);
      for (i = 0; i < G; i++) {
        if (mag[i] >= best_tau) t[i] = (f32_bits(w[i]) >> 31) ? -1 : 1;
      }
    }
  }
  return ORACLE_OK;
}

/* Descending comparator for qsort on doubles. */
static int cmp_desc(const void* a, const void* b) {
  double x = *(const double*)a, y = *(const double*)b;
  return (x < y) - (x > y);
}

/*
 * The Eq. 5 rule in plain fp64 for a group of any size n: sort |w| descending, running
 * sums S_k, objective S_k^2/k at the ends of runs of equal magnitudes, first maximum.
 * Outputs the threshold (smallest kept magnitude), the kept count and alpha = S/k.
 */
int oracle_ternarize_group_f64(const double* w, int64_t n, double* tau_out, int64_t* k_out,
                               double* alpha_out) {
  double* a;
  int64_t i, best_k = 0;
  double S = 0.0, best_J = -1.0, best_S = 0.0;
  if (n < 1) return ORACLE_ERR_ARG;
  a = (double*)malloc(sizeof(double) * (size_t)n);
  if (!a) return ORACLE_ERR_ARG;
  for (i = 0; i < n; i++) {
    if (!isfinite(w[i])) {
      free(a);
      return ORACLE_ERR_NONFINITE;
    }
    a[i] = fabs(w[i]);
  }
  qsort(a, (size_t)n, sizeof(double), cmp_desc);
  for (i = 0; i < n; i++) {
    if (a[i] == 0.0) break;
    S += a[i];
    if (i + 1 == n || a[i + 1] < a[i]) {
      double J = S * S / (double)(i + 1);
      if (J > best_J) {
        best_J = J;
        best_k = i + 1;
        best_S = S;
      }
    }
  }
  *k_out = best_k;
  *tau_out = best_k ? a[best_k - 1] : 0.0;
  *alpha_out = best_k ? best_S / (double)best_k : 0.0;
  free(a);
  return ORACLE_OK;
}

/*
 * Eq. 2: the M x Kred weight matrix (row m = one output filter, Kred in (r, s, c) order)
 * is split into independent groups of G consecutive elements along Kred; each row is
 * zero-padded to Kp = ceil(Kred/G)*G.  Outputs t [M][Kp] in {-1,0,1} and alpha
 * [M][Kp/G].  Returns the first error seen (groups with an error get t = 0, alpha = 0).
 */
int oracle_ternarize(const float* w, int M, int Kred, int G, int8_t* t, float* alpha) {
  int m, g, j;
  int ng, Kp, status = ORACLE_OK;
  float buf[ORACLE_MAX_G];
  if (M < 0 || Kred < 0 || G < 1 || G > ORACLE_MAX_G) return ORACLE_ERR_ARG;
  ng = (Kred + G - 1) / G;
  Kp = ng * G;
  for (m = 0; m < M; m++) {
    for (g = 0; g < ng; g++) {
      int st;
      for (j = 0; j < G; j++) {
        int k = g * G + j;
        buf[j] = k < Kred ? w[(size_t)m * Kred + k] : 0.0f;
      }
      st = oracle_ternarize_group(buf, G, t + (size_t)m * Kp + (size_t)g * G,
                                  alpha + (size_t)m * ng + g);
      if (st != ORACLE_OK && status == ORACLE_OK) status = st;
    }
  }
  return status;
}

/*
 * 2-bit code words.  Code of t: 0 -> 00, +1 -> 01, -1 -> 11.  Element j of a row goes to
 * word j/16 of that row, bits [2(j%16), 2(j%16)+1]; each row has ceil(Kp/16) words and
 * unused bits are 0.
 */
void oracle_pack_codes(const int8_t* t, int M, int Kp, uint32_t* codes) {
  int m, j;
  int wrow = (Kp + 15) / 16;
  memset(codes, 0, sizeof(uint32_t) * (size_t)M * (size_t)wrow);
  for (m = 0; m < M; m++) {
    for (j = 0; j < Kp; j++) {
      int8_t v = t[(size_t)m * Kp + j];
      uint32_t c = v == 0 ? 0u : (v > 0 ? 1u : 3u);
      codes[(size_t)m * wrow + j / 16] |= c << (2 * (j % 16));
    }
  }
}

static int qmax_of(int type) {
  switch (type) {
    case ORACLE_U8: return 255;
    case ORACLE_S8: return 127;
    case ORACLE_U4: return 15;
    case ORACLE_S4: return 7;
  }
  return -1;
}

static int qmin_of(int type) {
  switch (type) {
    case ORACLE_U8: return 0;
    case ORACLE_S8: return -128;
    case ORACLE_U4: return 0;
    case ORACLE_S4: return -8;
  }
  return 1;
}

static int is_unsigned(int type) { return type == ORACLE_U8 || type == ORACLE_U4; }

/*
 * Dynamic fixed point shared exponent (Section 4): the smallest integer E with
 * m * 2^-E <= qmax, m = max |x| (max(x, 0) for the unsigned types); E = 0 when m = 0;
 * E is clamped to [-149, 127].
 */
int oracle_dfp_exponent(const float* x, size_t n, int type, int* E_out) {
  size_t i;
  double m = 0.0;
  int E, qmax = qmax_of(type);
  if (qmax < 0) return ORACLE_ERR_ARG;
  for (i = 0; i < n; i++) {
    double v = (double)x[i];
    if (!isfinite(v)) return ORACLE_ERR_NONFINITE;
    if (is_unsigned(type)) v = v > 0.0 ? v : 0.0;
    else v = fabs(v);
    if (v > m) m = v;
  }
  if (m == 0.0) {
    *E_out = 0;
    return ORACLE_OK;
  }
  E = -400;
  while (ldexp(m, -E) > (double)qmax) E++;
  if (E < -149) E = -149;
  if (E > 127) E = 127;
  *E_out = E;
  return ORACLE_OK;
}

/*
 * DFP quantisation: q_i = clamp(round_half_even(x_i * 2^-E), qmin, qmax), scale = 2^E.
 * If scale_in > 0 it is used as the scale and must be a power of two; otherwise E comes
 * from oracle_dfp_exponent.  q holds one int32 code per element (unpacked).
 */
int oracle_quantize(const float* x, size_t n, int type, float scale_in, int32_t* q,
                    float* scale_out, int* E_out) {
  size_t i;
  int E = 0, st;
  int qmax = qmax_of(type), qmin = qmin_of(type);
  if (qmax < 0) return ORACLE_ERR_ARG;
  if (scale_in > 0.0f) {
    int ex;
    double fr = frexp((double)scale_in, &ex);
    if (!isfinite(scale_in) || fr != 0.5) return ORACLE_ERR_ARG;
    E = ex - 1;
    for (i = 0; i < n; i++)
      if (!isfinite(x[i])) return ORACLE_ERR_NONFINITE;
  } else {
    st = oracle_dfp_exponent(x, n, type, &E);
    if (st != ORACLE_OK) return st;
  }
  for (i = 0; i < n; i++) {
    double v = nearbyint(ldexp((double)x[i], -E)); /* default rounding: half to even */
    if (v > qmax) v = qmax;
    if (v < qmin) v = qmin;
    q[i] = (int32_t)v;
  }
  *scale_out = (float)ldexp(1.0, E);
  if (E_out) *E_out = E;
  return ORACLE_OK;
}

/* Bytes for 8-bit types; for 4-bit types element 2i -> low nibble of byte i, 2i+1 -> high
 * nibble (two's complement for the signed type). */
void oracle_pack_act(const int32_t* q, size_t n, int type, uint8_t* out) {
  size_t i;
  if (type == ORACLE_U8 || type == ORACLE_S8) {
    for (i = 0; i < n; i++) out[i] = (uint8_t)(q[i] & 0xff);
    return;
  }
  memset(out, 0, (n + 1) / 2);
  for (i = 0; i < n; i++) out[i / 2] |= (uint8_t)((q[i] & 0xf) << (4 * (i % 2)));
}

/* One im2col column: the Kred = R*S*Cg codes seen by output position (b, ho, wo) of conv
 * group gi, in (r, s, c) order, zero outside the image; zero-padded to Kp. */
static void im2col_column(const int32_t* q, int H, int W, int C, int R, int S, int stride,
                          int pad, int Cg, int gi, int b, int ho, int wo, int Kp,
                          int64_t* col) {
  int r, s, c, j = 0;
  for (r = 0; r < R; r++) {
    for (s = 0; s < S; s++) {
      int hi = ho * stride - pad + r;
      int wi = wo * stride - pad + s;
      int inside = hi >= 0 && hi < H && wi >= 0 && wi < W;
      for (c = 0; c < Cg; c++) {
        col[j++] = inside ? q[(((size_t)b * H + hi) * W + wi) * C + (size_t)gi * Cg + c] : 0;
      }
    }
  }
  while (j < Kp) col[j++] = 0;
}

static int conv_geometry(int H, int W, int C, int R, int S, int stride, int pad, int groups,
                         int M, int G, int* Ho, int* Wo, int* Cg, int* Kred, int* Kp,
                         int* ng) {
  if (H <= 0 || W <= 0 || C <= 0 || R <= 0 || S <= 0 || stride <= 0 || pad < 0 ||
      groups <= 0 || M <= 0 || G <= 0 || C % groups || M % groups)
    return ORACLE_ERR_ARG;
  *Ho = (H + 2 * pad - R) / stride + 1;
  *Wo = (W + 2 * pad - S) / stride + 1;
  if (*Ho <= 0 || *Wo <= 0) return ORACLE_ERR_ARG;
  *Cg = C / groups;
  *Kred = R * S * (*Cg);
  *ng = (*Kred + G - 1) / G;
  *Kp = (*ng) * G;
  return ORACLE_OK;
}

/* y[m] = s_x * sum_g alpha[m][g] * s[m][g] over one column, with s[m][g] =
 * sum_{j in g} t[m][j] * col[j] in int64 (Eq. 2 applied to the convolution; the int32
 * accumulator of Section 4 holds these sums exactly).  ymag = s_x * sum_g |alpha*s|. */
static void contract_column(const int64_t* col, const int8_t* t, const float* alpha, int m0,
                            int m1, int Kp, int G, int ng, double act_scale, double* y,
                            double* ymag) {
  int m, g, j;
  for (m = m0; m < m1; m++) {
    double acc = 0.0, mag = 0.0;
    for (g = 0; g < ng; g++) {
      int64_t s = 0;
      for (j = g * G; j < (g + 1) * G; j++) s += (int64_t)t[(size_t)m * Kp + j] * col[j];
      acc += (double)alpha[(size_t)m * ng + g] * (double)s;
      mag += fabs((double)alpha[(size_t)m * ng + g] * (double)s);
    }
    y[m] = act_scale * acc;
    if (ymag) ymag[m] = act_scale * mag;
  }
}

/*
 * Grouped-ternary convolution over NHWC codes q [B][H][W][C] with weights t [M][Kp],
 * alpha [M][ng] as from oracle_ternarize (Kred = R*S*C/groups); output y and ymag
 * [B][Ho][Wo][M] (fp64).  groups is the convolution's channel grouping (AlexNet towers).
 */
int oracle_conv2d(const int32_t* q, double act_scale, int B, int H, int W, int C, int R,
                  int S, int stride, int pad, int groups, const int8_t* t,
                  const float* alpha, int M, int G, double* y, double* ymag) {
  int Ho, Wo, Cg, Kred, Kp, ng, b, ho, wo, gi;
  int64_t* col;
  int st = conv_geometry(H, W, C, R, S, stride, pad, groups, M, G, &Ho, &Wo, &Cg, &Kred,
                         &Kp, &ng);
  if (st != ORACLE_OK || B <= 0) return ORACLE_ERR_ARG;
  col = (int64_t*)malloc(sizeof(int64_t) * (size_t)Kp);
  if (!col) return ORACLE_ERR_ARG;
  for (b = 0; b < B; b++)
    for (ho = 0; ho < Ho; ho++)
      for (wo = 0; wo < Wo; wo++) {
        size_t p = ((size_t)b * Ho + ho) * Wo + wo;
        int Mg = M / groups;
        for (gi = 0; gi < groups; gi++) {
          im2col_column(q, H, W, C, R, S, stride, pad, Cg, gi, b, ho, wo, Kp, col);
          contract_column(col, t, alpha, gi * Mg, (gi + 1) * Mg, Kp, G, ng, act_scale,
                          y + p * M, ymag ? ymag + p * M : NULL);
        }
      }
  free(col);
  return ORACLE_OK;
}

/* The same contraction at npos listed flat output positions p = (b*Ho + ho)*Wo + wo;
 * outputs y and ymag [npos][M]. */
int oracle_conv2d_at(const int32_t* q, double act_scale, int B, int H, int W, int C, int R,
                     int S, int stride, int pad, int groups, const int8_t* t,
                     const float* alpha, int M, int G, const int64_t* pos, int64_t npos,
                     double* y, double* ymag) {
  int Ho, Wo, Cg, Kred, Kp, ng, gi;
  int64_t i;
  int64_t* col;
  int st = conv_geometry(H, W, C, R, S, stride, pad, groups, M, G, &Ho, &Wo, &Cg, &Kred,
                         &Kp, &ng);
  if (st != ORACLE_OK || B <= 0) return ORACLE_ERR_ARG;
  col = (int64_t*)malloc(sizeof(int64_t) * (size_t)Kp);
  if (!col) return ORACLE_ERR_ARG;
  for (i = 0; i < npos; i++) {
    int64_t p = pos[i];
    int wo = (int)(p % Wo), ho = (int)((p / Wo) % Ho), b = (int)(p / ((int64_t)Wo * Ho));
    int Mg = M / groups;
    if (p < 0 || b >= B) {
      free(col);
      return ORACLE_ERR_ARG;
    }
    for (gi = 0; gi < groups; gi++) {
      im2col_column(q, H, W, C, R, S, stride, pad, Cg, gi, b, ho, wo, Kp, col);
      contract_column(col, t, alpha, gi * Mg, (gi + 1) * Mg, Kp, G, ng, act_scale,
                      y + (size_t)i * M, ymag ? ymag + (size_t)i * M : NULL);
    }
  }
  free(col);
  return ORACLE_OK;
}

/* Fully connected form: activations q [P][Kred] (unpacked codes), y and ymag [P][M]. */
int oracle_gemm(const int32_t* q, double act_scale, int P, int Kred, const int8_t* t,
                const float* alpha, int M, int G, double* y, double* ymag) {
  int p, j, ng, Kp;
  int64_t* col;
  if (P < 0 || Kred <= 0 || M <= 0 || G <= 0) return ORACLE_ERR_ARG;
  ng = (Kred + G - 1) / G;
  Kp = ng * G;
  col = (int64_t*)malloc(sizeof(int64_t) * (size_t)Kp);
  if (!col) return ORACLE_ERR_ARG;
  for (p = 0; p < P; p++) {
    for (j = 0; j < Kp; j++) col[j] = j < Kred ? q[(size_t)p * Kred + j] : 0;
    contract_column(col, t, alpha, 0, M, Kp, G, ng, act_scale, y + (size_t)p * M,
                    ymag ? ymag + (size_t)p * M : NULL);
  }
  free(col);
  return ORACLE_OK;
}

/* Group sums s[m][g][p] = sum_{j in g} t[m][j] * q[p][j] for q [P][Kred]; int64 out. */
int oracle_group_sums(const int32_t* q, int P, int Kred, const int8_t* t, int M, int G,
                      int64_t* s) {
  int p, m, g, j, ng, Kp;
  if (P < 0 || Kred <= 0 || M <= 0 || G <= 0) return ORACLE_ERR_ARG;
  ng = (Kred + G - 1) / G;
  Kp = ng * G;
  for (m = 0; m < M; m++)
    for (g = 0; g < ng; g++)
      for (p = 0; p < P; p++) {
        int64_t acc = 0;
        for (j = g * G; j < (g + 1) * G && j < Kred; j++)
          acc += (int64_t)t[(size_t)m * Kp + j] * q[(size_t)p * Kred + j];
        s[((size_t)m * ng + g) * P + p] = acc;
      }
  return ORACLE_OK;
}

/*
 * Group sums of a convolution (the 32-bit accumulators of Section 4 inside Eq. 2) at npos
 * listed flat output positions p = (b*Ho + ho)*Wo + wo: for filter m of conv group gi and
 * group g of its reduction vector, s[m][g][i] = sum_{j in g} t[m][j] * col[j] with col the
 * im2col column of position pos[i] for conv group gi.  q NHWC codes [B][H][W][C]; t
 * [M][Kp]; s int64 [M][ng][npos].
 */
int oracle_conv2d_group_sums(const int32_t* q, int B, int H, int W, int C, int R, int S,
                             int stride, int pad, int groups, const int8_t* t, int M, int G,
                             const int64_t* pos, int64_t npos, int64_t* s) {
  int Ho, Wo, Cg, Kred, Kp, ng, gi, m, g, j;
  int64_t i;
  int64_t* col;
  int st = conv_geometry(H, W, C, R, S, stride, pad, groups, M, G, &Ho, &Wo, &Cg, &Kred,
                         &Kp, &ng);
  if (st != ORACLE_OK || B <= 0 || npos < 0) return ORACLE_ERR_ARG;
  col = (int64_t*)malloc(sizeof(int64_t) * (size_t)Kp);
  if (!col) return ORACLE_ERR_ARG;
  for (i = 0; i < npos; i++) {
    int64_t p = pos[i];
    int wo = (int)(p % Wo), ho = (int)((p / Wo) % Ho), b = (int)(p / ((int64_t)Wo * Ho));
    int Mg = M / groups;
    if (p < 0 || b >= B) {
      free(col);
      return ORACLE_ERR_ARG;
    }
    for (gi = 0; gi < groups; gi++) {
      im2col_column(q, H, W, C, R, S, stride, pad, Cg, gi, b, ho, wo, Kp, col);
      for (m = gi * Mg; m < (gi + 1) * Mg; m++)
        for (g = 0; g < ng; g++) {
          int64_t acc = 0;
          for (j = g * G; j < (g + 1) * G; j++) acc += (int64_t)t[(size_t)m * Kp + j] * col[j];
          s[((size_t)m * ng + g) * (size_t)npos + (size_t)i] = acc;
        }
    }
  }
  free(col);
  return ORACLE_OK;
}

/*
 * Dense 8-bit-weight convolution (the first layer is kept at 8w-8a, Section 4):
 * wq int8 [M][Kred] with per-filter scale wscale[m]; y = s_x * wscale[m] * sum wq*col,
 * the dot product exact in int64.  Outputs y, ymag [B][Ho][Wo][M].
 */
int oracle_conv2d_w8(const int32_t* q, double act_scale, int B, int H, int W, int C, int R,
                     int S, int stride, int pad, int groups, const int8_t* wq,
                     const float* wscale, int M, double* y, double* ymag) {
  int Ho, Wo, Cg, Kred, Kp, ng, b, ho, wo, gi, m, j;
  int64_t* col;
  int st = conv_geometry(H, W, C, R, S, stride, pad, groups, M, 1, &Ho, &Wo, &Cg, &Kred,
                         &Kp, &ng);
  if (st != ORACLE_OK || B <= 0) return ORACLE_ERR_ARG;
  col = (int64_t*)malloc(sizeof(int64_t) * (size_t)Kp);
  if (!col) return ORACLE_ERR_ARG;
  for (b = 0; b < B; b++)
    for (ho = 0; ho < Ho; ho++)
      for (wo = 0; wo < Wo; wo++) {
        size_t p = ((size_t)b * Ho + ho) * Wo + wo;
        int Mg = M / groups;
        for (gi = 0; gi < groups; gi++) {
          im2col_column(q, H, W, C, R, S, stride, pad, Cg, gi, b, ho, wo, Kp, col);
          for (m = gi * Mg; m < (gi + 1) * Mg; m++) {
            int64_t acc = 0;
            double v;
            for (j = 0; j < Kred; j++) acc += (int64_t)wq[(size_t)m * Kred + j] * col[j];
            v = act_scale * (double)wscale[m] * (double)acc;
            y[p * M + m] = v;
            if (ymag) ymag[p * M + m] = fabs(v);
          }
        }
      }
  free(col);
  return ORACLE_OK;
}

/*
 * Threshold ternarization with an analytical threshold (Section 3: t_i = sign(w_i) if
 * |w_i| > Delta, else 0; Lemma 1 and its Gaussian counterpart).  One threshold per group
 * of G (per_layer = 0) or one for the whole M x Kred layer (per_layer = 1):
 *   rule 0, exponential magnitudes (Lemma 1): Delta = mean |w|;
 *   rule 1, Gaussian weights: Delta = ORACLE_Z_GAUSS * rms(w), rms(w) the maximum-
 *     likelihood sigma of N(0, sigma) that the paper names, and ORACLE_Z_GAUSS the z that
 *     maximises phi(z)^2 / (1 - Phi(z)): for w ~ N(0, sigma^2) and many elements, the
 *     threshold objective (sum_{|w| > Delta} |w|)^2 / |I_Delta| is proportional to that
 *     function of z = Delta / sigma (the Gaussian counterpart of the Lemma 1 derivation).
 * alpha = mean of the kept |w| (for a fixed support, the alpha of Eq. 4; 0 if none is
 * kept): per group when per_layer = 0, one value for the layer (written to every
 * alpha[m][g]) when per_layer = 1 -- the one-scaling-factor-per-layer baseline.  The
 * statistics cover the real weights only (a row's zero padding is not counted).  All sums
 * are fp64 in element order (row-major over the layer when per_layer = 1); the threshold
 * is kept in fp64 and compared with |w| (fp32 promoted exactly); alpha = (float)(S / k).
 * delta_out (may be NULL) receives the per-group thresholds [M][ng] (or one per layer).
 * Non-finite weights: ORACLE_ERR_NONFINITE, and the affected groups (or the layer) get
 * t = 0, alpha = 0.
 */
#define ORACLE_Z_GAUSS 0.6120031809624808

static double threshold_of(double sum_abs, double sum_sq, int64_t n, int rule) {
  if (n == 0) return 0.0;
  if (rule == 0) return sum_abs / (double)n;
  return ORACLE_Z_GAUSS * sqrt(sum_sq / (double)n);
}

int oracle_ternarize_threshold(const float* w, int M, int Kred, int G, int rule, int per_layer,
                               int8_t* t, float* alpha, double* delta_out) {
  int m, g, j;
  int ng, Kp;
  if (M < 0 || Kred < 0 || G < 1 || (rule != 0 && rule != 1)) return ORACLE_ERR_ARG;
  ng = (Kred + G - 1) / G;
  Kp = ng * G;
  memset(t, 0, (size_t)M * Kp);
  if (per_layer) {
    double sa = 0.0, sq = 0.0, kept = 0.0, delta;
    int64_t n = (int64_t)M * Kred, k = 0;
    size_t i;
    float a;
    for (i = 0; i < (size_t)n; i++) {
      if (!isfinite(w[i])) {
        for (i = 0; i < (size_t)M * ng; i++) alpha[i] = 0.0f;
        if (delta_out) delta_out[0] = 0.0;
        return ORACLE_ERR_NONFINITE;
      }
      sa += fabs((double)w[i]);
      sq += (double)w[i] * (double)w[i];
    }
    delta = threshold_of(sa, sq, n, rule);
    for (m = 0; m < M; m++)
      for (j = 0; j < Kred; j++) {
        const double v = (double)w[(size_t)m * Kred + j];
        if (fabs(v) > delta) {
          t[(size_t)m * Kp + j] = v > 0 ? 1 : -1;
          kept += fabs(v);
          k++;
        }
      }
    a = k ? (float)(kept / (double)k) : 0.0f;
    for (i = 0; i < (size_t)M * ng; i++) alpha[i] = a;
    if (delta_out) delta_out[0] = delta;
    return ORACLE_OK;
  }
  {
    int status = ORACLE_OK;
    for (m = 0; m < M; m++) {
      for (g = 0; g < ng; g++) {
        const int j0 = g * G, j1 = j0 + G < Kred ? j0 + G : Kred;
        double sa = 0.0, sq = 0.0, kept = 0.0, delta;
        int64_t k = 0;
        int bad = 0;
        for (j = j0; j < j1; j++) {
          const float v = w[(size_t)m * Kred + j];
          if (!isfinite(v)) bad = 1;
          sa += fabs((double)v);
          sq += (double)v * (double)v;
        }
        if (bad) {
          alpha[(size_t)m * ng + g] = 0.0f;
          if (delta_out) delta_out[(size_t)m * ng + g] = 0.0;
          status = ORACLE_ERR_NONFINITE;
          continue;
        }
        delta = threshold_of(sa, sq, j1 - j0, rule);
        for (j = j0; j < j1; j++) {
          const double v = (double)w[(size_t)m * Kred + j];
          if (fabs(v) > delta) {
            t[(size_t)m * Kp + j] = v > 0 ? 1 : -1;
            kept += fabs(v);
            k++;
          }
        }
        alpha[(size_t)m * ng + g] = k ? (float)(kept / (double)k) : 0.0f;
        if (delta_out) delta_out[(size_t)m * ng + g] = delta;
      }
    }
    return status;
  }
}

/*
 * Ternary error of each group, err[m][g] = sum_{j in g} (w_j - alpha[m][g] * t_j)^2 in
 * fp64, element order, over the real weights (Section 3: the element-wise error E).
 */
int oracle_ternary_error(const float* w, int M, int Kred, int G, const int8_t* t, const float* alpha,
                         double* err) {
  int m, g, j;
  int ng, Kp;
  if (M < 0 || Kred < 0 || G < 1) return ORACLE_ERR_ARG;
  ng = (Kred + G - 1) / G;
  Kp = ng * G;
  for (m = 0; m < M; m++)
    for (g = 0; g < ng; g++) {
      const int j0 = g * G, j1 = j0 + G < Kred ? j0 + G : Kred;
      const double a = (double)alpha[(size_t)m * ng + g];
      double e = 0.0;
      for (j = j0; j < j1; j++) {
        const double d = (double)w[(size_t)m * Kred + j] - a * (double)t[(size_t)m * Kp + j];
        e += d * d;
      }
      err[(size_t)m * ng + g] = e;
    }
  return ORACLE_OK;
}

/*
 * Fixed-point scaling factors (Section 4: the alphas of the groups are quantized to 8/4-bit
 * fixed point).  Reading (the paper does not say how the exponent is shared): the ng
 * alphas of one filter row share one DFP exponent, and the rule is oracle_quantize's with
 * the unsigned 8-bit (bits = 8) or 4-bit (bits = 4) type, since alpha >= 0:
 *   a[m][g] = clamp(round_half_even(alpha[m][g] * 2^-E_m), 0, 2^bits - 1), scale[m] = 2^E_m.
 * The contraction then uses alpha' = a * 2^E_m (exact in fp32).  a holds one int32 per
 * value (unpacked).
 */
int oracle_quantize_alpha(const float* alpha, int M, int ng, int bits, int32_t* a, float* scale) {
  int m, st = ORACLE_OK;
  if (M < 0 || ng < 0 || (bits != 8 && bits != 4)) return ORACLE_ERR_ARG;
  for (m = 0; m < M; m++) {
    int E;
    const int r = oracle_quantize(alpha + (size_t)m * ng, (size_t)ng, bits == 8 ? ORACLE_U8 : ORACLE_U4, 0.0f,
                                  a + (size_t)m * ng, scale + m, &E);
    if (r != ORACLE_OK) {
      memset(a + (size_t)m * ng, 0, sizeof(int32_t) * (size_t)ng);
      scale[m] = 0.0f;
      if (st == ORACLE_OK) st = r;
    }
  }
  return st;
}
