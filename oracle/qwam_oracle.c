/*
 * qwam_oracle.c -- CPU oracle for the Action-Subspace Protection (ASP) linear layer.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the slow, plainly written reference that the CUDA
 * path is checked against.  Only the tests, the smoke check and the CPU-baseline leg of the
 * benchmark may load it; the library itself never does.  It shares no code, header, table or
 * helper with the CUDA path.
 *
 * Arithmetic: float64 for real numbers, int64 for integer partial sums.  Compiled with
 * -ffp-contract=off so that every operation below rounds exactly as written, on x86-64 and on
 * aarch64 alike.
 *
 * What it follows (paper: "Q-WAM", arxiv 2609.33269):
 *   - Sec. 2 "Post-Training Quantization", Eq. (quant): Q_b(X) = s * round(X / s) with
 *     s = max|X| / (2^(b-1) - 1), one scale per group of consecutive entries; b = 4 gives /7.
 *   - App. B.1 "Quantization settings and kernels": symmetric, round to nearest, one scale per
 *     group of consecutive input channels, weights offline, activations per token at run time,
 *     activation scale = group absmax / 7; weight codes stored as 4-bit values.
 *   - Sec. 3.2 "Splitting the layer", Eq. (xsplit) and Eq. (asp):
 *       x = V(V^T x) + x_perp,  x_perp = (I - VV^T) x,
 *       W^T x ~= (V^T W)^T (V^T x) + Q4(W_perp)^T Q4(x_perp),  W_perp = (I - VV^T) W.
 *   - Table 3: per-group W4A4 costs 4.50 bits per weight at group 32, i.e. a 16-bit weight scale.
 *
 * Row-major notation of this file: X [M,K] holds one token per row, W [K,N] maps K inputs to N
 * outputs (Y = X W is the paper's y = W^T x for every token), U [K,r] is the paper's V.
 *
 * Readings of points the paper leaves open (each is one line of the design notes):
 *   R1  format: INT4 codes in [-7, 7] (absmax/7 never produces -8), group G along K.
 *   R2  round to nearest = nearest integer to the EXACT quotient x/s, ties to even.
 *   R3  activation scale: float32, s_x = RN_f32(amax / 7) of the group's absmax.
 *   R4  weight scale: float16, s_w = RN_f16(amax / 7) computed from the float64 absmax.
 *   R5  codes are taken against the stored (rounded) scale; a zero scale gives zero codes.
 *   R6  the "16-bit" branch is float16: p_hat = RN_f16(x U), B_hat = RN_f16(U^T W).
 *   R7  the branch uses float64 B_f = U^T W for the deflation, B_hat only for the output.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define QO_OK 0
#define QO_EINVAL (-1)
#define QO_ERANGE (-2)

/* ---- number formats ------------------------------------------------------------------ */

/* bfloat16 bits -> value: the upper half of an IEEE binary32. */
static double bf16_value(uint16_t b) {
  uint32_t u = (uint32_t)b << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return (double)f;
}

/* binary16 bits -> value, from the IEEE 754 encoding (bias 15, 10 fraction bits). */
static double f16_value(uint16_t h) {
  int s = h >> 15, e = (h >> 10) & 31, m = h & 1023;
  double v;
  if (e == 0)
    v = ldexp((double)m, -24);
  else if (e == 31)
    v = m ? NAN : INFINITY;
  else
    v = ldexp((double)(m + 1024), e - 25);
  return s ? -v : v;
}

/* value -> binary16 bits, round to nearest, ties to even (IEEE 754 roundTiesToEven).
 * The value is scaled by a power of two (exact) so that one quantum of its binade becomes 1,
 * and nearbyint() (default rounding mode: ties to even) rounds it. */
static uint16_t f16_bits_rn(double x) {
  uint16_t sign = signbit(x) ? 0x8000 : 0;
  double a = fabs(x);
  if (isnan(x)) return 0x7e00;
  if (a == 0.0) return sign;
  if (a >= 65520.0) return sign | 0x7c00; /* halfway to 2^16 and beyond round to infinity */
  int e2;
  frexp(a, &e2);
  int E = e2 - 1; /* a in [2^E, 2^(E+1)) */
  if (E < -14) E = -14; /* subnormal binade: quantum 2^-24 */
  double q = nearbyint(ldexp(a, 10 - E)); /* number of quanta, 0 .. 2048 */
  if (q >= 2048.0) {
    q = 1024.0;
    E += 1;
  }
  if (E == -14 && q < 1024.0) return sign | (uint16_t)q; /* subnormal */
  return sign | (uint16_t)(((E + 15) << 10) | ((int)q - 1024));
}

/* ---- the quantizer of Eq. (quant) ------------------------------------------------------ */

/* Nearest integer to the exact quotient x/s, ties to even (reading R2); s > 0.
 * c = nearbyint(fl(x/s)) is within one of the answer.  For the operand formats used here
 * (x in float32 or float64, s in float32 or float16, |x| <= ~7.5 s) both c*s and x - c*s are
 * exact in float64, so the remainder e decides the rounding exactly. */
static int nearest_code(double x, double s) {
  double c = nearbyint(x / s);
  double e = x - c * s;
  double t = 2.0 * fabs(e);
  if (t > s)
    c += (e > 0.0) ? 1.0 : -1.0;
  else if (t == s && fmod(c, 2.0) != 0.0)
    c += (e > 0.0) ? 1.0 : -1.0;
  return (int)c;
}

/* ---- offline packing: Eq. (asp), W_perp derivation, Eq. (quant) on weights ------------- */

/* W_bf16 [K,N] bf16 bits; U [K,r] float32 (orthonormal columns; ignored when r == 0).
 * Outputs: qw [N,K] int8 codes, sw [K/G,N] float16 bits, Bh [r,N] float16 bits,
 *          Bf [r,N] float64 (optional), Wperp [K,N] float64 (optional). */
int qo_pack(const uint16_t* W_bf16, const float* U, int K, int N, int r, int G, int8_t* qw,
            uint16_t* sw, uint16_t* Bh, double* Bf_out, double* Wperp_out) {
  if (K <= 0 || N <= 0 || r < 0 || r > K || G <= 0 || K % G) return QO_EINVAL;
  int status = QO_OK;
  double* Bf = (double*)calloc((size_t)(r > 0 ? r : 1) * N, sizeof(double));
  double* Wp = (double*)malloc((size_t)K * N * sizeof(double));
  if (!Bf || !Wp) {
    free(Bf);
    free(Wp);
    return QO_EINVAL;
  }
  /* B_f = U^T W  (r x N): the weight of the 16-bit branch, V^T W in the paper. */
#pragma omp parallel for schedule(static)
  for (int n = 0; n < N; ++n)
    for (int j = 0; j < r; ++j) {
      double acc = 0.0;
      for (int k = 0; k < K; ++k) acc += (double)U[(size_t)k * r + j] * bf16_value(W_bf16[(size_t)k * N + n]);
      Bf[(size_t)j * N + n] = acc;
    }
  /* W_perp = (I - U U^T) W = W - U B_f. */
#pragma omp parallel for schedule(static)
  for (int k = 0; k < K; ++k)
    for (int n = 0; n < N; ++n) {
      double acc = 0.0;
      for (int j = 0; j < r; ++j) acc += (double)U[(size_t)k * r + j] * Bf[(size_t)j * N + n];
      Wp[(size_t)k * N + n] = bf16_value(W_bf16[(size_t)k * N + n]) - acc;
    }
  /* Per output channel n and group g of G consecutive inputs: s_w = RN_f16(amax/7), codes. */
  int ng = K / G;
#pragma omp parallel for schedule(static) reduction(min : status)
  for (int n = 0; n < N; ++n)
    for (int g = 0; g < ng; ++g) {
      double amax = 0.0;
      for (int k = g * G; k < (g + 1) * G; ++k) {
        double a = fabs(Wp[(size_t)k * N + n]);
        if (a > amax) amax = a;
      }
      uint16_t sbits = f16_bits_rn(amax / 7.0);
      double s = f16_value(sbits);
      if (isinf(s)) status = QO_ERANGE;
      sw[(size_t)g * N + n] = sbits;
      for (int k = g * G; k < (g + 1) * G; ++k) {
        int c = (s > 0.0 && !isinf(s)) ? nearest_code(Wp[(size_t)k * N + n], s) : 0;
        if (c < -7 || c > 7) status = QO_ERANGE;
        qw[(size_t)n * K + k] = (int8_t)c;
      }
    }
  for (size_t i = 0; i < (size_t)r * N; ++i) {
    Bh[i] = f16_bits_rn(Bf[i]);
    if ((Bh[i] & 0x7c00) == 0x7c00) status = QO_ERANGE;
  }
  if (Bf_out && r > 0) memcpy(Bf_out, Bf, (size_t)r * N * sizeof(double));
  if (Wperp_out) memcpy(Wperp_out, Wp, (size_t)K * N * sizeof(double));
  free(Bf);
  free(Wp);
  return status;
}

/* ---- run-time activation path: Eq. (xsplit), then Eq. (quant) per token and group ------- */

/* X_bf16 [M,K] bf16 bits; U [K,r] float32.
 * Outputs: qx [M,K] int8 codes, sx [M,K/G] float32 scales, ph [M,r] float16 bits,
 *          p [M,r] float64 (optional), Xperp [M,K] float64 (optional). */
int qo_quantize_act(const uint16_t* X_bf16, const float* U, int M, int K, int r, int G, int8_t* qx,
                    float* sx, uint16_t* ph, double* p_out, double* Xperp_out) {
  if (M < 0 || K <= 0 || r < 0 || r > K || G <= 0 || K % G) return QO_EINVAL;
  int status = QO_OK;
  int ng = K / G;
#pragma omp parallel reduction(min : status)
  {
    double* x = (double*)malloc((size_t)K * sizeof(double));
    double* p = (double*)malloc((size_t)(r > 0 ? r : 1) * sizeof(double));
#pragma omp for schedule(static)
    for (int m = 0; m < M; ++m) {
      for (int k = 0; k < K; ++k) x[k] = bf16_value(X_bf16[(size_t)m * K + k]);
      /* protected coordinates p = x U (r values), the V^T x of Eq. (xsplit) */
      for (int j = 0; j < r; ++j) {
        double acc = 0.0;
        for (int k = 0; k < K; ++k) acc += x[k] * (double)U[(size_t)k * r + j];
        p[j] = acc;
      }
      /* remainder x_perp = x - p U^T, in place */
      for (int k = 0; k < K; ++k) {
        double acc = 0.0;
        for (int j = 0; j < r; ++j) acc += p[j] * (double)U[(size_t)k * r + j];
        x[k] -= acc;
      }
      if (Xperp_out) memcpy(Xperp_out + (size_t)m * K, x, (size_t)K * sizeof(double));
      for (int j = 0; j < r; ++j) {
        ph[(size_t)m * r + j] = f16_bits_rn(p[j]);
        if ((ph[(size_t)m * r + j] & 0x7c00) == 0x7c00) status = QO_ERANGE;
        if (p_out) p_out[(size_t)m * r + j] = p[j];
      }
      for (int g = 0; g < ng; ++g) {
        double amax = 0.0;
        for (int k = g * G; k < (g + 1) * G; ++k)
          if (fabs(x[k]) > amax) amax = fabs(x[k]);
        float s = (float)(amax / 7.0);
        sx[(size_t)m * ng + g] = s;
        for (int k = g * G; k < (g + 1) * G; ++k) {
          int c = (s > 0.0f) ? nearest_code(x[k], (double)s) : 0;
          if (c < -7 || c > 7) status = QO_ERANGE;
          qx[(size_t)m * K + k] = (int8_t)c;
        }
      }
    }
    free(x);
    free(p);
  }
  return status;
}

/* The quantizer alone, applied to a given float32 remainder R [M,K] (reading R3 with an exact
 * float32 input: RN_f32(amax/7) through float64 is exact rounding of the true quotient because
 * 53 >= 2*24 + 2).  Outputs q [M,K] int8 and s [M,K/G] float32. */
int qo_quantize_residual_f32(const float* R, int M, int K, int G, int8_t* q, float* s_out) {
  if (M < 0 || K <= 0 || G <= 0 || K % G) return QO_EINVAL;
  int status = QO_OK;
  int ng = K / G;
#pragma omp parallel for schedule(static) reduction(min : status)
  for (int m = 0; m < M; ++m)
    for (int g = 0; g < ng; ++g) {
      float amax = 0.0f;
      for (int k = g * G; k < (g + 1) * G; ++k) {
        float a = fabsf(R[(size_t)m * K + k]);
        if (a > amax) amax = a;
      }
      float s = (float)((double)amax / 7.0);
      s_out[(size_t)m * ng + g] = s;
      for (int k = g * G; k < (g + 1) * G; ++k) {
        int c = (s > 0.0f) ? nearest_code((double)R[(size_t)m * K + k], (double)s) : 0;
        if (c < -7 || c > 7) status = QO_ERANGE;
        q[(size_t)m * K + k] = (int8_t)c;
      }
    }
  return status;
}

/* ---- the layer output, Eq. (asp) -------------------------------------------------------- */

/* Y[m,n] = sum_g s_x[m,g] s_w[g,n] P_g[m,n]  +  sum_j p_hat[m,j] B_hat[j,n],
 * P_g[m,n] = sum_{k in group g} qx[m,k] qw[n,k]  (exact int64).
 * Each group term s_x * s_w * P_g has at most 24 + 11 + 13 significant bits, so it is exact in
 * float64; only the sum over groups and branch terms rounds. */
int qo_linear(const int8_t* qx, const float* sx, const uint16_t* ph, const int8_t* qw,
              const uint16_t* sw, const uint16_t* Bh, int M, int K, int N, int r, int G, double* Y) {
  if (M < 0 || K <= 0 || N <= 0 || r < 0 || G <= 0 || K % G) return QO_EINVAL;
  int ng = K / G;
  double* swv = (double*)malloc((size_t)ng * N * sizeof(double));
  double* bhv = (double*)malloc((size_t)(r > 0 ? r : 1) * N * sizeof(double));
  if (!swv || !bhv) {
    free(swv);
    free(bhv);
    return QO_EINVAL;
  }
  for (size_t i = 0; i < (size_t)ng * N; ++i) swv[i] = f16_value(sw[i]);
  for (size_t i = 0; i < (size_t)r * N; ++i) bhv[i] = f16_value(Bh[i]);
#pragma omp parallel for schedule(dynamic, 4)
  for (int m = 0; m < M; ++m)
    for (int n = 0; n < N; ++n) {
      double y = 0.0;
      for (int g = 0; g < ng; ++g) {
        int64_t P = 0;
        for (int k = g * G; k < (g + 1) * G; ++k)
          P += (int64_t)qx[(size_t)m * K + k] * (int64_t)qw[(size_t)n * K + k];
        y += (double)sx[(size_t)m * ng + g] * swv[(size_t)g * N + n] * (double)P;
      }
      double b = 0.0;
      for (int j = 0; j < r; ++j) b += f16_value(ph[(size_t)m * r + j]) * bhv[(size_t)j * N + n];
      Y[(size_t)m * N + n] = y + b;
    }
  free(swv);
  free(bhv);
  return QO_OK;
}

/* Eq. (asp) before quantization (Q replaced by the identity):
 * Y = p B_f + X_perp W_perp, all float64.  Equals X W up to float64 rounding. */
int qo_linear_split_exact(const double* p, const double* Xperp, const double* Bf, const double* Wperp,
                          int M, int K, int N, int r, double* Y) {
  if (M < 0 || K <= 0 || N <= 0 || r < 0) return QO_EINVAL;
#pragma omp parallel for schedule(static)
  for (int m = 0; m < M; ++m)
    for (int n = 0; n < N; ++n) {
      double a = 0.0, b = 0.0;
      for (int j = 0; j < r; ++j) a += p[(size_t)m * r + j] * Bf[(size_t)j * N + n];
      for (int k = 0; k < K; ++k) b += Xperp[(size_t)m * K + k] * Wperp[(size_t)k * N + n];
      Y[(size_t)m * N + n] = a + b;
    }
  return QO_OK;
}

/* Number formats exposed for the pins (tests compare them with library conversions). */
uint16_t qo_f16_bits_rn(double x) { return f16_bits_rn(x); }
double qo_f16_value(uint16_t h) { return f16_value(h); }
int qo_nearest_code(double x, double s) { return nearest_code(x, s); }
