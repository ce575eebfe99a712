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
 *   - Sec. 3 "Post-Training Quantization", Eq. (quant): Q_b(X) = s * round(X / s) with
 *     s = max|X| / (2^(b-1) - 1), one scale per group of consecutive entries; b = 4 gives /7.
 *   - App. B.1 "Quantization settings and kernels": symmetric, round to nearest, one scale per
 *     group of consecutive input channels, weights offline, activations per token at run time,
 *     activation scale = group absmax / 7; weight codes stored as 4-bit values.
 *   - Sec. 4.2 "Splitting the layer", Eq. (xsplit) and Eq. (asp):
 *       x = V(V^T x) + x_perp,  x_perp = (I - VV^T) x,
 *       W^T x ~= (V^T W)^T (V^T x) + Q4(W_perp)^T Q4(x_perp),  W_perp = (I - VV^T) W.
 *   - Table 3: per-group W4A4 costs 4.50 bits per weight at group 32, i.e. a 16-bit weight scale.
 *   - Sec. 3 Eq. (pair) and App. B.1: smoothing and a block Hadamard rotation in front of the
 *     quantizer, x~ = H diag(s)^-1 x and W~ = H diag(s) W, H applied by the fast Walsh-Hadamard
 *     transform in blocks of B (qo_block_fwht); the layer then runs on x~ and W~ (the *_f64 entry
 *     points take float64 inputs).
 *
 * Row-major notation of this file: X [M,K] holds one token per row, W [K,N] maps K inputs to N
 * outputs (Y = X W is the paper's y = W^T x for every token), U [K,r] is the paper's V.
 *
 * Readings of points the paper leaves open (each is one line of the design notes):
 *   R1  format: INT4 codes in [-7, 7] (absmax/7 never produces -8), group G along K.
 *   R2  round to nearest = nearest integer to the EXACT quotient x/s, ties to even.
 *   R3  activation scale: bfloat16, s_x = RN_bf16(amax / 7) of the group's absmax, one rounding
 *       of the exact quotient (ties to even).
 *   R4  weight scale: bfloat16 (the 16-bit scale of Table 3), s_w = RN_bf16(amax / 7) of the
 *       float64 absmax, one rounding of the exact quotient.
 *   R5  codes are taken against the stored (rounded) scale; a zero scale gives zero codes; the
 *       code is the nearest one in [-7, 7] (it saturates), which differs from the nearest
 *       integer only for bfloat16-subnormal scales (below 2^-126), where rounding amax / 7 to
 *       few significant bits can leave amax / s above 7.5.
 *   R6  the "16-bit" branch is float16: p_hat = RN_f16(x U), B_hat = RN_f16(U^T W).
 *   R7  the branch uses float64 B_f = U^T W for the deflation, B_hat only for the output.
 *   R11 on float64 activations (the rotated x~) the scale follows R3 on the float64 absmax.
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

/* bfloat16 bits of RN_bf16(a / 7) for the exact quotient of a finite a >= 0, ties to even
 * (readings R3 and R4).  q = fl64(a / 7) lies within half a float64 unit of a / 7, so when q is
 * itself a bfloat16 value it is the answer; otherwise the two bfloat16 values around q are
 * n u and (n + 1) u, u the quantum of q's binade (8 significant bits; the subnormal binade of
 * bfloat16 below 2^-126 has u = 2^-133), and comparing a with 7 (n + 1/2) u -- a product of at
 * most 12 significant bits, exact in float64 -- decides between them. */
static uint16_t bf16_bits_div7_rn(double a) {
  if (!(a > 0.0)) return 0;
  const double q = a / 7.0;
  int e2;
  frexp(q, &e2);
  int E = e2 - 1; /* q in [2^E, 2^(E+1)) */
  if (E < -126) E = -126;
  const double u = ldexp(1.0, E - 7);
  const double n = floor(q / u); /* q / u is a power-of-two scaling: exact */
  double v;
  if (n * u == q) {
    v = q;
  } else {
    const double t = 7.0 * ((n + 0.5) * u);
    if (a > t)
      v = (n + 1.0) * u;
    else if (a < t)
      v = n * u;
    else
      v = (fmod(n, 2.0) == 0.0) ? n * u : (n + 1.0) * u;
  }
  if (v > 3.3895313892515355e38) return 0x7f80; /* above the largest bfloat16: infinity */
  /* v lies on the bfloat16 grid, hence on the float32 grid: the upper half of its float32 bits */
  const float f = (float)v;
  uint32_t b;
  memcpy(&b, &f, sizeof b);
  return (uint16_t)(b >> 16);
}

/* ---- the quantizer of Eq. (quant) ------------------------------------------------------ */

/* Nearest code in [-7, 7] to the exact quotient x/s, ties to even (readings R2, R5); s > 0.
 * c = nearbyint(fl(x/s)) is within one of the answer.  For the operand formats used here
 * (x in float32 or float64, s in bfloat16, float32 or float16, |x| <= ~7.5 s) both c*s and x - c*s are
 * exact in float64, so the remainder e decides the rounding exactly. */
static int nearest_code(double x, double s) {
  double c = nearbyint(x / s);
  double e = x - c * s;
  double t = 2.0 * fabs(e);
  if (t > s)
    c += (e > 0.0) ? 1.0 : -1.0;
  else if (t == s && fmod(c, 2.0) != 0.0)
    c += (e > 0.0) ? 1.0 : -1.0;
  if (c > 7.0) c = 7.0;
  if (c < -7.0) c = -7.0;
  return (int)c;
}

/* ---- offline packing: Eq. (asp), W_perp derivation, Eq. (quant) on weights ------------- */

/* W_bf16 [K,N] bf16 bits; U [K,r] float32 (orthonormal columns; ignored when r == 0).
 * Outputs: qw [N,K] int8 codes, sw [K/G,N] bfloat16 bits, Bh [r,N] float16 bits,
 *          Bf [r,N] float64 (optional), Wperp [K,N] float64 (optional). */
static int pack_core(const double* W, const float* U, int K, int N, int r, int G, int8_t* qw, uint16_t* sw,
                     uint16_t* Bh, double* Bf_out, double* Wperp_out) {
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
      for (int k = 0; k < K; ++k) acc += (double)U[(size_t)k * r + j] * W[(size_t)k * N + n];
      Bf[(size_t)j * N + n] = acc;
    }
  /* W_perp = (I - U U^T) W = W - U B_f. */
#pragma omp parallel for schedule(static)
  for (int k = 0; k < K; ++k)
    for (int n = 0; n < N; ++n) {
      double acc = 0.0;
      for (int j = 0; j < r; ++j) acc += (double)U[(size_t)k * r + j] * Bf[(size_t)j * N + n];
      Wp[(size_t)k * N + n] = W[(size_t)k * N + n] - acc;
    }
  /* Per output channel n and group g of G consecutive inputs: s_w = RN_bf16(amax/7), codes. */
  int ng = K / G;
#pragma omp parallel for schedule(static) reduction(min : status)
  for (int n = 0; n < N; ++n)
    for (int g = 0; g < ng; ++g) {
      double amax = 0.0;
      for (int k = g * G; k < (g + 1) * G; ++k) {
        double a = fabs(Wp[(size_t)k * N + n]);
        if (a > amax) amax = a;
      }
      uint16_t sbits = bf16_bits_div7_rn(amax);
      double s = bf16_value(sbits);
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

int qo_pack(const uint16_t* W_bf16, const float* U, int K, int N, int r, int G, int8_t* qw,
            uint16_t* sw, uint16_t* Bh, double* Bf_out, double* Wperp_out) {
  if (K <= 0 || N <= 0) return QO_EINVAL;
  double* W = (double*)malloc((size_t)K * N * sizeof(double));
  if (!W) return QO_EINVAL;
  for (size_t i = 0; i < (size_t)K * N; ++i) W[i] = bf16_value(W_bf16[i]);
  int st = pack_core(W, U, K, N, r, G, qw, sw, Bh, Bf_out, Wperp_out);
  free(W);
  return st;
}

/* The same packing of a float64 weight W [K,N] (the smoothed and rotated W~ of Eq. (pair)). */
int qo_pack_f64(const double* W, const float* U, int K, int N, int r, int G, int8_t* qw, uint16_t* sw,
                uint16_t* Bh, double* Bf_out, double* Wperp_out) {
  return pack_core(W, U, K, N, r, G, qw, sw, Bh, Bf_out, Wperp_out);
}

/* ---- run-time activation path: Eq. (xsplit), then Eq. (quant) per token and group ------- */

/* X_bf16 [M,K] bf16 bits; U [K,r] float32.
 * Outputs: qx [M,K] int8 codes, sx [M,K/G] scales (bfloat16 values, held in float32),
 *          ph [M,r] float16 bits,
 *          p [M,r] float64 (optional), Xperp [M,K] float64 (optional). */
static int quantize_act_core(const uint16_t* X_bf16, const double* X_f64, const float* U, int M, int K, int r,
                             int G, int8_t* qx, float* sx, uint16_t* ph, double* p_out, double* Xperp_out) {
  if (M < 0 || K <= 0 || r < 0 || r > K || G <= 0 || K % G) return QO_EINVAL;
  int status = QO_OK;
  int ng = K / G;
#pragma omp parallel reduction(min : status)
  {
    double* x = (double*)malloc((size_t)K * sizeof(double));
    double* p = (double*)malloc((size_t)(r > 0 ? r : 1) * sizeof(double));
#pragma omp for schedule(static)
    for (int m = 0; m < M; ++m) {
      for (int k = 0; k < K; ++k) x[k] = X_bf16 ? bf16_value(X_bf16[(size_t)m * K + k]) : X_f64[(size_t)m * K + k];
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
        float s = (float)bf16_value(bf16_bits_div7_rn(amax));
        if (isinf(s)) status = QO_ERANGE;
        sx[(size_t)m * ng + g] = s;
        for (int k = g * G; k < (g + 1) * G; ++k) {
          int c = (s > 0.0f && !isinf(s)) ? nearest_code(x[k], (double)s) : 0;
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

int qo_quantize_act(const uint16_t* X_bf16, const float* U, int M, int K, int r, int G, int8_t* qx,
                    float* sx, uint16_t* ph, double* p_out, double* Xperp_out) {
  return quantize_act_core(X_bf16, NULL, U, M, K, r, G, qx, sx, ph, p_out, Xperp_out);
}

/* The same activation path on float64 activations X [M,K] (the smoothed and rotated x~). */
int qo_quantize_act_f64(const double* X, const float* U, int M, int K, int r, int G, int8_t* qx, float* sx,
                        uint16_t* ph, double* p_out, double* Xperp_out) {
  if (!X && M > 0) return QO_EINVAL;
  return quantize_act_core(NULL, X, U, M, K, r, G, qx, sx, ph, p_out, Xperp_out);
}

/* The rotation H of Eq. (pair) applied with the fast Walsh-Hadamard transform, the method the paper
 * names for it (App. B.1: blocks of B, the largest power of two dividing n, at most 1024).  For
 * each of `count` vectors of length n (element i of vector v at data[v * vstride + i * estride]):
 * y_i = x_i * scale[i] (or x_i / scale[i] when divide != 0; no scaling when scale is NULL), then
 * butterflies (a + b, a - b) at spans 1, 2, 4, ..., B/2 inside each block, then each entry times
 * 1/sqrt(B).  Every product and sum is one float64 rounding, in this order, in place. */
int qo_block_fwht(double* data, int count, int n, long vstride, long estride, const double* scale, int divide) {
  if (count < 0 || n <= 0) return QO_EINVAL;
  int B = 1;
  while (n % (2 * B) == 0 && 2 * B <= 1024) B *= 2;
  const double nrm = 1.0 / sqrt((double)B);
#pragma omp parallel for schedule(static)
  for (int v = 0; v < count; ++v) {
    double* x = data + (long)v * vstride;
    if (scale)
      for (int i = 0; i < n; ++i) {
        const long a = (long)i * estride;
        x[a] = divide ? x[a] / scale[i] : x[a] * scale[i];
      }
    for (int h = 1; h < B; h *= 2)
      for (int b0 = 0; b0 < n; b0 += B)
        for (int u0 = 0; u0 < B; u0 += 2 * h)
          for (int q = 0; q < h; ++q) {
            const long a = (long)(b0 + u0 + q) * estride, c = (long)(b0 + u0 + q + h) * estride;
            const double xa = x[a], xc = x[c];
            x[a] = xa + xc;
            x[c] = xa - xc;
          }
    for (int i = 0; i < n; ++i) x[(long)i * estride] *= nrm;
  }
  return QO_OK;
}

/* The quantizer alone, applied to a given float32 remainder R [M,K] (reading R3 on the float32
 * absmax).  Outputs q [M,K] int8 and s [M,K/G] (bfloat16 values, held in float32). */
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
      float s = (float)bf16_value(bf16_bits_div7_rn((double)amax));
      if (isinf(s)) status = QO_ERANGE;
      s_out[(size_t)m * ng + g] = s;
      for (int k = g * G; k < (g + 1) * G; ++k) {
        int c = (s > 0.0f && !isinf(s)) ? nearest_code((double)R[(size_t)m * K + k], (double)s) : 0;
        if (c < -7 || c > 7) status = QO_ERANGE;
        q[(size_t)m * K + k] = (int8_t)c;
      }
    }
  return status;
}

/* ---- the layer output, Eq. (asp) -------------------------------------------------------- */

/* Y[m,n] = sum_g s_x[m,g] s_w[g,n] P_g[m,n]  +  sum_j p_hat[m,j] B_hat[j,n],
 * P_g[m,n] = sum_{k in group g} qx[m,k] qw[n,k]  (exact int64).
 * Each group term s_x * s_w * P_g has at most 8 + 8 + 13 significant bits, so it is exact in
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
  for (size_t i = 0; i < (size_t)ng * N; ++i) swv[i] = bf16_value(sw[i]);
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
uint16_t qo_bf16_bits_div7_rn(double a) { return bf16_bits_div7_rn(a); }

/* ==== NVFP4 variant (App. B.1: on Blackwell GPUs the paper stores E2M1 values with an E4M3
 * scale per group of 16 elements, for weights and activations, and one extra float32 scale per
 * weight tensor).  The paper gives the storage format only; the readings below fix the rest.
 *   N1  E2M1 (OCP FP4): sign | 2-bit exponent (bias 1) | 1-bit mantissa.  Magnitudes of codes
 *       0..7: 0, 0.5, 1, 1.5, 2, 3, 4, 6.  Rounding to E2M1 is to nearest, ties to an even
 *       mantissa bit, and saturates at 6.
 *   N2  E4M3 (OCP FP8, "FN"): sign | 4-bit exponent (bias 7) | 3-bit mantissa; no infinities;
 *       largest finite 448; subnormals m * 2^-9.  Rounding is to nearest, ties to even, and
 *       saturates at 448.
 *   N3  activations, per token and block b of 16 consecutive K entries of x_perp:
 *       s = RN_e4m3(RN_f32(amax_b / 6)),  code = RN_e2m1(x / s) of the exact quotient,
 *       s == 0 -> codes 0.  The remainder x_perp stays in float64 (Eq. (xsplit) in exact
 *       arithmetic, as for the INT4 activations); amax_b / 6 is rounded to float64 and then
 *       to float32.  For a float32 x, RN_e2m1(RN_f32(x / s)) = RN_e2m1(x / s): a float32 step
 *       next to a midpoint product moves x / s by more than half a float32 unit of it, so the
 *       float32 quotient lands on an E2M1 midpoint only when x / s is that midpoint.
 *   N4  weights: s_g = RN_f32(amax(W_perp) / (6 * 448)); per output channel n and block b,
 *       s_b = RN_e4m3(amax_b / (6 s_g)) and code = RN_e2m1(w / (s_b s_g)), both from the
 *       float64 quotient (whose one rounding cannot change a 4-bit or 2-bit result:
 *       53 >= 2 * 4 + 2); s_g == 0 or s_b == 0 -> codes 0.
 *   N5  output: y = s_g * sum_b s_a s_b sum_{k in b} e2m1(qa) e2m1(qb)  +  sum_j p_hat_j B_hat_j.
 * Block length is 16; K must be a multiple of 16. */

#define QO_FP4_BLOCK 16

/* E2M1 code (4 bits) -> value. */
static double e2m1_value(int c) {
  static const double mag[8] = {0.0, 0.5, 1.0, 1.5, 2.0, 3.0, 4.0, 6.0};
  double v = mag[c & 7];
  return (c & 8) ? -v : v;
}

/* E4M3 bits -> value (reading N2).  0x7f / 0xff are NaN. */
static double e4m3_value(uint8_t b) {
  int s = b >> 7, e = (b >> 3) & 15, m = b & 7;
  double v;
  if (e == 15 && m == 7)
    v = NAN;
  else if (e == 0)
    v = ldexp((double)m, -9);
  else
    v = ldexp((double)(8 + m), e - 10);
  return s ? -v : v;
}

/* value -> E4M3 bits, nearest, ties to even, saturating at 448 (reading N2).  As in f16_bits_rn:
 * scale by a power of two so that one quantum of the binade is 1, then nearbyint(). */
static uint8_t e4m3_bits_rn(double x) {
  uint8_t sign = signbit(x) ? 0x80 : 0;
  double a = fabs(x);
  if (isnan(x)) return 0x7f;
  if (a == 0.0) return sign;
  if (a >= 448.0) return sign | 0x7e; /* saturate */
  int e2;
  frexp(a, &e2);
  int E = e2 - 1;        /* a in [2^E, 2^(E+1)) */
  if (E < -6) E = -6;    /* subnormal binade: quantum 2^-9 */
  double q = nearbyint(ldexp(a, 3 - E)); /* quanta of 2^(E-3): 0 .. 16 */
  if (q >= 16.0) {
    q = 8.0;
    E += 1;
  }
  if (E == -6 && q < 8.0) return sign | (uint8_t)q; /* subnormal (or zero) */
  if (E > 8) return sign | 0x7e;                   /* 2^9 and beyond: above 448 */
  int code = ((E + 7) << 3) | ((int)q - 8);
  if (code > 0x7e) code = 0x7e;                    /* 464 .. 480 round to 448 by saturation */
  return sign | (uint8_t)code;
}

/* RN_e2m1(x / s) of the exact quotient (s > 0), readings N1 and N3: |x| is compared with the
 * midpoints 0.25, 0.75, ..., 5 of the magnitude grid times s (products of at most 3 and 4
 * significant bits, exact in float64); on a midpoint the code with the even mantissa bit wins,
 * and beyond 5 s the code saturates at 6. */
static int e2m1_code_ratio(double x, double s) {
  static const double mid[7] = {0.25, 0.75, 1.25, 1.75, 2.5, 3.5, 5.0};
  const double a = fabs(x);
  int c = 7;
  for (int i = 0; i < 7; ++i) {
    const double ms = mid[i] * s;
    if (a < ms) {
      c = i;
      break;
    }
    if (a == ms) {
      c = (i & 1) ? i + 1 : i; /* codes i and i + 1 differ in the mantissa bit: keep the even */
      break;
    }
  }
  if (c == 0) return 0; /* +0 for any sign */
  return (x < 0.0) ? (c | 8) : c;
}

/* value -> E2M1 code, nearest, ties to even mantissa, saturating at 6 (reading N1).
 * Exhaustive over the eight magnitudes: the nearest one wins; on a tie the one whose code is
 * even (mantissa bit 0). */
static int e2m1_code_rn(double x) {
  double a = fabs(x);
  int best = 0;
  double bestd = INFINITY;
  if (a >= 6.0) {
    best = 7;
  } else {
    for (int c = 0; c < 8; ++c) {
      double d = fabs(a - e2m1_value(c));
      if (d < bestd || (d == bestd && (c & 1) == 0)) {
        best = c;
        bestd = d;
      }
    }
  }
  if (best == 0) return 0; /* +0 for any sign */
  return (x < 0.0) ? (best | 8) : best;
}

/* Offline packing of the NVFP4 variant: W_perp as in qo_pack, then reading N4.
 * Outputs: qw [N,K] E2M1 codes (one per byte), sfw [N,K/16] E4M3 bits, *sg, Bh [r,N]. */
static int pack_nvfp4_core(const double* W, const float* U, int K, int N, int r, uint8_t* qw, uint8_t* sfw,
                           float* sg_out, uint16_t* Bh) {
  if (K <= 0 || N <= 0 || r < 0 || r > K || K % QO_FP4_BLOCK) return QO_EINVAL;
  int status = QO_OK;
  double* Bf = (double*)calloc((size_t)(r > 0 ? r : 1) * N, sizeof(double));
  double* Wp = (double*)malloc((size_t)K * N * sizeof(double));
  if (!Bf || !Wp) {
    free(Bf);
    free(Wp);
    return QO_EINVAL;
  }
#pragma omp parallel for schedule(static)
  for (int n = 0; n < N; ++n)
    for (int j = 0; j < r; ++j) {
      double acc = 0.0;
      for (int k = 0; k < K; ++k) acc += (double)U[(size_t)k * r + j] * W[(size_t)k * N + n];
      Bf[(size_t)j * N + n] = acc;
    }
#pragma omp parallel for schedule(static)
  for (int k = 0; k < K; ++k)
    for (int n = 0; n < N; ++n) {
      double acc = 0.0;
      for (int j = 0; j < r; ++j) acc += (double)U[(size_t)k * r + j] * Bf[(size_t)j * N + n];
      Wp[(size_t)k * N + n] = W[(size_t)k * N + n] - acc;
    }
  double amax = 0.0;
  for (size_t i = 0; i < (size_t)K * N; ++i)
    if (fabs(Wp[i]) > amax) amax = fabs(Wp[i]);
  const float sg = (float)(amax / (6.0 * 448.0));
  *sg_out = sg;
  const int nb = K / QO_FP4_BLOCK;
#pragma omp parallel for schedule(static)
  for (int n = 0; n < N; ++n)
    for (int b = 0; b < nb; ++b) {
      double ab = 0.0;
      for (int k = b * QO_FP4_BLOCK; k < (b + 1) * QO_FP4_BLOCK; ++k)
        if (fabs(Wp[(size_t)k * N + n]) > ab) ab = fabs(Wp[(size_t)k * N + n]);
      uint8_t sb = (sg > 0.0f) ? e4m3_bits_rn(ab / (6.0 * (double)sg)) : 0;
      sfw[(size_t)n * nb + b] = sb;
      double scale = e4m3_value(sb) * (double)sg; /* exact: 4 x 24 significant bits */
      for (int k = b * QO_FP4_BLOCK; k < (b + 1) * QO_FP4_BLOCK; ++k)
        qw[(size_t)n * K + k] = (uint8_t)((scale > 0.0) ? e2m1_code_rn(Wp[(size_t)k * N + n] / scale) : 0);
    }
  for (size_t i = 0; i < (size_t)r * N; ++i) {
    Bh[i] = f16_bits_rn(Bf[i]);
    if ((Bh[i] & 0x7c00) == 0x7c00) status = QO_ERANGE;
  }
  free(Bf);
  free(Wp);
  return status;
}

int qo_pack_nvfp4(const uint16_t* W_bf16, const float* U, int K, int N, int r, uint8_t* qw, uint8_t* sfw,
                  float* sg_out, uint16_t* Bh) {
  if (K <= 0 || N <= 0) return QO_EINVAL;
  double* W = (double*)malloc((size_t)K * N * sizeof(double));
  if (!W) return QO_EINVAL;
  for (size_t i = 0; i < (size_t)K * N; ++i) W[i] = bf16_value(W_bf16[i]);
  const int st = pack_nvfp4_core(W, U, K, N, r, qw, sfw, sg_out, Bh);
  free(W);
  return st;
}

/* The NVFP4 pack of a float64 weight (the smoothed and rotated W~). */
int qo_pack_nvfp4_f64(const double* W, const float* U, int K, int N, int r, uint8_t* qw, uint8_t* sfw,
                      float* sg_out, uint16_t* Bh) {
  if (!W) return QO_EINVAL;
  return pack_nvfp4_core(W, U, K, N, r, qw, sfw, sg_out, Bh);
}

/* Reading N3 on one remainder row segment of 16 entries. */
static void quantize_block_nvfp4(const double* x, uint8_t* q, uint8_t* sf) {
  double amax = 0.0;
  for (int k = 0; k < QO_FP4_BLOCK; ++k)
    if (fabs(x[k]) > amax) amax = fabs(x[k]);
  /* RN_f32(amax / 6): for a float32 amax the double rounding through float64 is innocuous */
  const float t = (float)(amax / 6.0);
  const uint8_t sb = e4m3_bits_rn((double)t);
  *sf = sb;
  const double s = e4m3_value(sb);
  for (int k = 0; k < QO_FP4_BLOCK; ++k) q[k] = (uint8_t)((s > 0.0) ? e2m1_code_ratio(x[k], s) : 0);
}

/* Run-time activation path of the NVFP4 variant: Eq. (xsplit) as in qo_quantize_act (the
 * remainder in float64), then reading N3.
 * Outputs: qx [M,K] E2M1 codes, sfx [M,K/16] E4M3 bits, ph [M,r] float16 bits. */
static int quantize_act_nvfp4_core(const uint16_t* X_bf16, const double* X_f64, const float* U, int M, int K, int r,
                                   uint8_t* qx, uint8_t* sfx, uint16_t* ph) {
  if (M < 0 || K <= 0 || r < 0 || r > K || K % QO_FP4_BLOCK) return QO_EINVAL;
  int status = QO_OK;
  const int nb = K / QO_FP4_BLOCK;
#pragma omp parallel reduction(min : status)
  {
    double* x = (double*)malloc((size_t)K * sizeof(double));
    double* xp = (double*)malloc((size_t)K * sizeof(double));
    double* p = (double*)malloc((size_t)(r > 0 ? r : 1) * sizeof(double));
#pragma omp for schedule(static)
    for (int m = 0; m < M; ++m) {
      for (int k = 0; k < K; ++k) x[k] = X_bf16 ? bf16_value(X_bf16[(size_t)m * K + k]) : X_f64[(size_t)m * K + k];
      for (int j = 0; j < r; ++j) {
        double acc = 0.0;
        for (int k = 0; k < K; ++k) acc += x[k] * (double)U[(size_t)k * r + j];
        p[j] = acc;
      }
      for (int k = 0; k < K; ++k) {
        double acc = 0.0;
        for (int j = 0; j < r; ++j) acc += p[j] * (double)U[(size_t)k * r + j];
        xp[k] = x[k] - acc;
      }
      for (int j = 0; j < r; ++j) {
        ph[(size_t)m * r + j] = f16_bits_rn(p[j]);
        if ((ph[(size_t)m * r + j] & 0x7c00) == 0x7c00) status = QO_ERANGE;
      }
      for (int b = 0; b < nb; ++b)
        quantize_block_nvfp4(xp + b * QO_FP4_BLOCK, qx + (size_t)m * K + b * QO_FP4_BLOCK, sfx + (size_t)m * nb + b);
    }
    free(x);
    free(xp);
    free(p);
  }
  return status;
}

int qo_quantize_act_nvfp4(const uint16_t* X_bf16, const float* U, int M, int K, int r, uint8_t* qx,
                          uint8_t* sfx, uint16_t* ph) {
  return quantize_act_nvfp4_core(X_bf16, NULL, U, M, K, r, qx, sfx, ph);
}

/* The NVFP4 activation path on float64 activations (the smoothed and rotated x~). */
int qo_quantize_act_nvfp4_f64(const double* X, const float* U, int M, int K, int r, uint8_t* qx, uint8_t* sfx,
                              uint16_t* ph) {
  if (!X && M > 0) return QO_EINVAL;
  return quantize_act_nvfp4_core(NULL, X, U, M, K, r, qx, sfx, ph);
}

/* Reading N3 alone on a given float32 remainder R [M,K] -> qx [M,K], sfx [M,K/16]. */
int qo_quantize_residual_nvfp4_f32(const float* R, int M, int K, uint8_t* qx, uint8_t* sfx) {
  if (M < 0 || K <= 0 || K % QO_FP4_BLOCK) return QO_EINVAL;
  const int nb = K / QO_FP4_BLOCK;
#pragma omp parallel for schedule(static)
  for (int m = 0; m < M; ++m)
    for (int b = 0; b < nb; ++b) {
      double x[QO_FP4_BLOCK]; /* float32 values, widened exactly */
      for (int k = 0; k < QO_FP4_BLOCK; ++k) x[k] = (double)R[(size_t)m * K + b * QO_FP4_BLOCK + k];
      quantize_block_nvfp4(x, qx + (size_t)m * K + b * QO_FP4_BLOCK, sfx + (size_t)m * nb + b);
    }
  return QO_OK;
}

/* Reading N5: the layer output of the NVFP4 variant in float64. */
int qo_linear_nvfp4(const uint8_t* qx, const uint8_t* sfx, const uint16_t* ph, const uint8_t* qw,
                    const uint8_t* sfw, float sg, const uint16_t* Bh, int M, int K, int N, int r, double* Y) {
  if (M < 0 || K <= 0 || N <= 0 || r < 0 || K % QO_FP4_BLOCK) return QO_EINVAL;
  const int nb = K / QO_FP4_BLOCK;
  double* bhv = (double*)malloc((size_t)(r > 0 ? r : 1) * N * sizeof(double));
  if (!bhv) return QO_EINVAL;
  for (size_t i = 0; i < (size_t)r * N; ++i) bhv[i] = f16_value(Bh[i]);
#pragma omp parallel for schedule(dynamic, 4)
  for (int m = 0; m < M; ++m)
    for (int n = 0; n < N; ++n) {
      double y = 0.0;
      for (int b = 0; b < nb; ++b) {
        double P = 0.0; /* sum of 16 products of E2M1 values: exact (quarter-integers below 600) */
        for (int k = b * QO_FP4_BLOCK; k < (b + 1) * QO_FP4_BLOCK; ++k)
          P += e2m1_value(qx[(size_t)m * K + k]) * e2m1_value(qw[(size_t)n * K + k]);
        y += e4m3_value(sfx[(size_t)m * nb + b]) * e4m3_value(sfw[(size_t)n * nb + b]) * P;
      }
      double br = 0.0;
      for (int j = 0; j < r; ++j) br += f16_value(ph[(size_t)m * r + j]) * bhv[(size_t)j * N + n];
      Y[(size_t)m * N + n] = (double)sg * y + br;
    }
  free(bhv);
  return QO_OK;
}

/* NVFP4 number formats exposed for the pins. */
double qo_e2m1_value(int c) { return e2m1_value(c); }
int qo_e2m1_code_rn(double x) { return e2m1_code_rn(x); }
double qo_e4m3_value(uint8_t b) { return e4m3_value(b); }
uint8_t qo_e4m3_bits_rn(double x) { return e4m3_bits_rn(x); }
