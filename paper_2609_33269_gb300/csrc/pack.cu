// pack.cu -- offline packing of one ASP layer (Sec. 4.2 Eq. (asp) and the derivation of the
// deflated weight W_perp = (I - U U^T) W; Eq. (quant) of Sec. 3 applied to W_perp per output
// channel and group, App. B.1; or, for the NVFP4 variant of App. B.1, E2M1 codes with an E4M3
// scale per 16 K and one float32 scale per tensor).  float64 on the device, untimed.
//
// Every float64 operation is an explicit IEEE intrinsic (__dmul_rn, __dadd_rn, ...) so that no
// multiply-add is contracted: sums run in index order, each product and sum rounded once.
#include <cmath>
#include <cuda_fp4.h>
#include <cuda_fp8.h>

#include "internal.h"
#include "ptx.cuh"

namespace qwam {
namespace {

// The weight entering the pack: bf16 W, or the float64 smoothed and rotated W~ (exact either way).
__device__ __forceinline__ double wval(const __nv_bfloat16* W, size_t i) {
  return static_cast<double>(__bfloat162float(W[i]));
}
__device__ __forceinline__ double wval(const double* W, size_t i) { return W[i]; }

// B_f[j, n] = sum_k U[k, j] W[k, n]  (k ascending), float64.
template <typename WT>
__global__ void branch_weight_kernel(const WT* __restrict__ W, const float* __restrict__ U, int K, int N,
                                     int r, double* __restrict__ Bf) {
  int n = blockIdx.x * blockDim.x + threadIdx.x;
  int j = blockIdx.y;
  if (n >= N) return;
  double acc = 0.0;
  for (int k = 0; k < K; ++k) {
    double u = static_cast<double>(U[static_cast<size_t>(k) * r + j]);
    double w = wval(W, static_cast<size_t>(k) * N + n);
    acc = __dadd_rn(acc, __dmul_rn(u, w));
  }
  Bf[static_cast<size_t>(j) * N + n] = acc;
}

// W_perp[k, n] = W[k, n] - sum_j U[k, j] B_f[j, n]  (j ascending).
template <typename WT>
__device__ __forceinline__ double wperp(const WT* __restrict__ W, const float* __restrict__ U,
                                        const double* __restrict__ Bf, int N, int r, int k, int n) {
  double acc = 0.0;
  for (int j = 0; j < r; ++j)
    acc = __dadd_rn(acc, __dmul_rn(static_cast<double>(U[static_cast<size_t>(k) * r + j]),
                                   Bf[static_cast<size_t>(j) * N + n]));
  return __dsub_rn(wval(W, static_cast<size_t>(k) * N + n), acc);
}

// Nearest code in [-7, 7] to the exact quotient w / s, ties to even (saturating, which only a
// bfloat16-subnormal scale can need).  s is a bfloat16 value and w a float64 with |w| <= ~9 s,
// so c * s and w - c * s are exact in float64 and the remainder decides the rounding.
__device__ __forceinline__ int nearest_code_f64(double w, double s) {
  double c = rint(__ddiv_rn(w, s));
  double e = __dsub_rn(w, __dmul_rn(c, s));
  double t = 2.0 * fabs(e);
  bool odd = (static_cast<long long>(c) & 1LL) != 0;
  if (t > s || (t == s && odd)) c = __dadd_rn(c, e > 0.0 ? 1.0 : -1.0);
  return min(7, max(-7, static_cast<int>(c)));
}

// s_w = RN_bf16(a / 7) of the exact quotient (a >= 0, float64), ties to even.  The float64
// quotient q is within half a float64 unit of a / 7; if q is on the bfloat16 grid it is the
// answer, else the grid points n u < q < (n + 1) u (u = 2^(E - 7) for q in [2^E, 2^(E+1)), and
// 2^-133 below 2^-126) are decided by comparing a with 7 (n + 1/2) u, exact in float64.  Returns
// the bfloat16; infinity above the largest finite bfloat16.
__device__ __forceinline__ __nv_bfloat16 bf16_div7_f64(double a) {
  if (!(a > 0.0)) return __float2bfloat16_rn(0.0f);
  const double q = __ddiv_rn(a, 7.0);
  int E = ilogb(q);
  if (E < -126) E = -126;
  const double u = ldexp(1.0, E - 7);
  const double n = floor(__dmul_rn(q, ldexp(1.0, 7 - E)));
  double v = __dmul_rn(n, u);
  if (v != q) {
    const double t = __dmul_rn(7.0, __dmul_rn(__dadd_rn(n, 0.5), u));
    const bool up = a > t || (a == t && fmod(n, 2.0) != 0.0);
    if (up) v = __dmul_rn(__dadd_rn(n, 1.0), u);
  }
  if (v > 3.3895313892515355e38) return __ushort_as_bfloat16(static_cast<unsigned short>(0x7f80));
  return __float2bfloat16_rn(static_cast<float>(v));  // exact: v lies on the bfloat16 grid
}

// One thread per (output channel n, group g): s_w = RN_bf16(absmax / 7), codes packed 4 bits
// each into qw[n, :] as OB4 words (ob4_word: word j holds k = 8j..8j+7 as offset-binary nibbles,
// the form the GEMM turns into float16 pairs).
template <typename WT>
__global__ void quantize_weight_kernel(const WT* __restrict__ W, const float* __restrict__ U,
                                       const double* __restrict__ Bf, int K, int N, int r, int G, int N_pad,
                                       uint8_t* __restrict__ qw, __nv_bfloat16* __restrict__ sw, int* err) {
  int n = blockIdx.x * blockDim.x + threadIdx.x;
  int g = blockIdx.y;
  if (n >= N) return;
  double amax = 0.0;
  for (int k = g * G; k < (g + 1) * G; ++k) amax = fmax(amax, fabs(wperp(W, U, Bf, N, r, k, n)));
  const __nv_bfloat16 sb = bf16_div7_f64(amax);
  const double s = static_cast<double>(__bfloat162float(sb));
  sw[static_cast<size_t>(g) * N_pad + n] = sb;
  bool ok_scale = isfinite(s);
  if (!ok_scale) atomicOr(err, kErrRange);
  uint32_t* row = reinterpret_cast<uint32_t*>(qw + static_cast<size_t>(n) * (K / 2));
  for (int k = g * G; k < (g + 1) * G; k += 8) {
    int c[8];
    for (int i = 0; i < 8; ++i) {
      c[i] = 0;
      if (s > 0.0 && ok_scale) c[i] = nearest_code_f64(wperp(W, U, Bf, N, r, k + i, n), s);
    }
    row[k / 8] = ob4_word(c);
  }
}

// The INT4 GEMM's per-column copies (one thread per column n < N_pad): with
// b_n = max(7 max_g s_w[g, n], max_j |B_hat[n, j]|), e_n = 10 - floor(log2 b_n) clamped to
// [-126, 126] (0 for an all-zero column), s_w 2^e_n and B_hat 2^e_n rounded to float16 (exact
// while they stay above 2^-21 and 2^-24 of the column's largest value, which lies in
// [2^10, 2^11)) and the float32 factor 2^-e_n that the epilogue applies.
__global__ void column_shift_kernel(const __nv_bfloat16* __restrict__ sw, const __half* __restrict__ Bh, int ng,
                                    int N_pad, int r_pad, __half* __restrict__ swh, __half* __restrict__ Bhs,
                                    float* __restrict__ fcol) {
  const int n = blockIdx.x * blockDim.x + threadIdx.x;
  if (n >= N_pad) return;
  double b = 0.0;
  for (int g = 0; g < ng; ++g)
    b = fmax(b, __dmul_rn(7.0, static_cast<double>(__bfloat162float(sw[static_cast<size_t>(g) * N_pad + n]))));
  for (int j = 0; j < r_pad; ++j)
    b = fmax(b, fabs(static_cast<double>(__half2float(Bh[static_cast<size_t>(n) * r_pad + j]))));
  int e = 0;
  if (b > 0.0) e = min(126, max(-126, 10 - ilogb(b)));
  fcol[n] = static_cast<float>(ldexp(1.0, -e));
  const double f = ldexp(1.0, e);
  for (int g = 0; g < ng; ++g) {
    const size_t i = static_cast<size_t>(g) * N_pad + n;
    swh[i] = __double2half(__dmul_rn(static_cast<double>(__bfloat162float(sw[i])), f));
  }
  for (int j = 0; j < r_pad; ++j) {
    const size_t i = static_cast<size_t>(n) * r_pad + j;
    Bhs[i] = __double2half(__dmul_rn(static_cast<double>(__half2float(Bh[i])), f));
  }
}

// B_hat[n, j] = RN_f16(B_f[j, n]), K-major for the branch MMA, zero beyond r.
__global__ void branch_half_kernel(const double* __restrict__ Bf, int N, int r, int r_pad, __half* __restrict__ Bh,
                                   int* err) {
  int n = blockIdx.x * blockDim.x + threadIdx.x;
  if (n >= N) return;
  for (int j = 0; j < r_pad; ++j) {
    __half v = __float2half(0.0f);
    if (j < r) {
      v = __double2half(Bf[static_cast<size_t>(j) * N + n]);
      if (!isfinite(__half2float(v))) atomicOr(err, kErrRange);
    }
    Bh[static_cast<size_t>(n) * r_pad + j] = v;
  }
}

// bf16 hi/lo split of U: hi = RN_bf16(u), lo = RN_bf16(u - hi).  Written twice: transposed
// [2 r_pad, K] for the projection X U, and [K, ku3] as (hi, lo, hi) for the reconstruction.
// Up is the basis of the projection and Ur that of the reconstruction: both U, or, for a rotated
// layer, diag(s)^-1 H U and diag(s) H U.
__global__ void split_basis_kernel(const float* __restrict__ Up, const float* __restrict__ Ur, int K, int r, int r_pad,
                                   int ku3, __nv_bfloat16* __restrict__ ucat_t, __nv_bfloat16* __restrict__ ucat3) {
  int k = blockIdx.x * blockDim.x + threadIdx.x;
  if (k >= K) return;
  for (int j = 0; j < r_pad; ++j) {
    const float up = (j < r) ? Up[static_cast<size_t>(k) * r + j] : 0.0f;
    const float ur = (j < r) ? Ur[static_cast<size_t>(k) * r + j] : 0.0f;
    const __nv_bfloat16 phi = __float2bfloat16_rn(up);
    const __nv_bfloat16 plo = __float2bfloat16_rn(up - __bfloat162float(phi));
    const __nv_bfloat16 rhi = __float2bfloat16_rn(ur);
    const __nv_bfloat16 rlo = __float2bfloat16_rn(ur - __bfloat162float(rhi));
    ucat_t[static_cast<size_t>(j) * K + k] = phi;
    ucat_t[static_cast<size_t>(r_pad + j) * K + k] = plo;
    __nv_bfloat16* row = ucat3 + static_cast<size_t>(k) * ku3;
    row[j] = rhi;
    row[r_pad + j] = rlo;
    row[2 * r_pad + j] = rhi;
  }
  for (int j = 3 * r_pad; j < ku3; ++j) ucat3[static_cast<size_t>(k) * ku3 + j] = __float2bfloat16_rn(0.0f);
}

// The same two bases in float32, transposed to [r_pad, K] (zero rows beyond r), for the small-M
// activation kernel: its lanes then read consecutive channels of one column.
__global__ void basis32_kernel(const float* __restrict__ Up, const float* __restrict__ Ur, int K, int r, int r_pad,
                               float* __restrict__ up32, float* __restrict__ ur32) {
  int k = blockIdx.x * blockDim.x + threadIdx.x;
  if (k >= K) return;
  for (int j = 0; j < r_pad; ++j) {
    up32[static_cast<size_t>(j) * K + k] = (j < r) ? Up[static_cast<size_t>(k) * r + j] : 0.0f;
    if (ur32 != up32) ur32[static_cast<size_t>(j) * K + k] = (j < r) ? Ur[static_cast<size_t>(k) * r + j] : 0.0f;
  }
}

// ---- NVFP4 variant (App. B.1: E2M1 codes, an E4M3 scale per 16 K, one float32 scale per tensor)

// One thread per (output channel n, block b of 16 K): the block's absmax of |W_perp| (float64),
// and the tensor's absmax by an atomic max on the bit pattern (non-negative doubles order as
// unsigned integers).
template <typename WT>
__global__ void block_amax_nvfp4_kernel(const WT* __restrict__ W, const float* __restrict__ U,
                                        const double* __restrict__ Bf, int K, int N, int r, double* __restrict__ bam,
                                        unsigned long long* __restrict__ amax_bits) {
  int n = blockIdx.x * blockDim.x + threadIdx.x;
  int b = blockIdx.y;
  if (n >= N) return;
  double a = 0.0;
  for (int k = b * kFp4Block; k < (b + 1) * kFp4Block; ++k) a = fmax(a, fabs(wperp(W, U, Bf, N, r, k, n)));
  bam[static_cast<size_t>(n) * (K / kFp4Block) + b] = a;
  atomicMax(amax_bits, static_cast<unsigned long long>(__double_as_longlong(a)));
}

// E4M3 bits -> value (exact in float64).
__device__ __forceinline__ double e4m3_to_double(__nv_fp8_storage_t b) {
  __half_raw hr = __nv_cvt_fp8_to_halfraw(b, __NV_E4M3);
  return static_cast<double>(__half2float(__half(hr)));
}

// One thread per (n, b): s_g = RN_f32(amax / (6 * 448)); s_b = RN_e4m3(amax_b / (6 s_g)) and the
// codes RN_e2m1(w / (s_b s_g)), each from the float64 quotient (one rounding to a 4-bit format),
// saturating; a code of magnitude zero is stored as 0.  Codes are packed two per byte, low nibble =
// even k; the block scale goes to its atom (see internal.h).
template <typename WT>
__global__ void quantize_weight_nvfp4_kernel(const WT* __restrict__ W, const float* __restrict__ U,
                                             const double* __restrict__ Bf, int K, int N, int r,
                                             const double* __restrict__ bam,
                                             const unsigned long long* __restrict__ amax_bits,
                                             uint8_t* __restrict__ qw, uint8_t* __restrict__ sfw,
                                             float* __restrict__ sg_out) {
  int n = blockIdx.x * blockDim.x + threadIdx.x;
  int b = blockIdx.y;
  if (n >= N) return;
  const double amax = __longlong_as_double(static_cast<long long>(*amax_bits));
  const float sg = __double2float_rn(__ddiv_rn(amax, 2688.0));  // 6 * 448
  if (n == 0 && b == 0) *sg_out = sg;
  __nv_fp8_storage_t sb = 0;
  if (sg > 0.0f) {
    const double q = __ddiv_rn(bam[static_cast<size_t>(n) * (K / kFp4Block) + b], __dmul_rn(6.0, static_cast<double>(sg)));
    sb = __nv_cvt_double_to_fp8(q, __NV_SATFINITE, __NV_E4M3);
  }
  const int nr = n % 128;
  sfw[(static_cast<size_t>(n / 128) * (K / 64) + b / 4) * kSfAtom + (nr % 32) * 16 + (nr / 32) * 4 + (b % 4)] = sb;
  const double scale = __dmul_rn(e4m3_to_double(sb), static_cast<double>(sg));  // exact
  uint32_t lo = 0, hi = 0;
  for (int i = 0; i < kFp4Block; ++i) {
    uint32_t c = 0;
    if (scale > 0.0) {
      const double u = __ddiv_rn(wperp(W, U, Bf, N, r, b * kFp4Block + i, n), scale);
      c = static_cast<uint32_t>(__nv_cvt_double_to_fp4(u, __NV_E2M1, cudaRoundNearest)) & 0xFu;
      if ((c & 7u) == 0u) c = 0u;  // zero has one code
    }
    if (i < 8)
      lo |= c << (4 * i);
    else
      hi |= c << (4 * (i - 8));
  }
  *reinterpret_cast<uint2*>(qw + static_cast<size_t>(n) * (K / 2) + b * (kFp4Block / 2)) = make_uint2(lo, hi);
}

// ---- smoothing and block Hadamard rotation (Sec. 3 Eq. (pair); App. B.1), float64

// Columns n0 .. n0+15 of rows [kb, kb + B) of A [K, N] (bf16 or float32), each times scale[k]
// when scale is given, through the block Walsh-Hadamard butterflies (a + b, a - b) at spans
// 1, 2, ..., B/2, then times nrm = 1/sqrt(B): out [K, N] float64.  Within one span the pairs are
// disjoint, so every entry sees the same float64 operations in the same order as a sequential
// transform, whatever thread takes it.
constexpr int kRotCols = 16;
template <typename AT>
__global__ void __launch_bounds__(256) rotate_cols_kernel(const AT* __restrict__ A, const float* __restrict__ scale,
                                                          int N, int B, double nrm, double* __restrict__ out) {
  extern __shared__ double tile[];  // [B][kRotCols]
  const int kb = blockIdx.x * B, n0 = blockIdx.y * kRotCols;
  for (int i = threadIdx.x; i < B * kRotCols; i += blockDim.x) {
    const int k = i / kRotCols, c = i % kRotCols, n = n0 + c;
    double v = 0.0;
    if (n < N) {
      v = static_cast<double>(static_cast<float>(A[static_cast<size_t>(kb + k) * N + n]));
      if (scale) v = __dmul_rn(v, static_cast<double>(scale[kb + k]));
    }
    tile[i] = v;
  }
  for (int h = 1; h < B; h *= 2) {
    __syncthreads();
    for (int i = threadIdx.x; i < (B / 2) * kRotCols; i += blockDim.x) {
      const int pr = i / kRotCols, c = i % kRotCols;
      const int a = (pr / h) * 2 * h + pr % h, b = a + h;
      const double xa = tile[a * kRotCols + c], xb = tile[b * kRotCols + c];
      tile[a * kRotCols + c] = __dadd_rn(xa, xb);
      tile[b * kRotCols + c] = __dsub_rn(xa, xb);
    }
  }
  __syncthreads();
  for (int i = threadIdx.x; i < B * kRotCols; i += blockDim.x) {
    const int k = i / kRotCols, n = n0 + i % kRotCols;
    if (n < N) out[static_cast<size_t>(kb + k) * N + n] = __dmul_rn(tile[i], nrm);
  }
}

// From HU [K, r] (float64): the projection basis diag(s)^-1 H U and the reconstruction basis
// diag(s) H U, each rounded once to float32; and RN_f32(nrm / s_k), nrm = 1/sqrt(B), the factor
// the run-time rotation applies before its butterflies.
__global__ void rotated_bases_kernel(const double* __restrict__ HU, const float* __restrict__ sm, int K, int r,
                                     double nrm, float* __restrict__ Up, float* __restrict__ Ur,
                                     float* __restrict__ inv_s) {
  const int k = blockIdx.x * blockDim.x + threadIdx.x;
  if (k >= K) return;
  const double sk = sm ? static_cast<double>(sm[k]) : 1.0;
  inv_s[k] = __double2float_rn(__ddiv_rn(nrm, sk));
  for (int j = 0; j < r; ++j) {
    const double v = HU[static_cast<size_t>(k) * r + j];
    Up[static_cast<size_t>(k) * r + j] = __double2float_rn(__ddiv_rn(v, sk));
    Ur[static_cast<size_t>(k) * r + j] = __double2float_rn(__dmul_rn(v, sk));
  }
}

// Every factor must be a positive finite number.
__global__ void check_scale_kernel(const float* __restrict__ sm, int K, int* err) {
  const int k = blockIdx.x * blockDim.x + threadIdx.x;
  if (k < K && !(sm[k] > 0.0f && isfinite(sm[k]))) atomicOr(err, kErrRange);
}

template <typename WT>
cudaError_t pack_nvfp4(Handle& h, const WT* W, const float* U, const float* Up, const float* Ur, cudaStream_t s) {
  const int K = h.K, N = h.N, r = h.r;
  const int nb = K / kFp4Block;
  double* Bf = nullptr;
  double* bam = nullptr;
  unsigned long long* amax = nullptr;
  float* sg_dev = nullptr;
  cudaError_t e = cudaMalloc(&Bf, sizeof(double) * static_cast<size_t>(r > 0 ? r : 1) * N);
  if (e == cudaSuccess) e = cudaMalloc(&bam, sizeof(double) * static_cast<size_t>(N) * nb);
  if (e == cudaSuccess) e = cudaMalloc(&amax, 16);
  if (e == cudaSuccess) e = cudaMemsetAsync(amax, 0, 16, s);
  if (e == cudaSuccess) {
    sg_dev = reinterpret_cast<float*>(amax + 1);
    const int T = 128;
    if (r > 0) branch_weight_kernel<<<dim3((N + T - 1) / T, r), T, 0, s>>>(W, U, K, N, r, Bf);
    block_amax_nvfp4_kernel<<<dim3((N + T - 1) / T, nb), T, 0, s>>>(W, U, Bf, K, N, r, bam, amax);
    quantize_weight_nvfp4_kernel<<<dim3((N + T - 1) / T, nb), T, 0, s>>>(W, U, Bf, K, N, r, bam, amax, h.qw, h.sfw,
                                                                          sg_dev);
    if (r > 0) {
      branch_half_kernel<<<(N + T - 1) / T, T, 0, s>>>(Bf, N, r, h.r_pad, h.Bh, h.err);
      if (h.ucat_t)  // kernel (a)'s tensor-core bases (r_pad <= kMaxRank)
        split_basis_kernel<<<(K + T - 1) / T, T, 0, s>>>(Up, Ur, K, r, h.r_pad, h.ku3, h.ucat_t, h.ucat3);
      basis32_kernel<<<(K + T - 1) / T, T, 0, s>>>(Up, Ur, K, r, h.r_pad, h.up32, h.ur32);
    }
    e = cudaGetLastError();
    cudaError_t e2 = cudaStreamSynchronize(s);
    if (e == cudaSuccess) e = e2;
    if (e == cudaSuccess) e = cudaMemcpy(&h.sg, sg_dev, sizeof(float), cudaMemcpyDeviceToHost);
  }
  cudaFree(Bf);
  cudaFree(bam);
  cudaFree(amax);
  return e;
}

template <typename WT>
cudaError_t pack_int4(Handle& h, const WT* W, const float* U, const float* Up, const float* Ur, cudaStream_t s) {
  const int K = h.K, N = h.N, r = h.r;
  double* Bf = nullptr;
  cudaError_t e = cudaMalloc(&Bf, sizeof(double) * static_cast<size_t>(r > 0 ? r : 1) * N);
  if (e != cudaSuccess) return e;
  const int T = 128;
  if (r > 0) {
    branch_weight_kernel<<<dim3((N + T - 1) / T, r), T, 0, s>>>(W, U, K, N, r, Bf);
  }
  quantize_weight_kernel<<<dim3((N + T - 1) / T, K / h.G), T, 0, s>>>(W, U, Bf, K, N, r, h.G, h.N_pad, h.qw, h.sw,
                                                                     h.err);
  if (r > 0) {
    branch_half_kernel<<<(N + T - 1) / T, T, 0, s>>>(Bf, N, r, h.r_pad, h.Bh, h.err);
    if (h.ucat_t)  // kernel (a)'s tensor-core bases (r_pad <= kMaxRank)
      split_basis_kernel<<<(K + T - 1) / T, T, 0, s>>>(Up, Ur, K, r, h.r_pad, h.ku3, h.ucat_t, h.ucat3);
    basis32_kernel<<<(K + T - 1) / T, T, 0, s>>>(Up, Ur, K, r, h.r_pad, h.up32, h.ur32);
  }
  column_shift_kernel<<<(h.N_pad + T - 1) / T, T, 0, s>>>(h.sw, h.Bh, K / h.G, h.N_pad, h.r_pad, h.swh, h.Bhs, h.fcol);
  e = cudaGetLastError();
  cudaError_t e2 = cudaStreamSynchronize(s);
  cudaFree(Bf);
  return e != cudaSuccess ? e : e2;
}

}  // namespace

cudaError_t launch_pack_nvfp4(Handle& h, const __nv_bfloat16* W, const float* U, cudaStream_t s) {
  return pack_nvfp4(h, W, U, U, U, s);
}

cudaError_t launch_pack(Handle& h, const __nv_bfloat16* W, const float* U, cudaStream_t s) {
  return pack_int4(h, W, U, U, U, s);
}

// W~ = H diag(s) W and H U in float64, the two run-time bases and 1/s, then the ordinary pack of
// W~ against U (U spans the protected directions in the rotated coordinates).
cudaError_t launch_pack_rotated(Handle& h, const __nv_bfloat16* W, const float* sm, const float* U, cudaStream_t s) {
  const int K = h.K, N = h.N, r = h.r, B = h.hb;
  const double nrm = 1.0 / std::sqrt(static_cast<double>(B));
  const size_t smem = sizeof(double) * B * kRotCols;
  double* Wt = nullptr;
  double* HU = nullptr;
  float* Upr = nullptr;
  cudaError_t e = cudaFuncSetAttribute(rotate_cols_kernel<__nv_bfloat16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(rotate_cols_kernel<float>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(smem));
  if (e == cudaSuccess) e = cudaMalloc(&Wt, sizeof(double) * static_cast<size_t>(K) * N);
  if (e == cudaSuccess) e = cudaMalloc(&HU, sizeof(double) * static_cast<size_t>(K) * (r > 0 ? r : 1));
  if (e == cudaSuccess) e = cudaMalloc(&Upr, sizeof(float) * 2 * static_cast<size_t>(K) * (r > 0 ? r : 1));
  if (e == cudaSuccess) {
    const int T = 128;
    if (sm) check_scale_kernel<<<(K + T - 1) / T, T, 0, s>>>(sm, K, h.err);
    rotate_cols_kernel<__nv_bfloat16><<<dim3(K / B, (N + kRotCols - 1) / kRotCols), 256, smem, s>>>(W, sm, N, B, nrm, Wt);
    if (r > 0)
      rotate_cols_kernel<float><<<dim3(K / B, (r + kRotCols - 1) / kRotCols), 256, smem, s>>>(U, nullptr, r, B, nrm, HU);
    float* Up = Upr;
    float* Ur = Upr + static_cast<size_t>(K) * (r > 0 ? r : 1);
    rotated_bases_kernel<<<(K + T - 1) / T, T, 0, s>>>(HU, sm, K, r, nrm, Up, Ur, h.inv_s);
    e = cudaGetLastError();
    if (e == cudaSuccess)
      e = h.fmt == kFmtNvfp4 ? pack_nvfp4(h, static_cast<const double*>(Wt), U, Up, Ur, s)
                             : pack_int4(h, static_cast<const double*>(Wt), U, Up, Ur, s);
  }
  cudaStreamSynchronize(s);
  cudaFree(Wt);
  cudaFree(HU);
  cudaFree(Upr);
  return e;
}

}  // namespace qwam
