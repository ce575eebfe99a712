// subspace.cu -- the offline choice of what ASP protects (Q-WAM Sec. 4.2-4.3; App. A; App. B.1).
//
//   smoothing factors   s_j = max|X_j|^alpha / max|W_j,:|^(1 - alpha)          (App. B.1)
//   rotated AOG         G~  = H diag(gamma) G diag(gamma) H                      (Sec. 4.2)
//   action subspace     V   = the eigenvectors of the r largest eigenvalues of G~ (Sec. 4.2; App. A)
//   action mass         mu_E = sum of tr G~ over an expert's layers               (Sec. 4.3, Eq. (mass))
//
// H is block diagonal with normalised Sylvester Hadamard blocks of size B, the largest power of
// two dividing d (at most 1024).  G~ is formed with two passes of a block fast Walsh-Hadamard
// transform along rows (the second on the transpose), with the gamma scaling folded into the first.
//
// The top-r eigenvectors come from subspace iteration with p = r + max(8, r/2) vectors: W = G~ V,
// then V = orth(W) by CholeskyQR2 (the Gram matrix, its Cholesky factor and that factor's inverse in
// float64), and at the end a Rayleigh-Ritz step: the p x p matrix V^T G~ V is diagonalised on the
// host by cyclic Jacobi in float64 and V is rotated onto its top r eigenvectors.  The error of the
// subspace falls like (lambda_{p+1} / lambda_r)^iters; the start vectors are a fixed hash of the
// index, so the result depends only on G~.
#include <algorithm>
#include <cmath>
#include <vector>

#include "internal.h"

namespace qwam {
namespace {

constexpr int kPMax = 96;  // largest subspace (r + oversampling) handled

size_t align256(size_t b) { return (b + 255) & ~size_t(255); }

__device__ __forceinline__ float block_max(float v) {
  __shared__ float red[32];
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
  __syncthreads();
  if (threadIdx.x < 32) {
    v = threadIdx.x < (blockDim.x >> 5) ? red[threadIdx.x] : 0.0f;
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  }
  return v;  // valid in thread 0
}

// s_j for input channel j (row j of W [K, N]); a zero maximum leaves the channel unsmoothed.
__global__ void smoothing_kernel(const float* xmax, const __nv_bfloat16* W, int N, double alpha, float* s) {
  const int j = blockIdx.x;
  float m = 0.0f;
  for (int n = threadIdx.x; n < N; n += blockDim.x) m = fmaxf(m, fabsf(__bfloat162float(W[static_cast<size_t>(j) * N + n])));
  m = block_max(m);
  if (threadIdx.x == 0) {
    const double x = xmax[j];
    s[j] = (x > 0.0 && m > 0.0f) ? static_cast<float>(pow(x, alpha) / pow(static_cast<double>(m), 1.0 - alpha)) : 1.0f;
  }
}

// out[i, :] = normalised block FWHT (block B) of the row (g_i g_j in[i, j])_j; g may be null.
__global__ void row_fwht_kernel(const float* in, const float* g, int d, int B, float nrm, float* out) {
  extern __shared__ float row[];
  const int i = blockIdx.x;
  const float gi = g ? g[i] : 1.0f;
  for (int j = threadIdx.x; j < d; j += blockDim.x) row[j] = in[static_cast<size_t>(i) * d + j] * (g ? gi * g[j] : 1.0f);
  __syncthreads();
  const int half = B >> 1;
  for (int h = 1; h < B; h <<= 1) {
    for (int t = threadIdx.x; t < d / 2; t += blockDim.x) {
      const int b = t / half, q = t % half;
      const int u = b * B + (q / h) * 2 * h + q % h;  // butterfly (u, u + h) of block b
      const float x = row[u], y = row[u + h];
      row[u] = x + y;
      row[u + h] = x - y;
    }
    __syncthreads();
  }
  for (int j = threadIdx.x; j < d; j += blockDim.x) out[static_cast<size_t>(i) * d + j] = row[j] * nrm;
}

__global__ void transpose_kernel(const float* in, int d, float* out) {
  __shared__ float t[32][33];
  const int x0 = blockIdx.x * 32, y0 = blockIdx.y * 32;
  for (int k = threadIdx.y; k < 32; k += blockDim.y) {
    const int y = y0 + k, x = x0 + threadIdx.x;
    if (y < d && x < d) t[k][threadIdx.x] = in[static_cast<size_t>(y) * d + x];
  }
  __syncthreads();
  for (int k = threadIdx.y; k < 32; k += blockDim.y) {
    const int y = x0 + k, x = y0 + threadIdx.x;
    if (y < d && x < d) out[static_cast<size_t>(y) * d + x] = t[threadIdx.x][k];
  }
}

__global__ void trace_kernel(const float* A, int d, double* out) {
  __shared__ double red[256];
  double s = 0.0;
  for (int i = threadIdx.x; i < d; i += blockDim.x) s += A[static_cast<size_t>(i) * d + i];
  red[threadIdx.x] = s;
  __syncthreads();
  for (int w = blockDim.x / 2; w > 0; w >>= 1) {
    if (static_cast<int>(threadIdx.x) < w) red[threadIdx.x] += red[threadIdx.x + w];
    __syncthreads();
  }
  if (threadIdx.x == 0) *out = red[0];
}

// Start vectors: a fixed hash of the index, uniform in [-1, 1).
__global__ void start_kernel(float* V, int n) {
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= n) return;
  uint32_t h = static_cast<uint32_t>(idx) * 2654435761u + 0x9E3779B9u;
  h ^= h >> 16;
  h *= 0x85EBCA6Bu;
  h ^= h >> 13;
  h *= 0xC2B2AE35u;
  h ^= h >> 16;
  V[idx] = static_cast<float>(h >> 8) * (2.0f / 16777216.0f) - 1.0f;
}

// W = A V, A [d, d] row-major, V and W [d, p] row-major (p <= kPMax).  A CTA: 32 rows of A.
__global__ void __launch_bounds__(256) av_kernel(const float* A, const float* V, int d, int p, float* W) {
  __shared__ float As[32][33];
  __shared__ float Vs[32][kPMax];
  const int t = threadIdx.x, r = t >> 3, cq = t & 7;
  const int row0 = blockIdx.x * 32;
  float acc[kPMax / 8];
#pragma unroll
  for (int k = 0; k < kPMax / 8; ++k) acc[k] = 0.0f;
  for (int k0 = 0; k0 < d; k0 += 32) {
    for (int e = t; e < 32 * 32; e += 256) {
      const int rr = e >> 5, kk = e & 31;
      As[rr][kk] = (row0 + rr < d && k0 + kk < d) ? A[static_cast<size_t>(row0 + rr) * d + k0 + kk] : 0.0f;
    }
    for (int e = t; e < 32 * kPMax; e += 256) {
      const int kk = e / kPMax, c = e % kPMax;
      Vs[kk][c] = (k0 + kk < d && c < p) ? V[static_cast<size_t>(k0 + kk) * p + c] : 0.0f;
    }
    __syncthreads();
#pragma unroll 4
    for (int kk = 0; kk < 32; ++kk) {
      const float a = As[r][kk];
#pragma unroll
      for (int k = 0; k < kPMax / 8; ++k) acc[k] = fmaf(a, Vs[kk][cq + 8 * k], acc[k]);
    }
    __syncthreads();
  }
  if (row0 + r < d) {
#pragma unroll
    for (int k = 0; k < kPMax / 8; ++k) {
      const int c = cq + 8 * k;
      if (c < p) W[static_cast<size_t>(row0 + r) * p + c] = acc[k];
    }
  }
}

// part[b] = X^T Y over rows [32 b, 32 b + 32), in float64 (X, Y [d, p] row-major; part [p, p]).
__global__ void __launch_bounds__(256) gram_kernel(const float* X, const float* Y, int d, int p, double* part) {
  __shared__ float Xs[32][kPMax], Ys[32][kPMax];
  const int row0 = blockIdx.x * 32;
  for (int e = threadIdx.x; e < 32 * p; e += blockDim.x) {
    const int rr = e / p, c = e % p;
    const bool in = row0 + rr < d;
    Xs[rr][c] = in ? X[static_cast<size_t>(row0 + rr) * p + c] : 0.0f;
    Ys[rr][c] = in ? Y[static_cast<size_t>(row0 + rr) * p + c] : 0.0f;
  }
  __syncthreads();
  double* out = part + static_cast<size_t>(blockIdx.x) * p * p;
  for (int e = threadIdx.x; e < p * p; e += blockDim.x) {
    const int a = e / p, c = e % p;
    double s = 0.0;
    for (int rr = 0; rr < 32; ++rr) s += static_cast<double>(Xs[rr][a]) * static_cast<double>(Ys[rr][c]);
    out[e] = s;
  }
}

// out = the sum of the nparts partials, in partial order (a fixed order).
__global__ void reduce_parts_kernel(const double* part, int nparts, int n, double* out) {
  const int e = blockIdx.x * blockDim.x + threadIdx.x;
  if (e >= n) return;
  double s = 0.0;
  for (int b = 0; b < nparts; ++b) s += part[static_cast<size_t>(b) * n + e];
  out[e] = s;
}

// One CTA: L = chol(C) and Linv = L^-1 (both p x p, float64, row-major, in global scratch).  A
// pivot that is not positive (a rank-deficient block) is replaced by a tiny positive one.
__global__ void chol_inv_kernel(const double* C, int p, double* L, double* Linv) {
  for (int e = threadIdx.x; e < p * p; e += blockDim.x) {
    L[e] = 0.0;
    Linv[e] = 0.0;
  }
  __syncthreads();
  for (int k = 0; k < p; ++k) {
    if (threadIdx.x == 0) {
      double s = C[k * p + k];
      for (int j = 0; j < k; ++j) s -= L[k * p + j] * L[k * p + j];
      L[k * p + k] = sqrt(s > 1e-300 ? s : 1e-300);
    }
    __syncthreads();
    for (int i = k + 1 + threadIdx.x; i < p; i += blockDim.x) {
      double s = C[i * p + k];
      for (int j = 0; j < k; ++j) s -= L[i * p + j] * L[k * p + j];
      L[i * p + k] = s / L[k * p + k];
    }
    __syncthreads();
  }
  // forward substitution, one column of the inverse per thread
  for (int c = threadIdx.x; c < p; c += blockDim.x) {
    for (int i = c; i < p; ++i) {
      double s = (i == c) ? 1.0 : 0.0;
      for (int j = c; j < i; ++j) s -= L[i * p + j] * Linv[j * p + c];
      Linv[i * p + c] = s / L[i * p + i];
    }
  }
}

// V[i, c] = sum_{k <= c} W[i, k] Linv[c, k]  (V = W Linv^T: orthonormal columns when Linv^-1 is
// the Cholesky factor of W^T W).
__global__ void apply_linv_kernel(const float* W, const double* Linv, int d, int p, float* V) {
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= d * p) return;
  const int i = idx / p, c = idx % p;
  double s = 0.0;
  for (int k = 0; k <= c; ++k) s += static_cast<double>(W[static_cast<size_t>(i) * p + k]) * Linv[c * p + k];
  V[idx] = static_cast<float>(s);
}

// out[i, j] = sum_k V[i, k] Q[k, j] for j < r (V [d, p], Q [p, r] float64).
__global__ void rotate_kernel(const float* V, const double* Q, int d, int p, int r, float* out) {
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= d * r) return;
  const int i = idx / r, j = idx % r;
  double s = 0.0;
  for (int k = 0; k < p; ++k) s += static_cast<double>(V[static_cast<size_t>(i) * p + k]) * Q[k * r + j];
  out[idx] = static_cast<float>(s);
}

// Cyclic Jacobi eigendecomposition of the symmetric n x n matrix A (row-major, float64, destroyed):
// eigenvalues in w, eigenvectors in the columns of Z.
void jacobi_eigen(std::vector<double>& A, int n, std::vector<double>& w, std::vector<double>& Z) {
  Z.assign(static_cast<size_t>(n) * n, 0.0);
  for (int i = 0; i < n; ++i) Z[i * n + i] = 1.0;
  double norm = 0.0;
  for (double v : A) norm += v * v;
  for (int sweep = 0; sweep < 60; ++sweep) {
    double off = 0.0;
    for (int i = 0; i < n; ++i)
      for (int j = i + 1; j < n; ++j) off += A[i * n + j] * A[i * n + j];
    if (off <= 1e-30 * norm) break;
    for (int pi = 0; pi < n; ++pi)
      for (int q = pi + 1; q < n; ++q) {
        const double apq = A[pi * n + q];
        if (apq == 0.0) continue;
        const double theta = (A[q * n + q] - A[pi * n + pi]) / (2.0 * apq);
        const double t = (theta >= 0 ? 1.0 : -1.0) / (std::fabs(theta) + std::sqrt(theta * theta + 1.0));
        const double c = 1.0 / std::sqrt(t * t + 1.0), s = t * c;
        for (int k = 0; k < n; ++k) {  // A = J^T A J, columns pi and q then rows pi and q
          const double akp = A[k * n + pi], akq = A[k * n + q];
          A[k * n + pi] = c * akp - s * akq;
          A[k * n + q] = s * akp + c * akq;
        }
        for (int k = 0; k < n; ++k) {
          const double apk = A[pi * n + k], aqk = A[q * n + k];
          A[pi * n + k] = c * apk - s * aqk;
          A[q * n + k] = s * apk + c * aqk;
        }
        for (int k = 0; k < n; ++k) {
          const double zkp = Z[k * n + pi], zkq = Z[k * n + q];
          Z[k * n + pi] = c * zkp - s * zkq;
          Z[k * n + q] = s * zkp + c * zkq;
        }
      }
  }
  w.resize(n);
  for (int i = 0; i < n; ++i) w[i] = A[i * n + i];
}

struct SubspaceScratch {
  float *V, *W;
  double *part, *C, *L, *Linv, *Q;
};

size_t subspace_bytes(int d, int p, int r, SubspaceScratch* s, uint8_t* base) {
  const int nparts = (d + 31) / 32;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    uint8_t* q = base ? base + off : nullptr;
    off += align256(bytes);
    return q;
  };
  uint8_t* v = take(static_cast<size_t>(d) * p * 4);
  uint8_t* w = take(static_cast<size_t>(d) * p * 4);
  uint8_t* part = take(static_cast<size_t>(nparts) * p * p * 8);
  uint8_t* c = take(static_cast<size_t>(p) * p * 8);
  uint8_t* l = take(static_cast<size_t>(p) * p * 8);
  uint8_t* li = take(static_cast<size_t>(p) * p * 8);
  uint8_t* q = take(static_cast<size_t>(p) * r * 8);
  if (s) {
    s->V = reinterpret_cast<float*>(v);
    s->W = reinterpret_cast<float*>(w);
    s->part = reinterpret_cast<double*>(part);
    s->C = reinterpret_cast<double*>(c);
    s->L = reinterpret_cast<double*>(l);
    s->Linv = reinterpret_cast<double*>(li);
    s->Q = reinterpret_cast<double*>(q);
  }
  return off;
}

}  // namespace

int subspace_width(int d, int r) {
  int p = r + std::max(8, r / 2);
  if (p > d) p = d;
  if (p > kPMax) p = kPMax;
  return p;
}

size_t subspace_workspace_bytes(int d, int r) { return subspace_bytes(d, subspace_width(d, r), r, nullptr, nullptr); }

cudaError_t launch_smoothing(const float* xmax, const __nv_bfloat16* W, int K, int N, double alpha, float* s,
                             cudaStream_t st) {
  smoothing_kernel<<<K, 256, 0, st>>>(xmax, W, N, alpha, s);
  return cudaGetLastError();
}

cudaError_t launch_rotated_gramian(const float* G, const float* gamma, int d, float* Gt, float* work, cudaStream_t st) {
  int B = 1;
  while (d % (2 * B) == 0 && 2 * B <= 1024) B *= 2;
  const float nrm = static_cast<float>(1.0 / std::sqrt(static_cast<double>(B)));
  const size_t smem = static_cast<size_t>(d) * 4;
  cudaError_t e = cudaFuncSetAttribute(row_fwht_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  const dim3 tg((d + 31) / 32, (d + 31) / 32), tb(32, 8);
  row_fwht_kernel<<<d, 256, smem, st>>>(G, gamma, d, B, nrm, work);   // (D G D) H
  transpose_kernel<<<tg, tb, 0, st>>>(work, d, Gt);
  row_fwht_kernel<<<d, 256, smem, st>>>(Gt, nullptr, d, B, nrm, work);  // ((D G D) H)^T H
  transpose_kernel<<<tg, tb, 0, st>>>(work, d, Gt);                     // H (D G D) H
  return cudaGetLastError();
}

cudaError_t gramian_trace(const float* A, int d, double* host_out, cudaStream_t st) {
  double* dv = nullptr;
  cudaError_t e = cudaMallocAsync(reinterpret_cast<void**>(&dv), sizeof(double), st);
  if (e != cudaSuccess) return e;
  trace_kernel<<<1, 256, 0, st>>>(A, d, dv);
  e = cudaGetLastError();
  if (e == cudaSuccess) e = cudaMemcpyAsync(host_out, dv, sizeof(double), cudaMemcpyDeviceToHost, st);
  cudaFreeAsync(dv, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  return e;
}

cudaError_t action_subspace(const float* Gt, int d, int r, int iters, float* V_out, float* lambda, void* work,
                            cudaStream_t st) {
  const int p = subspace_width(d, r);
  SubspaceScratch s;
  subspace_bytes(d, p, r, &s, static_cast<uint8_t*>(work));
  const int nparts = (d + 31) / 32;
  const int n = d * p;
  const int T = 256;
  auto orthonormalize = [&](const float* Wsrc, float* Vdst) {  // Vdst = orth(Wsrc), CholeskyQR
    gram_kernel<<<nparts, T, 0, st>>>(Wsrc, Wsrc, d, p, s.part);
    reduce_parts_kernel<<<(p * p + T - 1) / T, T, 0, st>>>(s.part, nparts, p * p, s.C);
    chol_inv_kernel<<<1, 128, 0, st>>>(s.C, p, s.L, s.Linv);
    apply_linv_kernel<<<(n + T - 1) / T, T, 0, st>>>(Wsrc, s.Linv, d, p, Vdst);
  };
  start_kernel<<<(n + T - 1) / T, T, 0, st>>>(s.W, n);
  orthonormalize(s.W, s.V);
  orthonormalize(s.V, s.W);  // CholeskyQR2
  std::swap(s.V, s.W);
  for (int it = 0; it < iters; ++it) {
    av_kernel<<<(d + 31) / 32, 256, 0, st>>>(Gt, s.V, d, p, s.W);
    orthonormalize(s.W, s.V);
    orthonormalize(s.V, s.W);
    std::swap(s.V, s.W);
  }
  // Rayleigh-Ritz: T = V^T G~ V (p x p), diagonalised on the host
  av_kernel<<<(d + 31) / 32, 256, 0, st>>>(Gt, s.V, d, p, s.W);
  gram_kernel<<<nparts, T, 0, st>>>(s.V, s.W, d, p, s.part);
  reduce_parts_kernel<<<(p * p + T - 1) / T, T, 0, st>>>(s.part, nparts, p * p, s.C);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  std::vector<double> Tm(static_cast<size_t>(p) * p), w, Z;
  e = cudaMemcpyAsync(Tm.data(), s.C, Tm.size() * 8, cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) return e;
  for (int i = 0; i < p; ++i)  // symmetrise (the two halves differ by rounding)
    for (int j = i + 1; j < p; ++j) Tm[i * p + j] = Tm[j * p + i] = 0.5 * (Tm[i * p + j] + Tm[j * p + i]);
  jacobi_eigen(Tm, p, w, Z);
  std::vector<int> order(p);
  for (int i = 0; i < p; ++i) order[i] = i;
  std::stable_sort(order.begin(), order.end(), [&](int a, int b) { return w[a] > w[b]; });
  std::vector<double> Q(static_cast<size_t>(p) * r);
  std::vector<float> lam(r);
  for (int j = 0; j < r; ++j) {
    lam[j] = static_cast<float>(w[order[j]]);
    for (int k = 0; k < p; ++k) Q[static_cast<size_t>(k) * r + j] = Z[static_cast<size_t>(k) * p + order[j]];
  }
  e = cudaMemcpyAsync(s.Q, Q.data(), Q.size() * 8, cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess) e = cudaMemcpyAsync(lambda, lam.data(), r * 4, cudaMemcpyHostToDevice, st);
  if (e != cudaSuccess) return e;
  rotate_kernel<<<(d * r + T - 1) / T, T, 0, st>>>(s.V, s.Q, d, p, r, V_out);
  e = cudaGetLastError();
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  return e;
}

}  // namespace qwam
