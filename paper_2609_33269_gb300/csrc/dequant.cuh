// dequant.cuh -- float16 expansion of the packed 4-bit weights (INT4 format, Eq. (quant) with
// b = 4 and bfloat16 group scales), shared by kernel (b)'s on-the-fly conversion, the weight
// expansion kernel and kernel (a), which expands a call's weights while its own first pass waits
// on HBM.
//
// Every expanded value s c has at most 11 significant bits (an 8-bit scale times a 3-bit code):
// the float16 operations below are exact.
#pragma once

#include <cuda_fp16.h>
#include <stdint.h>

namespace qwam {

// Packed float16 pairs live in 32-bit registers throughout (low half = the even k).
__device__ __forceinline__ uint32_t mul_f16x2(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("mul.rn.f16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}
__device__ __forceinline__ uint32_t sub_f16x2(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("sub.rn.f16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}
__device__ __forceinline__ uint32_t f32x2_to_f16x2(float lo, float hi) {
  uint32_t d;
  asm("cvt.rn.f16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(hi), "f"(lo));
  return d;
}

// The dequantization constants of one scale s (float16, 8 significant bits): the pairs (s, s) and
// (s/16, s/16), both exact.
struct DqScale {
  uint32_t s1, s16;
};
__device__ __forceinline__ DqScale dq_scale(float s) {
  return DqScale{f32x2_to_f16x2(s, s), f32x2_to_f16x2(0.0625f * s, 0.0625f * s)};
}

// One OB4 word (codes k = 8j..8j+7, nibbles n = c + 8) times the scale -> four float16 pairs in k
// order.  Under the float16 pattern of 1024 (0x6400, whose unit in the last place is 1) the nibbles
// of bits 0..3 read as 1024 + n and those of bits 4..7 as 1024 + 16 n; subtracting 1032 or 1152
// leaves c or 16 c exactly, and multiplying by s or s/16 gives c s exactly (at most 11 significant
// bits).  Pairs 2 and 3 take the same steps on the word shifted down by 8.  Five integer and eight
// float16 operations per 8 codes.
__device__ __forceinline__ void dequant_word(uint32_t w, const DqScale& d, uint32_t* out) {
  constexpr uint32_t k1032 = 0x64086408u, k1152 = 0x64806480u, kMag = 0x64006400u;
  const uint32_t w2 = w >> 8;
  out[0] = mul_f16x2(sub_f16x2((w & 0x000F000Fu) | kMag, k1032), d.s1);
  out[1] = mul_f16x2(sub_f16x2((w & 0x00F000F0u) | kMag, k1152), d.s16);
  out[2] = mul_f16x2(sub_f16x2((w2 & 0x000F000Fu) | kMag, k1032), d.s1);
  out[3] = mul_f16x2(sub_f16x2((w2 & 0x00F000F0u) | kMag, k1152), d.s16);
}

// The float16 weights of one call, [N_pad, K + r_pad] row-major:
//   W16[n, k] = s_w[g, n] 2^e_n c[n, k]   for k < K (g = k / G)
//   W16[n, k] = B_hat[n, k - K] 2^e_n     for K <= k < K + r_pad.
struct W16Args {
  const uint32_t* qw;  // [N_pad, K/8] OB4 words
  const __half* swh;   // [K/G, N_pad] float16 s_w 2^e_n
  const __half* bhs;   // [N_pad, r_pad] float16 B_hat 2^e_n
  __half* w16;         // destination; nullptr: nothing to expand
  int K, r_pad, N_pad;
  int gshift;          // log2(G / 8): word j of a row belongs to group j >> gshift
};

// One thread's share of W16: the pieces (8 consecutive k of a row) first, first + stride, ...
// P pieces a round with all their loads issued before the first conversion, so that a thread keeps
// P loads in flight.  (N_pad (K + r_pad) / 8 < 2^31 for every layer the pack accepts: 32-bit piece
// indices.)  Consecutive threads take consecutive pieces, so that a warp's loads and stores are
// contiguous.
template <int P>
__device__ __forceinline__ void expand_w16(const W16Args& a, int first, int stride) {
  const int kp = a.K / 8;  // pieces of the K part per row
  const int ld = a.K + a.r_pad;
  const int total = a.N_pad * kp;
  for (int i0 = first; i0 < total; i0 += P * stride) {
    uint32_t w[P];
    unsigned short sc[P];
#pragma unroll
    for (int u = 0; u < P; ++u) {
      const int i = i0 + u * stride;
      w[u] = 0u;
      sc[u] = 0;
      if (i < total) {
        const int n = i / kp, j = i - n * kp;
        w[u] = a.qw[i];  // row n, word j
        sc[u] = __half_as_ushort(a.swh[static_cast<size_t>(j >> a.gshift) * a.N_pad + n]);
      }
    }
#pragma unroll
    for (int u = 0; u < P; ++u) {
      const int i = i0 + u * stride;
      if (i < total) {
        const int n = i / kp, j = i - n * kp;
        uint32_t v[4];
        dequant_word(w[u], dq_scale(__half2float(__ushort_as_half(sc[u]))), v);
        *reinterpret_cast<uint4*>(a.w16 + static_cast<size_t>(n) * ld + 8 * j) = make_uint4(v[0], v[1], v[2], v[3]);
      }
    }
  }
  // the branch columns: B_hat 2^e_n copied after the K part of each row
  const int bp = a.r_pad / 8;
  const int total_b = a.N_pad * bp;
  for (int i = first; i < total_b; i += stride) {
    const int n = i / bp, j = i - n * bp;
    *reinterpret_cast<uint4*>(a.w16 + static_cast<size_t>(n) * ld + a.K + 8 * j) =
        *reinterpret_cast<const uint4*>(a.bhs + static_cast<size_t>(n) * a.r_pad + 8 * j);
  }
}

}  // namespace qwam
