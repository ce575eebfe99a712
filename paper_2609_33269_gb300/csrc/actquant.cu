// actquant.cu -- kernel (a): the run-time activation path of the ASP layer.
//
//   p      = X U                (Sec. 4.2 Eq. (xsplit): the protected coordinates V^T x)
//   X_perp = X - p U^T          (the remainder (I - V V^T) x)
//   s_x    = RN_bf16(absmax(X_perp over a group) / 7),  codes = nearest(X_perp / s_x)
//                               (Eq. (quant) with b = 4; App. B.1: per token, per group)
//   p_hat  = RN_f16(p)          (the 16-bit branch input of Eq. (asp))
//
// One CTA owns 128 token rows (one TMEM lane per row) and a slice of K; the C CTAs of a
// thread-block cluster cover the whole of K for the same rows.  Each CTA streams its X slice
// through a TMA ring twice: pass 1 feeds p_part = X_slice [U_hi | U_lo] into TMEM (bf16
// tensor-core MMA, float32 accumulation); the CTAs' partial projections meet in a float32
// scratch in the workspace (through L2, one cluster barrier) and each CTA sums them in rank
// order, so every CTA sees the same p;
// pass 2 re-reads the slice (L2-resident by then) while the tensor cores form
// R = [p_hi | p_hi | p_lo] [U_hi | U_lo | U_hi]^T chunk by chunk, and the epilogue warps form
// X_perp = X - R in float32 and quantize it.  With r = 0 the kernel is one streaming pass.
//
// Outputs per token row m and group g (the activation workspace):
//   codes[m, :]   packed at four bits, OB4 words (ob4_word: word j holds k = 8j..8j+7 as
//                 offset-binary nibbles), which the GEMM expands to float16 values s_x c;
//   s_x[g, m]     bfloat16 scale;
//   p_hat[m, :]   float16.
// NVFP4 variant (App. B.1, the same kernel with one template flag): per block of 16 K an E4M3
// scale (in the 512-byte atoms the GEMM copies to tensor memory) and E2M1 codes, two per byte.
//
// Warp roles (576 threads): warp 0 TMA producer, warp 1 MMA issuer and TMEM owner, warps 2..17
// epilogue: in groups of four they cover the four 32-row TMEM quadrants, and the groups take
// (even chunks, columns 0..31), (odd, 0..31), (even, 32..63), (odd, 32..63) of each 64-column
// chunk, one thread per row.  A group of 64 columns has its absmax formed from the two halves'
// partial maxima, swapped through shared memory.  The quantizer's codes come from a fast
// rounding that an exact remainder test confirms (codes8_fast).  For an INT4 layer whose GEMM
// takes float16 weights, the epilogue warps first write those weights (expand_w16) while pass 1
// waits on HBM, when the launch asks for it (qwam_asp_linear).
//
// Also in this file, sharing kernel (a)'s quantizers (the same rounding, bit for bit):
//   rotquant_kernel  smoothing and block Hadamard rotation of the remainder (Sec. 3 Eq. (pair)),
//                    then quantization, one warp per token row and Hadamard block;
//   smallq_kernel    the whole activation path on the CUDA cores, one CTA per token row, for few
//                    tokens and for r = 0 layers (with the rotation for rotated layers);
//   debug kernels    the thread-per-row and warp-wide quantizers on caller-given rows (tests).
// launch_actquant at the end of the file chooses among them.
#include <algorithm>

#include "internal.h"
#include "ptx.cuh"

namespace qwam {
namespace {

struct ActArgs {
  int M, K, G, C, Kc, M_pad;
  uint8_t* codes;   // [M, K/2]: OB4 words (NVFP4: E2M1 codes, two per byte, low nibble = even k)
  uint8_t* sf;      // NVFP4: E4M3 block scales in 512-byte atoms
  __nv_bfloat16* scales;  // [K/G, M_pad]
  __half* phat;     // [M, RP]
  float* part;      // [C, M_pad, RP] float32: the CTAs' partial projections, exchanged through L2
  float* dump;      // optional [M, K]
  int resid_only;   // rotated layer: write the remainder to dump and stop (the rotation kernel quantizes)
  W16Args w;        // INT4 with r > 0: the call's float16 weights for the GEMM (w.w16 == nullptr: none)
  int* err;
  uint64_t timeout_ns;
};

constexpr int kNumRec = 4;  // TMEM reconstruction buffers (64 columns each)
constexpr int kActThreads = 576;  // warp 0 TMA, warp 1 MMA, warps 2..17 epilogue

template <int RP>
struct ActCfg {
  static constexpr int KU3 = RP == 0 ? 0 : ((3 * RP + 63) / 64) * 64;  // (hi, hi, lo) width, padded
  static constexpr int X_BYTES = kBM * kChunk * 2;                     // 16 KB, 128-byte swizzle
  static constexpr int U1_BYTES = 2 * RP * 128;                        // [U_hi|U_lo]^T chunk
  static constexpr int U2_BYTES = kChunk * KU3 * 2;                    // Ucat3 chunk, KU3/64 atoms
  static constexpr int U_BYTES = U1_BYTES > U2_BYTES ? U1_BYTES : U2_BYTES;
  static constexpr int STAGE = X_BYTES + U_BYTES;
  static constexpr int S = RP == 0 ? 8 : (RP <= 32 ? 4 : (RP <= 48 ? 3 : 2));
  static constexpr int AREC_BYTES = kBM * KU3 * 2;
  static constexpr int XAM_BYTES = 2 * 2 * 2 * kBM * 4;  // partial absmax: [use & 1][parity][half][row]
  static constexpr int NBAR = 2 * S + 3 + 2 * kNumRec + 8;
  static constexpr int SMEM = 1024 + S * STAGE + AREC_BYTES + XAM_BYTES + NBAR * 8 + 16;
  static constexpr uint32_t TMEM_COLS = 512;  // proj at col 0 (2*RP <= 128), rec buffers at 128 + 64 b
  static_assert(SMEM <= 232448, "kernel (a) shared memory above the 227 KB per-CTA limit");
};

constexpr float kMagic = 12582912.0f;  // 1.5 * 2^23: adding it rounds to an integer (ties to even)
constexpr int kMagicBits = 0x4B400000;

// Nearest code in [-7, 7] to the exact quotient x / s, ties to even (s > 0, |x| <= amax).
// c = rint(x * (1/s)) is the nearest integer or its neighbour; the remainder e = x - c s is exact
// in float32 (c and the true answer differ by at most one), and |e| < s/2 exactly when c is right
// and not a tie.  The correction is taken with selects rather than a branch: a branch per value
// keeps the compiler from overlapping the 64 independent roundings of a group.  The result
// saturates at -+7, which only a bfloat16-subnormal scale (few significant bits) can need.
__device__ __forceinline__ int nearest_code(float x, float s, float inv, float hs) {
  const float t = fmaf(x, inv, kMagic);
  const float c = t - kMagic;
  const float e = fmaf(-c, s, x);
  const int ci = __float_as_int(t) - kMagicBits;
  const float ae = fabsf(e);
  // |e| > s/2: the neighbour on e's side; |e| == s/2 (a tie): the even one of the two
  const int adj = static_cast<int>(ae > hs) | (static_cast<int>(ae == hs) & ci & 1);
  return min(7, max(-7, ci + (e > 0.0f ? adj : -adj)));
}
// Approximate reciprocal (the hardware's single-instruction estimate).  It only seeds the
// rounding in nearest_code, whose exact remainder test corrects a seed that is off by one.
__device__ __forceinline__ float rcp_approx(float x) {
  float r;
  asm("rcp.approx.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}

// s_x = RN_bf16(amax / 7) of the exact quotient, ties to even: the quotient rounded toward zero to
// float32 with its last bit set when the division is inexact (round to odd; the remainder
// amax - 7 q is exact), then rounded to the nearest bfloat16.  Rounding to odd first and to nearest
// after is exact rounding because 24 >= 8 + 2.
__device__ __forceinline__ float bf16_scale_div7(float amax) {
  const float q = __fdiv_rz(amax, 7.0f);
  const float rem = fmaf(-q, 7.0f, amax);
  const float qo = __uint_as_float(__float_as_uint(q) | (rem != 0.0f ? 1u : 0u));
  return __bfloat162float(__float2bfloat16_rn(qo));
}

// ---- packed float32 pairs: two IEEE round-to-nearest operations per instruction, each rounded
// exactly as its scalar form.
__device__ __forceinline__ uint64_t f2(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ void f2_split(uint64_t v, float& lo, float& hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ uint64_t fma_f32x2(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ uint64_t add_f32x2(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ uint64_t sub_f32x2(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}

// Eight values -> a candidate OB4 word, and the largest |x - c s| over them folded into emax.
// t = RN(x * inv + (1.5 * 2^23 + 8)) is an integer-valued float whose low four bits are c + 8 for
// the candidate code c = t - (1.5 * 2^23 + 8) (|c| <= 8), so the nibbles come straight from t's
// bits.  The candidate is the nearest code exactly when |x - c s| < s/2: a wrong neighbour and a
// tie both give |x - c s| >= s/2 (a rounded remainder keeps that order, s/2 being a float), which
// is the caller's test for the whole group.
constexpr float kMagic8 = 12582920.0f;
__device__ __forceinline__ uint32_t codes8_fast(const float* x, uint64_t inv2, uint64_t nsc2, float& emax) {
  const uint64_t m2 = f2(kMagic8, kMagic8), nm2 = f2(-kMagic8, -kMagic8);
  uint32_t t[8];
#pragma unroll
  for (int u = 0; u < 8; u += 2) {
    const uint64_t x2 = f2(x[u], x[u + 1]);
    const uint64_t t2 = fma_f32x2(x2, inv2, m2);
    const uint64_t e2 = fma_f32x2(add_f32x2(t2, nm2), nsc2, x2);
    float tl, th, el, eh;
    f2_split(t2, tl, th);
    f2_split(e2, el, eh);
    t[u] = __float_as_uint(tl);
    t[u + 1] = __float_as_uint(th);
    emax = fmaxf(emax, fmaxf(fabsf(el), fabsf(eh)));
  }
  // OB4: the code of k = 2p in bits 4p.., the code of k = 2p + 1 in bits 16 + 4p..
  uint32_t q[4];
#pragma unroll
  for (int p = 0; p < 4; ++p) q[p] = __byte_perm(t[2 * p], t[2 * p + 1], 0x5410) & 0x000F000Fu;
  return q[0] | (q[1] << 4) | (q[2] << 8) | (q[3] << 12);
}

// The codes of a group with the exact test per value (nearest_code): the path for a group whose
// fast candidates failed the remainder test, and for a zero or tiny scale.
template <int GS>
__device__ __forceinline__ void codes_exact(const float* xp, uint32_t* words, float sc) {
  // Codes are invariant under a common power-of-two scaling of the values and the scale (exact
  // in float32), which keeps 1/s finite for the rare group whose scale is tiny.
  const float k = (sc < 7.8886091e-31f) ? 1.2676506e30f : 1.0f;  // 2^-100, 2^100
  const float scs = sc * k;
  const float inv = sc > 0.0f ? rcp_approx(scs) : 0.0f;
  const float hs = 0.5f * scs;
#pragma unroll
  for (int w = 0; w < GS / 8; ++w) {
    int c[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) c[u] = nearest_code(xp[8 * w + u] * k, scs, inv, hs);
    words[w] = ob4_word(c);
  }
}

// The largest |x| of GS values, formed as a tree (max is exact, so the order does not matter),
// which keeps the dependency chain short.
template <int GS>
__device__ __forceinline__ float absmax(const float* xp) {
  float mx[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) mx[j] = fabsf(xp[j]);
#pragma unroll
  for (int i = 8; i < GS; ++i) mx[i & 7] = fmaxf(mx[i & 7], fabsf(xp[i]));
#pragma unroll
  for (int w = 4; w >= 1; w >>= 1)
#pragma unroll
    for (int j = 0; j < w; ++j) mx[j] = fmaxf(mx[j], mx[j + w]);
  return mx[0];
}

// GS values -> GS/8 OB4 words of their nearest codes under the scale sc.  The codes take the fast
// candidates of codes8_fast; values whose candidates fail the remainder test (a near-tie, rare),
// and a zero or tiny scale, are redone by the exact per-value test.
template <int GS>
__device__ __forceinline__ void codes_for_scale(const float* xp, uint32_t* words, float sc) {
  bool exact = !(sc >= 7.8886091e-31f);  // zero or tiny scale
  if (!exact) {
    const float inv = rcp_approx(sc);
    const uint64_t inv2 = f2(inv, inv), nsc2 = f2(-sc, -sc);
    float em[2] = {0.0f, 0.0f};
#pragma unroll
    for (int w = 0; w < GS / 8; ++w) words[w] = codes8_fast(xp + 8 * w, inv2, nsc2, em[w & 1]);
    exact = fmaxf(em[0], em[1]) >= 0.5f * sc;
  }
  if (exact) codes_exact<GS>(xp, words, sc);
}

// One group of GS remainder values -> scale and GS/8 OB4 words of codes.
template <int GS>
__device__ __forceinline__ void quantize_group(const float* xp, uint32_t* words, __nv_bfloat16* scale_out) {
  const float sc = bf16_scale_div7(absmax<GS>(xp));
  codes_for_scale<GS>(xp, words, sc);
  *scale_out = __float2bfloat16_rn(sc);  // exact: sc is a bfloat16 value
}

// ---- NVFP4 variant (App. B.1): one block of 16 remainder values -> E4M3 scale and E2M1 codes.
//   s = RN_e4m3(RN_f32(amax / 6)) (saturating at 448),  code = RN_e2m1(RN_f32(x / s)) (saturating
//   at 6; s == 0 gives zero codes; a result of magnitude zero is stored as code 0).
// The conversions are the hardware's round-to-nearest-even cvt forms; each is given the same
// value twice so that the result does not depend on which half of the pair a value lands in.
__device__ __forceinline__ uint32_t cvt_e4m3(float t) {
  uint16_t v;
  asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %1;" : "=h"(v) : "f"(t));
  return v & 0xFFu;
}
__device__ __forceinline__ float e4m3_value(uint32_t b) {
  const uint16_t pair = static_cast<uint16_t>(b | (b << 8));
  uint32_t h2;
  asm("cvt.rn.f16x2.e4m3x2 %0, %1;" : "=r"(h2) : "h"(pair));
  return __half2float(__ushort_as_half(static_cast<unsigned short>(h2 & 0xFFFFu)));
}
__device__ __forceinline__ uint32_t cvt_e2m1(float u) {
  uint32_t v;
  asm("{.reg .b8 t;\ncvt.rn.satfinite.e2m1x2.f32 t, %1, %1;\ncvt.u32.u8 %0, t;}" : "=r"(v) : "f"(u));
  return v & 0xFu;
}
// Two values -> their E2M1 codes in one byte, the first in the low nibble (cvt puts its first
// source operand in the upper half of the destination).
__device__ __forceinline__ uint32_t cvt_e2m1x2(float lo, float hi) {
  uint32_t v;
  asm("{.reg .b8 t;\ncvt.rn.satfinite.e2m1x2.f32 t, %1, %2;\ncvt.u32.u8 %0, t;}" : "=r"(v) : "f"(hi), "f"(lo));
  return v;
}
// 16 values -> two words of codes (k order, four bits each, low nibble first) and the scale byte.
// The codes are RN_e2m1 of the float32 quotient RN_f32(x / s).  The fast path rounds q = x * r
// (r the approximate reciprocal of s: |q - RN_f32(x / s)| < 2^-21 |q|) bracketed by the factors
// (1 -+ 2^-19): when both ends round to the same code, so does every value between them, the
// float32 quotient included.  A block with an end pair that differs (a quotient within 2^-19 of
// an E2M1 midpoint, rare) is recomputed with the correctly rounded division.
__device__ __forceinline__ uint32_t quantize_block_nvfp4(const float* x, uint32_t* w2) {
  float mx[4];
#pragma unroll
  for (int j = 0; j < 4; ++j) mx[j] = fmaxf(fmaxf(fabsf(x[j]), fabsf(x[j + 4])), fmaxf(fabsf(x[j + 8]), fabsf(x[j + 12])));
  const float amax = fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3]));
  const uint32_t sb = cvt_e4m3(__fdiv_rn(amax, 6.0f));
  const float sc = e4m3_value(sb);
  const float r = sc > 0.0f ? rcp_approx(sc) : 0.0f;
  constexpr float kDn = 1.0f - 1.0f / 524288.0f, kUp = 1.0f + 1.0f / 524288.0f;  // 1 -+ 2^-19
  uint32_t w[2] = {0u, 0u};
  bool near_mid = false;
#pragma unroll
  for (int h = 0; h < 2; ++h)
#pragma unroll
    for (int i = 0; i < 8; i += 2) {
      const float q0 = x[8 * h + i] * r, q1 = x[8 * h + i + 1] * r;
      const uint32_t lo = cvt_e2m1x2(q0 * kDn, q1 * kDn), hi = cvt_e2m1x2(q0 * kUp, q1 * kUp);
      near_mid |= lo != hi;
      w[h] |= lo << (4 * i);
    }
  if (near_mid) {
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      w[h] = 0u;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const float u = sc > 0.0f ? __fdiv_rn(x[8 * h + i], sc) : 0.0f;
        w[h] |= cvt_e2m1(u) << (4 * i);
      }
    }
  }
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    // a code whose magnitude bits are zero loses its sign bit
    const uint32_t nz = ((w[h] & 0x77777777u) + 0x77777777u) & 0x88888888u;
    w2[h] = w[h] & (0x77777777u | nz);
  }
  return sb;
}

template <int RP, bool NV>
__global__ void __launch_bounds__(kActThreads, 1)
    actquant_kernel(const __grid_constant__ CUtensorMap x_map, const __grid_constant__ CUtensorMap ut_map,
                    const __grid_constant__ CUtensorMap u3_map, const ActArgs a) {
  using Cfg = ActCfg<RP>;
  constexpr int S = Cfg::S;
  extern __shared__ uint8_t smem_raw[];
  pdl_launch_dependents();
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* stages = smem;
  uint8_t* arec = stages + S * Cfg::STAGE;
  float* xam = reinterpret_cast<float*>(arec + Cfg::AREC_BYTES);
  uint64_t* bars = reinterpret_cast<uint64_t*>(arec + Cfg::AREC_BYTES + Cfg::XAM_BYTES);
  uint64_t* full = bars;
  uint64_t* empty = bars + S;
  uint64_t* proj_done = bars + 2 * S;
  uint64_t* arec_ready = proj_done + 1;
  uint64_t* drain = proj_done + 2;
  uint64_t* tfull = proj_done + 3;
  uint64_t* tempty = tfull + kNumRec;
  uint64_t* xch = tempty + kNumRec;  // [parity * 4 + quadrant]: the two halves' partial absmax are in
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + Cfg::NBAR);
  int* abort_flag = reinterpret_cast<int*>(tmem_slot + 1);

  const uint32_t wid = warp_id(), lane = lane_id();
  const int C = a.C;
  const uint32_t rank = (RP > 0 && C > 1) ? cluster_ctarank() : 0u;
  const int cta_k = (RP > 0) ? static_cast<int>(rank) : static_cast<int>(blockIdx.x);
  const int k0 = cta_k * a.Kc;
  const int m0 = blockIdx.y * kBM;
  const int nch = a.Kc / kChunk;
  const int pass1 = RP > 0 ? nch : 0;  // pass-1 iterations before pass 2 in the ring order

  if (threadIdx.x == 0) {
    for (int i = 0; i < S; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 8);  // pass 2: the eight warps of one chunk parity; pass 1: the MMA commit + 7
    }
    mbar_init(proj_done, 1);
    mbar_init(arec_ready, 8);   // epilogue warps
    mbar_init(drain, 1);
    for (int i = 0; i < kNumRec; ++i) {
      mbar_init(&tfull[i], 1);
      mbar_init(&tempty[i], 8);   // the eight warps of one chunk parity
    }
    for (int i = 0; i < 8; ++i) mbar_init(&xch[i], 2);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (RP > 0 && wid == 1) {
    tmem_alloc(tmem_slot, Cfg::TMEM_COLS);
    tmem_relinquish();
  }
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = (RP > 0) ? *tmem_slot : 0u;
  const WaitCtl wc{abort_flag, a.err, globaltimer_ns() + a.timeout_ns};
  pdl_wait();  // every global access of this kernel comes after the previous kernel's

  auto stage_x = [&](int s) { return stages + s * Cfg::STAGE; };
  auto stage_u = [&](int s) { return stages + s * Cfg::STAGE + Cfg::X_BYTES; };

  if (wid == 0) {
    // ------------------------------------------------------------- TMA producer
    int it = 0, issued2 = 0;
    bool ok = true;
    auto produce = [&](bool first_pass, int c) {
      const int s = it % S;
      if (ok && it >= S) ok = mbar_wait_inline(&empty[s], ((it / S) & 1) ^ 1, wc);
      if (ok && elect_one()) {
        const uint32_t bytes = Cfg::X_BYTES + (first_pass ? Cfg::U1_BYTES : (RP > 0 ? Cfg::U2_BYTES : 0));
        mbar_arrive_expect_tx(&full[s], bytes);
        tma_load_2d(stage_x(s), &x_map, &full[s], k0 + c * kChunk, m0);
        if (first_pass) {
          tma_load_2d(stage_u(s), &ut_map, &full[s], k0 + c * kChunk, 0);
        } else if (RP > 0) {
          for (int q = 0; q < Cfg::KU3 / 64; ++q)
            tma_load_2d(stage_u(s) + q * 8192, &u3_map, &full[s], q * 64, k0 + c * kChunk);
        }
      }
      __syncwarp();
      ++it;
    };
    // The whole warp walks the ring (warp-uniform state); one elected lane issues each copy.
    if (elect_one()) tma_prefetch_desc(&x_map);
    __syncwarp();
    for (int c = 0; c < pass1; ++c) produce(true, c);
    for (; issued2 < nch && issued2 < S; ++issued2) produce(false, issued2);
    if (RP > 0) cluster_sync();
    for (; issued2 < nch; ++issued2) produce(false, issued2);
    // Let every load issued into the ring land before the CTA can exit.
    int never = 0;
    const WaitCtl dc{&never, a.err, globaltimer_ns() + a.timeout_ns};
    for (int j = (it > S ? it - S : 0); j < it; ++j) mbar_wait_inline(&full[j % S], (j / S) & 1, dc);
  } else if (wid == 1) {
    // ------------------------------------------------------------- MMA issuer
    if constexpr (RP > 0) {
      // The whole warp walks both passes (warp-uniform state); one elected lane issues.
      bool ok = true;
      {
        constexpr uint32_t idesc_proj = idesc_bf16(kBM, 2 * RP);
        for (int c = 0; c < nch && ok; ++c) {
          const int s = c % S;
          ok = mbar_wait_inline(&full[s], (c / S) & 1, wc);
          if (!ok) break;
          tc_fence_after();
          const uint32_t xa = smem_u32(stage_x(s)), ua = smem_u32(stage_u(s));
          if (elect_one()) {
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
              mma_f16(tmem, smem_desc(xa + kk * 32, 16, 1024, kSw128), smem_desc(ua + kk * 32, 16, 1024, kSw128),
                      idesc_proj, (c | kk) != 0);
            // the stage frees when these MMAs complete (the commit is the last of eight arrivals)
#pragma unroll
            for (int i = 0; i < 7; ++i) mbar_arrive(&empty[s]);
            mma_commit(&empty[s]);
          }
          __syncwarp();
        }
        if (elect_one()) mma_commit(proj_done);
      }
      __syncwarp();
      cluster_sync();
      {
        if (ok) ok = mbar_wait_inline(arec_ready, 0, wc);
        tc_fence_after();
        constexpr uint32_t idesc_rec = idesc_bf16(kBM, kChunk);
        const uint32_t ar = smem_u32(arec);
        for (int c = 0; c < nch && ok; ++c) {
          const int it = pass1 + c, s = it % S, b = c % kNumRec;
          ok = mbar_wait_inline(&full[s], (it / S) & 1, wc);
          if (ok && c >= kNumRec) ok = mbar_wait_inline(&tempty[b], ((c / kNumRec) & 1) ^ 1, wc);
          if (!ok) break;
          tc_fence_after();
          const uint32_t ua = smem_u32(stage_u(s));
          if (elect_one()) {
#pragma unroll
            for (int kk = 0; kk < 3 * RP / 16; ++kk) {
              const int q = kk >> 2, off = (kk & 3) * 32;
              mma_f16(tmem + 128 + 64 * b, smem_desc(ar + q * 16384 + off, 16, 1024, kSw128),
                      smem_desc(ua + q * 8192 + off, 16, 1024, kSw128), idesc_rec, kk != 0);
            }
            mma_commit(&tfull[b]);
          }
          __syncwarp();
        }
        // Make sure every MMA of this CTA has completed before TMEM is released.
        if (elect_one()) mma_commit(drain);
        __syncwarp();
        int never = 0;
        const WaitCtl dc{&never, a.err, globaltimer_ns() + a.timeout_ns};
        mbar_wait_inline(drain, 0, dc);
      }
      __syncwarp();
    }
  } else {
    // ------------------------------------------------------------- epilogue (thread = row)
    // Warp 2 + e (e = 0..15): TMEM quadrant wid & 3, chunk parity (e >> 2) & 1, and half e >> 3 of
    // each chunk's 64 columns in pass 2; the eight warps of half 0 also form p (pass 1's epilogue).
    const int quad = wid & 3;
    const int par = ((static_cast<int>(wid) - 2) >> 2) & 1;  // 0: even chunks, 1: odd chunks
    const int half = (static_cast<int>(wid) - 2) >> 3;
    const int row = quad * 32 + static_cast<int>(lane);
    const int m = m0 + row;
    const uint32_t tlane = tmem + (static_cast<uint32_t>(quad * 32) << 16);
    bool ok = true;

    if constexpr (!NV && RP > 0) {
      // The GEMM's float16 weights (expand_w16), a grid-stride share per epilogue thread, while
      // pass 1 waits on HBM.  The stream's previous GEMM, which read the region, has completed
      // (the wait at the top), and the GEMM of this call reads it only after this kernel completes.
      if (a.w.w16 != nullptr) {
        constexpr int kEpi = kActThreads - 64;
        expand_w16<8>(a.w, static_cast<int>(blockIdx.y * gridDim.x + blockIdx.x) * kEpi + static_cast<int>(threadIdx.x) - 64,
                      static_cast<int>(gridDim.x * gridDim.y) * kEpi);
      }
    }

    if constexpr (RP > 0) {
     if (half == 1) {
      cluster_sync();  // the exchange barrier of the projection below
     } else {
      constexpr int HR = RP / 2;  // projection columns handled by this thread (half of them)
      const int j0 = par * HR;
      // -- partial projection of this CTA's K slice: hi part + lo part, columns [j0, j0 + HR)
      ok = mbar_wait_inline(proj_done, 0, wc);
      tc_fence_after();
      float pp[HR];
#pragma unroll
      for (int q = 0; q < HR / 8; ++q) {
        uint32_t vh[8], vl[8];
        asm volatile(
            "tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];"
            : "=r"(vh[0]), "=r"(vh[1]), "=r"(vh[2]), "=r"(vh[3]), "=r"(vh[4]), "=r"(vh[5]), "=r"(vh[6]), "=r"(vh[7])
            : "r"(tlane + j0 + q * 8)
            : "memory");
        asm volatile(
            "tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];"
            : "=r"(vl[0]), "=r"(vl[1]), "=r"(vl[2]), "=r"(vl[3]), "=r"(vl[4]), "=r"(vl[5]), "=r"(vl[6]), "=r"(vl[7])
            : "r"(tlane + RP + j0 + q * 8)
            : "memory");
        tmem_ld_wait();
#pragma unroll
        for (int i = 0; i < 8; ++i) pp[q * 8 + i] = __uint_as_float(vh[i]) + __uint_as_float(vl[i]);
      }
      // -- the partial goes to the float32 scratch (slice `rank`, row m0 + row, columns
      //    [j0, j0 + HR)); the cluster barrier's release / acquire orders it before the reads below
      {
        float4* dst = reinterpret_cast<float4*>(a.part + (static_cast<size_t>(rank) * a.M_pad + m0 + row) * RP + j0);
#pragma unroll
        for (int j = 0; j < HR / 4; ++j) dst[j] = make_float4(pp[4 * j], pp[4 * j + 1], pp[4 * j + 2], pp[4 * j + 3]);
      }
      cluster_sync();  // every partial of the cluster is in the scratch
      // -- p for this thread's row and columns: the C partials summed in rank order (every CTA of
      //    the cluster forms the same p), the loads of QL slices in flight at a time
      float p[HR];
      {
        constexpr int QL = HR <= 16 ? 64 / HR : 2;  // at most 16 float4 loads per round
        const float* src = a.part + static_cast<size_t>(m0 + row) * RP + j0;
        const size_t slice = static_cast<size_t>(a.M_pad) * RP;
#pragma unroll
        for (int j = 0; j < HR; ++j) p[j] = 0.0f;
        for (int q0 = 0; q0 < C; q0 += QL) {
          float4 v[QL][HR / 4];
#pragma unroll
          for (int i = 0; i < QL; ++i)
#pragma unroll
            for (int j = 0; j < HR / 4; ++j)
              v[i][j] = q0 + i < C ? reinterpret_cast<const float4*>(src + (q0 + i) * slice)[j] : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
          for (int i = 0; i < QL; ++i) {
            if (q0 + i >= C) break;
#pragma unroll
            for (int j = 0; j < HR / 4; ++j) {
              // rank 0's slice starts the sum exactly (0 + x == x), then the others in order
              p[4 * j] += v[i][j].x;
              p[4 * j + 1] += v[i][j].y;
              p[4 * j + 2] += v[i][j].z;
              p[4 * j + 3] += v[i][j].w;
            }
          }
        }
      }
      // -- p_hat = RN_f16(p): each row written once, by the CTA whose rank owns its slice of rows
      if (row / (kBM / C) == static_cast<int>(rank) && m < a.M) {
#pragma unroll
        for (int j = 0; j < HR / 8; ++j) {
          uint32_t w[4];
#pragma unroll
          for (int t = 0; t < 4; ++t) {
            const __half2 h2 = __floats2half2_rn(p[8 * j + 2 * t], p[8 * j + 2 * t + 1]);
            w[t] = *reinterpret_cast<const uint32_t*>(&h2);
          }
          reinterpret_cast<uint4*>(a.phat + static_cast<size_t>(m) * RP + j0)[j] = make_uint4(w[0], w[1], w[2], w[3]);
        }
      }
      // -- A operand of the reconstruction: [p_hi | p_hi | p_lo | 0], 128-byte swizzle.
      //    This thread writes its columns j0..j0+HR-1 of each segment (8 bf16 = one 16-byte chunk).
      __nv_bfloat16 hi[HR], lo[HR];
#pragma unroll
      for (int j = 0; j < HR; ++j) {
        hi[j] = __float2bfloat16_rn(p[j]);
        lo[j] = __float2bfloat16_rn(p[j] - __bfloat162float(hi[j]));
      }
      auto put8 = [&](int col, const __nv_bfloat16* v) {  // col: multiple of 8
        uint32_t w[4];
#pragma unroll
        for (int t = 0; t < 4; ++t)
          w[t] = static_cast<uint32_t>(__bfloat16_as_ushort(v[2 * t])) |
                 (static_cast<uint32_t>(__bfloat16_as_ushort(v[2 * t + 1])) << 16);
        const int q = col >> 6, j = (col & 63) >> 3;
        *reinterpret_cast<uint4*>(arec + q * 16384 + row * 128 + ((j ^ (row & 7)) << 4)) =
            make_uint4(w[0], w[1], w[2], w[3]);
      };
#pragma unroll
      for (int c8 = 0; c8 < HR / 8; ++c8) {
        put8(j0 + 8 * c8, hi + 8 * c8);
        put8(RP + j0 + 8 * c8, hi + 8 * c8);
        put8(2 * RP + j0 + 8 * c8, lo + 8 * c8);
      }
      if (par == 1) {  // zero padding columns [3 RP, KU3)
        const __nv_bfloat16 z[8] = {};
        for (int col = 3 * RP; col < Cfg::KU3; col += 8) put8(col, z);
      }
      fence_proxy_async_smem();
      warp_arrive(arec_ready);
     }
    }

    // -- pass 2: remainder and quantization; this warp takes, of each chunk of its parity, the 32
    //    columns of its half for the 32 rows of its quadrant
    for (int c = par, use = 0; c < nch; c += 2, ++use) {
      const int it = pass1 + c, s = it % S;
      float xp[32];
      if constexpr (RP > 0) {
        const int b = c % kNumRec;
        if (ok) ok = mbar_wait_inline(&tfull[b], (c / kNumRec) & 1, wc);
        tc_fence_after();
        uint32_t r0[32];
        tmem_ld32(tlane + 128 + 64 * b + 32 * half, r0);
        tmem_ld_wait();
        tc_fence_before();
        warp_arrive(&tempty[b]);
#pragma unroll
        for (int i = 0; i < 32; ++i) xp[i] = __uint_as_float(r0[i]);
      }
      if (ok) ok = mbar_wait_inline(&full[s], (it / S) & 1, wc);
      const uint8_t* xs = stage_x(s) + row * 128;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const uint4 v = *reinterpret_cast<const uint4*>(xs + (((4 * half + j) ^ (row & 7)) << 4));
        const uint32_t wv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          const float lo_f = __uint_as_float(wv[t] << 16);
          const float hi_f = __uint_as_float(wv[t] & 0xFFFF0000u);
          if constexpr (RP > 0) {
            const uint64_t d = sub_f32x2(f2(lo_f, hi_f), f2(xp[8 * j + 2 * t], xp[8 * j + 2 * t + 1]));
            f2_split(d, xp[8 * j + 2 * t], xp[8 * j + 2 * t + 1]);
          } else {
            xp[8 * j + 2 * t] = lo_f;
            xp[8 * j + 2 * t + 1] = hi_f;
          }
        }
      }
      // The stage goes back to the TMA producer: order these generic-proxy reads before the
      // async-proxy write that will refill it; each of the eight warps that read it releases it.
      fence_proxy_async_smem();
      warp_arrive(&empty[s]);
      const bool live = ok && m < a.M;
      const int kc = k0 + c * kChunk + 32 * half;  // this half's first column
      if (a.dump) {
        if (live) {
          float4* d = reinterpret_cast<float4*>(a.dump + static_cast<size_t>(m) * a.K + kc);
#pragma unroll
          for (int i = 0; i < 8; ++i) d[i] = make_float4(xp[4 * i], xp[4 * i + 1], xp[4 * i + 2], xp[4 * i + 3]);
        }
        if (a.resid_only) continue;
      }
      uint8_t* crow = a.codes + static_cast<size_t>(m) * (a.K / 2) + kc / 2;
      if constexpr (NV) {
        if (!live) continue;
        uint32_t w[4];
        const uint32_t sf2 = quantize_block_nvfp4(xp, w) | (quantize_block_nvfp4(xp + 16, w + 2) << 8);
        *reinterpret_cast<uint4*>(crow) = make_uint4(w[0], w[1], w[2], w[3]);
        const int mr = m % kBM;
        *reinterpret_cast<uint16_t*>(a.sf + (static_cast<size_t>(m / kBM) * (a.K / 64) + (kc - 32 * half) / 64) * kSfAtom +
                                     (mr % 32) * 16 + (mr / 32) * 4 + 2 * half) = static_cast<uint16_t>(sf2);
        continue;
      }
      uint32_t words[4];
      if (a.G == 64) {
        // The group spans both halves: the two warps of this quadrant and parity swap their
        // partial absmax through shared memory (double-buffered by use, one pairwise barrier).
        float* slot = xam + ((use & 1) * 4 + par * 2) * kBM;
        const float am = absmax<32>(xp);
        slot[half * kBM + row] = am;
        warp_arrive(&xch[par * 4 + quad]);
        if (!mbar_wait_inline(&xch[par * 4 + quad], use & 1, wc)) ok = false;
        const float sc = bf16_scale_div7(fmaxf(am, slot[(half ^ 1) * kBM + row]));
        codes_for_scale<32>(xp, words, sc);
        if (half == 0 && live) a.scales[static_cast<size_t>((kc - 32 * half) / 64) * a.M_pad + m] = __float2bfloat16_rn(sc);
      } else {
        const float sc = bf16_scale_div7(absmax<32>(xp));
        codes_for_scale<32>(xp, words, sc);
        if (live) a.scales[static_cast<size_t>(kc / 32) * a.M_pad + m] = __float2bfloat16_rn(sc);
      }
      if (live) *reinterpret_cast<uint4*>(crow) = make_uint4(words[0], words[1], words[2], words[3]);
    }
  }

  __syncthreads();
  if (RP > 0 && wid == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, Cfg::TMEM_COLS);
  }
}

// Test support: the quantizers above applied to caller-given float32 rows (one thread per row
// and 64-value chunk), so that their rounding can be checked on chosen values.
template <bool NV>
__global__ void __launch_bounds__(128) debug_quantize_kernel(const float* R, int M, int K, int G, uint8_t* codes,
                                                               void* scales) {
  const int nch = K / kChunk;
  const long long idx = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (idx >= static_cast<long long>(M) * nch) return;
  const int m = static_cast<int>(idx / nch), c = static_cast<int>(idx % nch);
  float xp[kChunk];
  const float4* src = reinterpret_cast<const float4*>(R + static_cast<size_t>(m) * K + static_cast<size_t>(c) * kChunk);
#pragma unroll
  for (int i = 0; i < kChunk / 4; ++i) {
    const float4 v = src[i];
    xp[4 * i] = v.x;
    xp[4 * i + 1] = v.y;
    xp[4 * i + 2] = v.z;
    xp[4 * i + 3] = v.w;
  }
  if constexpr (NV) {
    uint32_t w[8];
    uint8_t* sf = static_cast<uint8_t*>(scales) + static_cast<size_t>(m) * (K / kFp4Block) + c * (kChunk / kFp4Block);
#pragma unroll
    for (int b = 0; b < 4; ++b) sf[b] = static_cast<uint8_t>(quantize_block_nvfp4(xp + 16 * b, w + 2 * b));
    uint4* dst = reinterpret_cast<uint4*>(codes + static_cast<size_t>(m) * (K / 2) + c * (kChunk / 2));
    dst[0] = make_uint4(w[0], w[1], w[2], w[3]);
    dst[1] = make_uint4(w[4], w[5], w[6], w[7]);
  } else {
    uint32_t words[8];
    __nv_bfloat16* sc = static_cast<__nv_bfloat16*>(scales) + static_cast<size_t>(m) * (K / G) + c * (kChunk / G);
    if (G == 64) {
      quantize_group<64>(xp, words, sc);
    } else {
      quantize_group<32>(xp, words, sc);
      quantize_group<32>(xp + 32, words + 4, sc + 1);
    }
    uint4* dst = reinterpret_cast<uint4*>(codes + static_cast<size_t>(m) * (K / 2) + c * (kChunk / 2));
    dst[0] = make_uint4(words[0], words[1], words[2], words[3]);
    dst[1] = make_uint4(words[4], words[5], words[6], words[7]);
  }
}

// ---- run-time smoothing and block Hadamard rotation (Sec. 3 Eq. (pair); App. B.1) ----------
//
//   x~_perp = H diag(s)^-1 v,  v = x (r = 0) or v = x - diag(s) H U p (r > 0, from kernel (a))
//
// then the same quantizers as kernel (a).  One warp takes one token row and one Hadamard block of
// B = 256 NSUB channels; lane l holds channels 256 c + 8 l .. + 7 of sub-block c.  The fast
// Walsh-Hadamard butterflies run at spans 1, 2, 4 inside a lane, 8 .. 128 across lanes
// (shuffles) and 256, 512 across the lane's sub-blocks.  The normalisation 1/sqrt(B) is folded
// into the per-channel factor applied first, RN_f32(1 / (sqrt(B) s_k)).  A quantization group
// (32 or 64 channels) is 4 or 8 neighbouring lanes, an NVFP4 block (16) two.
// Where the lane quantizers below write: the activation workspace of one handle.
struct QuantOut {
  int K, G, M_pad;
  uint8_t* codes;
  uint8_t* sf;
  __nv_bfloat16* scales;
};

struct RotArgs {
  int M, K;
  const float* inv_s;  // [K]: RN_f32(1 / (sqrt(B) s_k))
  float* dump;
  QuantOut q;
};

__device__ __forceinline__ void load8(const __nv_bfloat16* p, float* v) {
  const uint4 u = *reinterpret_cast<const uint4*>(p);
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
  for (int t = 0; t < 4; ++t) {
    v[2 * t] = __uint_as_float(w[t] << 16);
    v[2 * t + 1] = __uint_as_float(w[t] & 0xFFFF0000u);
  }
}
__device__ __forceinline__ void load8(const float* p, float* v) {
  const float4 a = reinterpret_cast<const float4*>(p)[0], b = reinterpret_cast<const float4*>(p)[1];
  v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
  v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}

// The lane's 8 values of an NVFP4 block half: one word of E2M1 codes (low nibble first), with the
// same bracketed fast path and exact fallback as quantize_block_nvfp4.
__device__ __forceinline__ uint32_t codes8_nvfp4(const float* x, float sc, float r) {
  constexpr float kDn = 1.0f - 1.0f / 524288.0f, kUp = 1.0f + 1.0f / 524288.0f;
  uint32_t w = 0u;
  bool near_mid = false;
#pragma unroll
  for (int i = 0; i < 8; i += 2) {
    const float q0 = x[i] * r, q1 = x[i + 1] * r;
    const uint32_t lo = cvt_e2m1x2(q0 * kDn, q1 * kDn), hi = cvt_e2m1x2(q0 * kUp, q1 * kUp);
    near_mid |= lo != hi;
    w |= lo << (4 * i);
  }
  if (near_mid) {
    w = 0u;
#pragma unroll
    for (int i = 0; i < 8; ++i) w |= cvt_e2m1(sc > 0.0f ? __fdiv_rn(x[i], sc) : 0.0f) << (4 * i);
  }
  const uint32_t nz = ((w & 0x77777777u) + 0x77777777u) & 0x88888888u;
  return w & (0x77777777u | nz);
}

// The quantizers of kernel (a) on a warp-wide layout: each lane holds 8 consecutive remainder
// values x (channels k .. k+7 of token row m, k a multiple of 8) and the lanes of one quantization
// group (INT4: G/8 lanes; NVFP4: 2 lanes per block of 16) are neighbours.  Writes the codes (INT4:
// the lane's OB4 word) and, from the group's first lane, its scale.  The scale and the codes are
// those of quantize_group / quantize_block_nvfp4, bit for bit.
template <bool NV>
__device__ __forceinline__ void quantize8_lanes(const float* x, int lane, int m, int k, const QuantOut& o) {
  constexpr unsigned kAll = 0xFFFFFFFFu;
  float am = 0.0f;
#pragma unroll
  for (int i = 0; i < 8; ++i) am = fmaxf(am, fabsf(x[i]));
  if constexpr (NV) {
    am = fmaxf(am, __shfl_xor_sync(kAll, am, 1));
    const uint32_t sb = cvt_e4m3(__fdiv_rn(am, 6.0f));
    const float sc = e4m3_value(sb);
    const uint32_t w = codes8_nvfp4(x, sc, sc > 0.0f ? rcp_approx(sc) : 0.0f);
    *reinterpret_cast<uint32_t*>(o.codes + static_cast<size_t>(m) * (o.K / 2) + k / 2) = w;
    if ((lane & 1) == 0) {
      const int mr = m % kBM;
      o.sf[(static_cast<size_t>(m / kBM) * (o.K / 64) + k / 64) * kSfAtom + (mr % 32) * 16 + (mr / 32) * 4 +
           (k % 64) / kFp4Block] = static_cast<uint8_t>(sb);
    }
  } else {
    am = fmaxf(am, __shfl_xor_sync(kAll, am, 1));
    am = fmaxf(am, __shfl_xor_sync(kAll, am, 2));
    if (o.G == 64) am = fmaxf(am, __shfl_xor_sync(kAll, am, 4));
    const float sc = bf16_scale_div7(am);
    uint32_t word = 0u;
    bool exact = !(sc >= 7.8886091e-31f);  // zero or tiny scale
    if (!exact) {
      const float inv = rcp_approx(sc);
      float em = 0.0f;
      word = codes8_fast(x, f2(inv, inv), f2(-sc, -sc), em);
      exact = em >= 0.5f * sc;
    }
    if (exact) codes_exact<8>(x, &word, sc);
    *reinterpret_cast<uint32_t*>(o.codes + static_cast<size_t>(m) * (o.K / 2) + k / 2) = word;
    if ((lane & (o.G / 8 - 1)) == 0) o.scales[static_cast<size_t>(k / o.G) * o.M_pad + m] = __float2bfloat16_rn(sc);
  }
}

template <typename TIn, int NSUB, bool NV>
__global__ void __launch_bounds__(256, 4) rotquant_kernel(const TIn* __restrict__ in, const RotArgs a) {
  pdl_launch_dependents();
  pdl_wait();
  const int lane = static_cast<int>(threadIdx.x & 31);
  // one warp per (token row, Hadamard block): many warps in flight, each with one block's work
  const int nblk = a.K / (256 * NSUB);
  const long long wg = static_cast<long long>(blockIdx.x) * 8 + (threadIdx.x >> 5);
  if (wg >= static_cast<long long>(a.M) * nblk) return;
  const int m = static_cast<int>(wg / nblk);
  const TIn* row = in + static_cast<size_t>(m) * a.K;
  constexpr unsigned kAll = 0xFFFFFFFFu;
  {
    const int kb = static_cast<int>(wg % nblk) * (256 * NSUB);
    float v[NSUB][8];
#pragma unroll
    for (int c = 0; c < NSUB; ++c) {
      const int k = kb + 256 * c + 8 * lane;
      float is[8];
      load8(row + k, v[c]);
      load8(a.inv_s + k, is);
#pragma unroll
      for (int i = 0; i < 8; ++i) v[c][i] *= is[i];
    }
#pragma unroll
    for (int h = 1; h < 8; h *= 2)
#pragma unroll
      for (int c = 0; c < NSUB; ++c)
#pragma unroll
        for (int i = 0; i < 8; ++i)
          if ((i & h) == 0) {
            const float x0 = v[c][i], x1 = v[c][i + h];
            v[c][i] = x0 + x1;
            v[c][i + h] = x0 - x1;
          }
#pragma unroll
    for (int x = 1; x < 32; x *= 2) {
      // lower lane: v + o; upper lane: o - v; both one exactly rounded fma with a +-1 factor
      const float sgn = (lane & x) ? -1.0f : 1.0f;
#pragma unroll
      for (int c = 0; c < NSUB; ++c)
#pragma unroll
        for (int i = 0; i < 8; ++i) v[c][i] = fmaf(v[c][i], sgn, __shfl_xor_sync(kAll, v[c][i], x));
    }
#pragma unroll
    for (int h = 1; h < NSUB; h *= 2)
#pragma unroll
      for (int c = 0; c < NSUB; ++c)
        if ((c & h) == 0)
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const float x0 = v[c][i], x1 = v[c + h][i];
            v[c][i] = x0 + x1;
            v[c + h][i] = x0 - x1;
          }
#pragma unroll
    for (int c = 0; c < NSUB; ++c) {
      const int k = kb + 256 * c + 8 * lane;
      float* x = v[c];
      if (a.dump) {
        float4* d = reinterpret_cast<float4*>(a.dump + static_cast<size_t>(m) * a.K + k);
        d[0] = make_float4(x[0], x[1], x[2], x[3]);
        d[1] = make_float4(x[4], x[5], x[6], x[7]);
      }
      quantize8_lanes<NV>(x, lane, m, k, a.q);
    }
  }
}

QuantOut quant_out(const Handle& h, const ActLayout& L, uint8_t* base) {
  QuantOut q;
  q.K = h.K;
  q.G = h.G;
  q.M_pad = L.M_pad;
  q.codes = base + L.codes_off;
  q.sf = base + L.scales_off;
  q.scales = reinterpret_cast<__nv_bfloat16*>(base + L.scales_off);
  return q;
}

template <typename TIn, bool NV>
cudaError_t launch_rotquant_t(const Handle& h, const TIn* in, const RotArgs& a, cudaStream_t s) {
  cudaLaunchConfig_t cfg = {};
  const long long warps = static_cast<long long>(a.M) * (a.K / h.hb);
  cfg.gridDim = dim3(static_cast<unsigned>((warps + 7) / 8), 1, 1);
  cfg.blockDim = dim3(256, 1, 1);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  switch (h.hb) {
    case 256: return cudaLaunchKernelEx(&cfg, rotquant_kernel<TIn, 1, NV>, in, a);
    case 512: return cudaLaunchKernelEx(&cfg, rotquant_kernel<TIn, 2, NV>, in, a);
    case 1024: return cudaLaunchKernelEx(&cfg, rotquant_kernel<TIn, 4, NV>, in, a);
    default: return cudaErrorInvalidValue;
  }
}

// ---- small-M activation path ------------------------------------------------------------------
//
// For a few token rows (the action-expert layers) the phases of kernel (a) -- TMA ring, tensor-core
// projection, cluster reduction, tensor-core reconstruction -- are mostly latency in series.  Here
// one CTA of four warps takes one token row on the CUDA cores, in float32:
//   p = x U        (per column, fma over the lane's channels in ascending order, then a fixed tree
//                   over the lanes and the four warps),
//   p_hat = RN_f16(p),
//   x_perp = x - p U^T  (per channel, fma over j ascending, then one subtraction),
// and the quantizers of kernel (a).  Lane l of warp w holds channels 256 c + 8 l .. + 7 of the
// 256-channel chunks c = w, w + 4, ...  The bases are the handle's float32 copies, transposed
// ([RP, K], zero rows beyond r), so that a warp reads 1 KB of one column per load.  For a rotated
// layer the bases are diag(s)^-1 H U and diag(s) H U (as for kernel (a)), and the remainder is
// rotated before it is quantized (the rotation kernel's transform, the cross-chunk spans of a
// Hadamard block through shared memory).
struct SmallArgs {
  int M, K;
  const float* up;  // [RP, K] projection basis
  const float* ur;  // [RP, K] reconstruction basis
  const float* inv_s;  // rotated layer: [K] RN_f32(1 / (sqrt(B) s_k)); the remainder is then rotated
  int hb;              // rotated layer: Hadamard block B (256, 512 or 1024)
  __half* phat;     // [M, RP]
  float* dump;      // optional [M, K]: x_perp
  QuantOut q;
};

template <int RP, bool NV, bool ROT>
__global__ void __launch_bounds__(128) smallq_kernel(const __nv_bfloat16* __restrict__ X, const SmallArgs a) {
  constexpr int RPS = RP > 0 ? RP : 1;
  constexpr int JB = RP <= 16 ? RPS : 8;  // basis columns loaded per batch
  __shared__ float red[4][RPS];
  __shared__ float4 xch[ROT ? 4 : 1][ROT ? 32 : 1][2];  // rotated layer: the four warps' chunks
  pdl_launch_dependents();
  pdl_wait();
  const int lane = static_cast<int>(threadIdx.x & 31), w = static_cast<int>(threadIdx.x >> 5);
  const int m = blockIdx.x;
  const __nv_bfloat16* row = X + static_cast<size_t>(m) * a.K;
  const int nc = a.K / 256;
  float p[RPS];
  if constexpr (RP > 0) {
    float pp[RP];
#pragma unroll
    for (int j = 0; j < RP; ++j) pp[j] = 0.0f;
    for (int c = w; c < nc; c += 4) {
      const int k = 256 * c + 8 * lane;
      float x[8];
      load8(row + k, x);
      // columns in batches of JB: all of a batch's loads are issued before its fmas
#pragma unroll
      for (int jb = 0; jb < RP; jb += JB) {
        float u[JB][8];
#pragma unroll
        for (int j = 0; j < JB; ++j) load8(a.up + static_cast<size_t>(jb + j) * a.K + k, u[j]);
#pragma unroll
        for (int j = 0; j < JB; ++j)
#pragma unroll
          for (int i = 0; i < 8; ++i) pp[jb + j] = fmaf(x[i], u[j][i], pp[jb + j]);
      }
    }
#pragma unroll
    for (int j = 0; j < RP; ++j)
#pragma unroll
      for (int off = 16; off >= 1; off >>= 1) pp[j] += __shfl_xor_sync(0xFFFFFFFFu, pp[j], off);
    if (lane == 0)
#pragma unroll
      for (int j = 0; j < RP; ++j) red[w][j] = pp[j];
    __syncthreads();
#pragma unroll
    for (int j = 0; j < RP; ++j) p[j] = (red[0][j] + red[1][j]) + (red[2][j] + red[3][j]);
    if (threadIdx.x < RP) {
      const int j = static_cast<int>(threadIdx.x);
      a.phat[static_cast<size_t>(m) * RP + j] = __float2half_rn((red[0][j] + red[1][j]) + (red[2][j] + red[3][j]));
    }
  }
  // A rotated layer walks the chunks in rounds of four (one per warp) so that the chunks of a
  // Hadamard block (B / 256 of them, aligned) are in the CTA at the same time.
  const int rounds = ROT ? (nc + 3) / 4 : 0;
  for (int c = w; ROT ? c < 4 * rounds : c < nc; c += 4) {
    const bool live = c < nc;
    const int k = 256 * (live ? c : 0) + 8 * lane;
    float x[8];
    load8(row + k, x);
    if constexpr (RP > 0) {
      float acc[8] = {0.0f, 0.0f, 0.0f, 0.0f, 0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
      for (int jb = 0; jb < RP; jb += JB) {
        float u[JB][8];
#pragma unroll
        for (int j = 0; j < JB; ++j) load8(a.ur + static_cast<size_t>(jb + j) * a.K + k, u[j]);
#pragma unroll
        for (int j = 0; j < JB; ++j)
#pragma unroll
          for (int i = 0; i < 8; ++i) acc[i] = fmaf(p[jb + j], u[j][i], acc[i]);
      }
#pragma unroll
      for (int i = 0; i < 8; ++i) x[i] -= acc[i];
    }
    if constexpr (ROT) {
      // x~_perp = H diag(s)^-1 (x - diag(s) H U p): the channel factor (1/sqrt(B) folded in), the
      // butterflies at spans 1, 2, 4 in the lane and 8 .. 128 across the lanes, then the
      // chunks of one block combined through shared memory (spans 256 and 512 as one sum with
      // the Sylvester signs).
      float is[8];
      load8(a.inv_s + k, is);
#pragma unroll
      for (int i = 0; i < 8; ++i) x[i] *= is[i];
#pragma unroll
      for (int h = 1; h < 8; h *= 2)
#pragma unroll
        for (int i = 0; i < 8; ++i)
          if ((i & h) == 0) {
            const float x0 = x[i], x1 = x[i + h];
            x[i] = x0 + x1;
            x[i + h] = x0 - x1;
          }
#pragma unroll
      for (int sh = 1; sh < 32; sh *= 2) {
        const float sgn = (lane & sh) ? -1.0f : 1.0f;
#pragma unroll
        for (int i = 0; i < 8; ++i) x[i] = fmaf(x[i], sgn, __shfl_xor_sync(0xFFFFFFFFu, x[i], sh));
      }
      const int nb = a.hb / 256;  // chunks per Hadamard block: 1, 2 or 4
      if (nb > 1) {
        xch[w][lane][0] = make_float4(x[0], x[1], x[2], x[3]);
        xch[w][lane][1] = make_float4(x[4], x[5], x[6], x[7]);
        __syncthreads();
        const int cl = w & (nb - 1), w0 = w - cl;  // this chunk's index in its block, the block's first warp
        float y[8] = {0.0f, 0.0f, 0.0f, 0.0f, 0.0f, 0.0f, 0.0f, 0.0f};
        for (int b = 0; b < nb; ++b) {
          const float sg = (__popc(cl & b) & 1) ? -1.0f : 1.0f;
          const float4 v0 = xch[w0 + b][lane][0], v1 = xch[w0 + b][lane][1];
          y[0] = fmaf(sg, v0.x, y[0]);
          y[1] = fmaf(sg, v0.y, y[1]);
          y[2] = fmaf(sg, v0.z, y[2]);
          y[3] = fmaf(sg, v0.w, y[3]);
          y[4] = fmaf(sg, v1.x, y[4]);
          y[5] = fmaf(sg, v1.y, y[5]);
          y[6] = fmaf(sg, v1.z, y[6]);
          y[7] = fmaf(sg, v1.w, y[7]);
        }
#pragma unroll
        for (int i = 0; i < 8; ++i) x[i] = y[i];
        __syncthreads();  // the exchange buffer is free for the next round
      }
    }
    if (!live) continue;
    if (a.dump) {
      float4* d = reinterpret_cast<float4*>(a.dump + static_cast<size_t>(m) * a.K + k);
      d[0] = make_float4(x[0], x[1], x[2], x[3]);
      d[1] = make_float4(x[4], x[5], x[6], x[7]);
    }
    quantize8_lanes<NV>(x, lane, m, k, a.q);
  }
}

template <int RP, bool NV>
cudaError_t launch_smallq_rp(const Handle& h, const void* X, const void* ws, int M, float* dump, cudaStream_t s) {
  const bool rot = h.rot;
  const ActLayout L = act_layout(h, M);
  uint8_t* base = static_cast<uint8_t*>(const_cast<void*>(ws));
  SmallArgs a;
  a.M = M;
  a.K = h.K;
  a.up = h.up32;
  a.ur = h.ur32;
  a.phat = reinterpret_cast<__half*>(base + L.phat_off);
  a.dump = dump;
  a.q = quant_out(h, L, base);
  a.inv_s = h.inv_s;
  a.hb = h.hb;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(M, 1, 1);
  cfg.blockDim = dim3(128, 1, 1);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (rot) return cudaLaunchKernelEx(&cfg, smallq_kernel<RP, NV, true>, static_cast<const __nv_bfloat16*>(X), a);
  return cudaLaunchKernelEx(&cfg, smallq_kernel<RP, NV, false>, static_cast<const __nv_bfloat16*>(X), a);
}

template <bool NV>
cudaError_t launch_smallq(const Handle& h, const void* X, const void* ws, int M, float* dump, cudaStream_t s) {
  switch (h.r_pad) {
    case 0: return launch_smallq_rp<0, NV>(h, X, ws, M, dump, s);
    case 16: return launch_smallq_rp<16, NV>(h, X, ws, M, dump, s);
    case 32: return launch_smallq_rp<32, NV>(h, X, ws, M, dump, s);
    case 48: return launch_smallq_rp<48, NV>(h, X, ws, M, dump, s);
    case 64: return launch_smallq_rp<64, NV>(h, X, ws, M, dump, s);
    default: return cudaErrorInvalidValue;
  }
}

// ---- the general-rank path (r_pad > kMaxRank, any rank up to K; K a multiple of 256) ---------
// Eq. (xsplit) on the CUDA cores, one CTA of four warps per token row, for ranks whose projection
// does not fit kernel (a)'s tensor-memory layout.  The row goes to shared memory in float32; warp
// w forms p_j for j = w, w + 4, ... as one warp-wide dot product over K (lane l takes channels
// 256 c + 8 l .. + 7), all four warps then form the remainder of their 256-channel chunks as
// x - sum_j p_j U[k, j] (j ascending) and quantize it with the lane quantizers, bit for bit those
// of the other paths.  It is the rank range's correctness path, not a tuned one: its cost grows
// as K r per token.
template <bool NV>
__global__ void __launch_bounds__(128) generalq_kernel(const __nv_bfloat16* __restrict__ X, const SmallArgs a, int RP) {
  extern __shared__ float gsm[];
  float* xs = gsm;          // [K] the row in float32
  float* ps = gsm + a.K;    // [RP] its projection
  pdl_launch_dependents();
  pdl_wait();
  const int lane = static_cast<int>(threadIdx.x & 31), w = static_cast<int>(threadIdx.x >> 5);
  const int m = blockIdx.x;
  const __nv_bfloat16* row = X + static_cast<size_t>(m) * a.K;
  const int nc = a.K / 256;
  for (int c = w; c < nc; c += 4) {
    const int k = 256 * c + 8 * lane;
    float x[8];
    load8(row + k, x);
    reinterpret_cast<float4*>(xs + k)[0] = make_float4(x[0], x[1], x[2], x[3]);
    reinterpret_cast<float4*>(xs + k)[1] = make_float4(x[4], x[5], x[6], x[7]);
  }
  __syncthreads();
  for (int j = w; j < RP; j += 4) {
    float acc = 0.0f;
    for (int c = 0; c < nc; ++c) {
      const int k = 256 * c + 8 * lane;
      float x[8], u[8];
      load8(xs + k, x);
      load8(a.up + static_cast<size_t>(j) * a.K + k, u);
#pragma unroll
      for (int i = 0; i < 8; ++i) acc = fmaf(x[i], u[i], acc);
    }
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) acc += __shfl_xor_sync(0xFFFFFFFFu, acc, off);
    if (lane == 0) {
      ps[j] = acc;
      a.phat[static_cast<size_t>(m) * RP + j] = __float2half_rn(acc);
    }
  }
  __syncthreads();
  for (int c = w; c < nc; c += 4) {
    const int k = 256 * c + 8 * lane;
    float x[8], acc[8] = {0.0f, 0.0f, 0.0f, 0.0f, 0.0f, 0.0f, 0.0f, 0.0f};
    load8(xs + k, x);
    for (int j = 0; j < RP; ++j) {
      float u[8];
      load8(a.ur + static_cast<size_t>(j) * a.K + k, u);
      const float pj = ps[j];
#pragma unroll
      for (int i = 0; i < 8; ++i) acc[i] = fmaf(pj, u[i], acc[i]);
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) x[i] -= acc[i];
    if (a.dump) {
      float4* d = reinterpret_cast<float4*>(a.dump + static_cast<size_t>(m) * a.K + k);
      d[0] = make_float4(x[0], x[1], x[2], x[3]);
      d[1] = make_float4(x[4], x[5], x[6], x[7]);
    }
    quantize8_lanes<NV>(x, lane, m, k, a.q);
  }
}

template <bool NV>
cudaError_t launch_general(const Handle& h, const void* X, const void* ws, int M, float* dump, cudaStream_t s) {
  const ActLayout L = act_layout(h, M);
  uint8_t* base = static_cast<uint8_t*>(const_cast<void*>(ws));
  SmallArgs a;
  a.M = M;
  a.K = h.K;
  a.up = h.up32;
  a.ur = h.ur32;
  a.phat = reinterpret_cast<__half*>(base + L.phat_off);
  a.dump = dump;
  a.q = quant_out(h, L, base);
  a.inv_s = nullptr;
  a.hb = 0;
  const size_t smem = sizeof(float) * (static_cast<size_t>(h.K) + h.r_pad);
  if (smem > 48 * 1024) {
    const cudaError_t e = cudaFuncSetAttribute(generalq_kernel<NV>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               static_cast<int>(smem));
    if (e != cudaSuccess) return e;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(M, 1, 1);
  cfg.blockDim = dim3(128, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, generalq_kernel<NV>, static_cast<const __nv_bfloat16*>(X), a, h.r_pad);
}

// Test support: the lane quantizers (quantize8_lanes, as the small-M and rotation kernels run
// them) applied to caller-given float32 rows, one warp per row and 256 values.
template <bool NV>
__global__ void __launch_bounds__(256) debug_lanes_kernel(const float* __restrict__ R, int M, const QuantOut q) {
  const long long wg = static_cast<long long>(blockIdx.x) * 8 + (threadIdx.x >> 5);
  const int nc = q.K / 256;
  if (wg >= static_cast<long long>(M) * nc) return;
  const int lane = static_cast<int>(threadIdx.x & 31);
  const int m = static_cast<int>(wg / nc), k = static_cast<int>(wg % nc) * 256 + 8 * lane;
  float x[8];
  load8(R + static_cast<size_t>(m) * q.K + k, x);
  quantize8_lanes<NV>(x, lane, m, k, q);
}

// Cluster size (CTAs along K per 128-row tile): as many as fit one wave of the GPU.

template <int RP, bool NV>
cudaError_t launch_rp(Handle& h, const ActMaps& am, const void* ws, int M, float* dump, bool resid_only,
                      cudaStream_t s, bool expand_w16) {
  using Cfg = ActCfg<RP>;
  const ActLayout L = act_layout(h, M);
  ActArgs a;
  a.M = M;
  a.K = h.K;
  a.G = h.G;
  const int tiles = (M + kBM - 1) / kBM;
  const int C = act_split(h.K, tiles, h.num_sms);
  a.C = C;
  a.Kc = h.K / C;
  a.M_pad = L.M_pad;
  uint8_t* base = static_cast<uint8_t*>(const_cast<void*>(ws));
  a.codes = base + L.codes_off;
  a.sf = base + L.scales_off;
  a.scales = reinterpret_cast<__nv_bfloat16*>(base + L.scales_off);
  a.phat = reinterpret_cast<__half*>(base + L.phat_off);
  a.part = reinterpret_cast<float*>(base + L.part_off);
  a.dump = dump;
  a.resid_only = resid_only ? 1 : 0;
  a.w = w16_args(h, L, ws);
  if (!expand_w16) a.w.w16 = nullptr;
  a.err = h.err;
  a.timeout_ns = deadline_budget_ns(h);

  static bool attr_done = false;
  if (!attr_done) {
    cudaError_t e = cudaFuncSetAttribute(actquant_kernel<RP, NV>, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::SMEM);
    if (e != cudaSuccess) return e;
    attr_done = true;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(C, tiles, 1);
  cfg.blockDim = dim3(kActThreads, 1, 1);
  cfg.dynamicSmemBytes = Cfg::SMEM;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (RP > 0) ? C : 1;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  const CUtensorMap& ut = (RP > 0) ? h.ucat_t_map : am.x_map;
  const CUtensorMap& u3 = (RP > 0) ? h.ucat3_map : am.x_map;
  return cudaLaunchKernelEx(&cfg, actquant_kernel<RP, NV>, am.x_map, ut, u3, a);
}

template <bool NV>
cudaError_t launch_fmt(Handle& h, const ActMaps& am, const void* ws, int M, float* dump, bool resid_only,
                       cudaStream_t s, bool expand_w16 = false) {
  switch (h.r_pad) {
    case 0: return launch_rp<0, NV>(h, am, ws, M, dump, resid_only, s, false);
    case 16: return launch_rp<16, NV>(h, am, ws, M, dump, resid_only, s, expand_w16);
    case 32: return launch_rp<32, NV>(h, am, ws, M, dump, resid_only, s, expand_w16);
    case 48: return launch_rp<48, NV>(h, am, ws, M, dump, resid_only, s, expand_w16);
    case 64: return launch_rp<64, NV>(h, am, ws, M, dump, resid_only, s, expand_w16);
    default: return cudaErrorInvalidValue;
  }
}

// Rotated layer: kernel (a) forms the remainder v = x - diag(s) H U p (and p_hat) into the
// workspace, then the rotation kernel maps it to x~_perp and quantizes; with r = 0 the rotation
// kernel reads X itself.  `dump` (optional) receives x~_perp.
template <bool NV>
cudaError_t launch_rotated(Handle& h, const ActMaps& am, const void* X, const void* ws, int M, float* dump,
                           cudaStream_t s, bool expand_w16) {
  const ActLayout L = act_layout(h, M);
  uint8_t* base = static_cast<uint8_t*>(const_cast<void*>(ws));
  RotArgs a;
  a.M = M;
  a.K = h.K;
  a.inv_s = h.inv_s;
  a.dump = dump;
  a.q = quant_out(h, L, base);
  if (h.r == 0) return launch_rotquant_t<__nv_bfloat16, NV>(h, static_cast<const __nv_bfloat16*>(X), a, s);
  float* resid = reinterpret_cast<float*>(base + L.resid_off);
  cudaError_t e = launch_fmt<NV>(h, am, ws, M, resid, true, s, expand_w16);
  if (e != cudaSuccess) return e;
  return launch_rotquant_t<float, NV>(h, resid, a, s);
}

}  // namespace

cudaError_t launch_debug_quantize_rows(const float* R, int M, int K, bool nvfp4, int G, uint8_t* codes,
                                       void* scales, cudaStream_t s) {
  const long long n = static_cast<long long>(M) * (K / kChunk);
  const int grid = static_cast<int>((n + 127) / 128);
  if (nvfp4)
    debug_quantize_kernel<true><<<grid, 128, 0, s>>>(R, M, K, G, codes, scales);
  else
    debug_quantize_kernel<false><<<grid, 128, 0, s>>>(R, M, K, G, codes, scales);
  return cudaGetLastError();
}

cudaError_t launch_debug_quantize_lanes(const float* R, int M, int K, bool nvfp4, int G, uint8_t* codes,
                                        uint8_t* scales, int M_pad, cudaStream_t s) {
  QuantOut q;
  q.K = K;
  q.G = G;
  q.M_pad = M_pad;
  q.codes = codes;
  q.sf = scales;
  q.scales = reinterpret_cast<__nv_bfloat16*>(scales);
  const long long warps = static_cast<long long>(M) * (K / 256);
  const int grid = static_cast<int>((warps + 7) / 8);
  if (nvfp4)
    debug_lanes_kernel<true><<<grid, 256, 0, s>>>(R, M, q);
  else
    debug_lanes_kernel<false><<<grid, 256, 0, s>>>(R, M, q);
  return cudaGetLastError();
}

cudaError_t launch_actquant(Handle& h, const ActMaps& am, const void* ws, int M, float* dump, cudaStream_t s,
                            bool expand_w16, bool* expanded) {
  const bool nv = h.fmt == kFmtNvfp4;
  if (expanded) *expanded = false;
  if (h.r_pad > kMaxRank) return nv ? launch_general<true>(h, am.x, ws, M, dump, s) : launch_general<false>(h, am.x, ws, M, dump, s);
  // The small-M kernel for few tokens, and for unrotated r = 0 layers at any token count (with no
  // projection its warp-wide pass beats kernel (a)'s tile pipeline: 15.0 against 19.0 us INT4 and
  // 14.6 against 30.0 us NVFP4 at M = 4096, K = 3072); small_m = 0 always takes kernel (a).
  if (h.K % 256 == 0 && h.small_m > 0 && (M <= h.small_m || (h.r == 0 && !h.rot)))
    return nv ? launch_smallq<true>(h, am.x, ws, M, dump, s) : launch_smallq<false>(h, am.x, ws, M, dump, s);
  // kernel (a) with a projection (r > 0), INT4: it can also write the GEMM's float16 weights
  const bool ex = expand_w16 && !nv && h.r_pad > 0 && act_layout(h, M).w16_off != 0;
  cudaError_t e;
  if (h.rot)
    e = nv ? launch_rotated<true>(h, am, am.x, ws, M, dump, s, false) : launch_rotated<false>(h, am, am.x, ws, M, dump, s, ex);
  else
    e = nv ? launch_fmt<true>(h, am, ws, M, dump, false, s) : launch_fmt<false>(h, am, ws, M, dump, false, s, ex);
  if (e == cudaSuccess && expanded) *expanded = ex;
  return e;
}

}  // namespace qwam
