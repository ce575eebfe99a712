// gemm.cu -- kernel (b): the 4-bit deflated path of Eq. (asp) with the 16-bit branch fused into
// the epilogue (Sec. 3.2; App. B.1 describes the paper's GEMM as one that keeps the weights
// packed at 4 bits and adds the protected branch in its epilogue).
//
//   Y[m, n] = sum_g s_x[m, g] s_w[g, n] P_g[m, n]  +  sum_j p_hat[m, j] B_hat[n, j]
//   P_g[m, n] = sum_{k in group g} q_x[m, k] q_w[n, k]          (exact integers)
//
// sm_103a has no integer tensor-core MMA, so the 4-bit codes (always in [-7, 7]) are expanded to
// E4M3, which represents every integer in [-16, 16] exactly, and multiplied with
// tcgen05.mma.kind::f8f6f4 into float32 TMEM accumulators.  Every product is an integer of
// magnitude <= 49 and every per-group sum is below 2^12, so the float32 accumulator holds the
// same integer an int32 accumulator would.  Each group gets its own accumulator (two TMEM
// buffers, double-buffered); the epilogue warps apply s_x * s_w in float32 and accumulate in
// registers.  After the last group, one kind::f16 MMA of K = r_pad forms p_hat B_hat^T into a
// TMEM buffer that the epilogue adds with scale 1.
//
// CTA tile 128 x 128 outputs; 448 threads: warp 0 TMA producer, warp 1 MMA issuer and TMEM
// owner, warps 2..5 expand packed nibbles to E4M3 (128-byte swizzled, K-major) and stage the
// group scales, warps 6..13 epilogue (thread = output row x 64 columns, float32 accumulators).
#include "internal.h"
#include "ptx.cuh"

namespace qwam {
namespace {

struct GemmArgs {
  int M, N, K, G;
  void* Y;
  int y_f32;
  int* err;
  uint64_t timeout_ns;
};

constexpr int SP = 4;   // packed stages
constexpr int SE = 2;   // expanded stages
constexpr int NSL = 8;  // scale slots (one group each)
constexpr int PA_BYTES = kBM * kGemmKS / 2;      // 8 KB packed A
constexpr int PB_BYTES = kGemmBN * kGemmKS / 2;  // 8 KB packed B
constexpr int PSX_BYTES = 4 * kBM * 4;           // up to 4 groups x 128 f32 activation scales
constexpr int PSW_BYTES = 4 * kGemmBN * 2;       // up to 4 groups x 128 f16 weight scales
constexpr int PSTAGE = PA_BYTES + PB_BYTES + PSX_BYTES + PSW_BYTES;  // 19 KB
constexpr int XA_BYTES = kBM * kGemmKS;          // 16 KB E4M3 A
constexpr int XB_BYTES = kGemmBN * kGemmKS;      // 16 KB E4M3 B
constexpr int XSTAGE = XA_BYTES + XB_BYTES;
constexpr int SLOT_BYTES = (kGemmBN + kBM) * 4;  // f32 weight scales + f32 activation scales

template <int RP>
struct GemmCfg {
  static constexpr int BR_BYTES = RP * kBM * 2;  // p_hat tile (and the B_hat tile), RP/8 boxes of 2 KB
  static constexpr int NBAR = 2 * SP + 2 * SE + 2 * NSL + 4 + 2;
  static constexpr int SMEM = 1024 + SE * XSTAGE + SP * PSTAGE + NSL * SLOT_BYTES + 2 * BR_BYTES + NBAR * 8 + 16;
};

// 4 two's-complement nibbles (low 16 bits of w) -> 4 E4M3 bytes of the same integers.
__device__ __forceinline__ uint32_t nibbles_to_e4m3(uint32_t w) {
  // E4M3 of 0..7 and of -8..-1 (indexed by the low three bits of the nibble).
  constexpr uint32_t P0 = 0x44403800u, P1 = 0x4E4C4A48u;
  constexpr uint32_t N0 = 0xCACCCED0u, N1 = 0xB8C0C4C8u;
  const uint32_t sel = w & 0x7777u;
  const uint32_t pos = __byte_perm(P0, P1, sel);
  const uint32_t neg = __byte_perm(N0, N1, sel);
  const uint32_t pick = ((w >> 1) & 0x4444u) | 0x3210u;
  return __byte_perm(pos, neg, pick);
}

template <int RP>
__global__ void __launch_bounds__(448, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap qx_map, const __grid_constant__ CUtensorMap qw_map,
                const __grid_constant__ CUtensorMap sx_map, const __grid_constant__ CUtensorMap sw_map,
                const __grid_constant__ CUtensorMap ph_map, const __grid_constant__ CUtensorMap bh_map,
                const GemmArgs a) {
  using Cfg = GemmCfg<RP>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* xring = smem;                          // SE x (A 16 KB | B 16 KB), 1024-aligned
  uint8_t* pring = xring + SE * XSTAGE;           // SP x (A | B | sx | sw)
  float* slots = reinterpret_cast<float*>(pring + SP * PSTAGE);  // NSL x (sw[128] | sx[128])
  uint8_t* br = reinterpret_cast<uint8_t*>(slots) + NSL * SLOT_BYTES;  // p_hat tile | B_hat tile
  uint64_t* bars = reinterpret_cast<uint64_t*>(br + 2 * Cfg::BR_BYTES);
  uint64_t* pfull = bars;
  uint64_t* pempty = pfull + SP;
  uint64_t* xfull = pempty + SP;
  uint64_t* xempty = xfull + SE;
  uint64_t* sfull = xempty + SE;
  uint64_t* sempty = sfull + NSL;
  uint64_t* tfull = sempty + NSL;
  uint64_t* tempty = tfull + 2;
  uint64_t* bfull = tempty + 2;
  uint64_t* drain = bfull + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + Cfg::NBAR);
  int* abort_flag = reinterpret_cast<int*>(tmem_slot + 1);

  const uint32_t wid = warp_id(), lane = lane_id();
  const int n0 = blockIdx.x * kGemmBN;
  const int m0 = blockIdx.y * kBM;
  const int G = a.G;
  const int gps = kGemmKS / G;                    // groups per stage (2 or 4)
  const int ngroups = a.K / G;
  const int nst = (a.K + kGemmKS - 1) / kGemmKS;  // the last stage may be partly past K (zero-filled)

  if (threadIdx.x == 0) {
    for (int i = 0; i < SP; ++i) {
      mbar_init(&pfull[i], 1);
      mbar_init(&pempty[i], 128);
    }
    for (int i = 0; i < SE; ++i) {
      mbar_init(&xfull[i], 128);
      mbar_init(&xempty[i], 1);
    }
    for (int i = 0; i < NSL; ++i) {
      mbar_init(&sfull[i], 128);
      mbar_init(&sempty[i], 256);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&tfull[i], 1);
      mbar_init(&tempty[i], 256);
    }
    mbar_init(bfull, 1);
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (wid == 1) {
    tmem_alloc(tmem_slot, 256);
    tmem_relinquish();
  }
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const WaitCtl wc{abort_flag, a.err, globaltimer_ns() + a.timeout_ns};

  if (wid == 0) {
    // ------------------------------------------------------------- TMA producer
    if (lane == 0) {
      bool ok = true;
      if constexpr (RP > 0) {
        mbar_arrive_expect_tx(bfull, 2 * Cfg::BR_BYTES);
        for (int b = 0; b < RP / 8; ++b) {
          tma_load_2d(br + b * 2048, &ph_map, bfull, b * 8, m0);
          tma_load_2d(br + Cfg::BR_BYTES + b * 2048, &bh_map, bfull, b * 8, n0);
        }
      }
      const uint32_t bytes = PA_BYTES + PB_BYTES + gps * (kBM * 4 + kGemmBN * 2);
      for (int st = 0; st < nst; ++st) {
        const int s = st % SP;
        if (st >= SP) ok = mbar_wait(&pempty[s], ((st / SP) & 1) ^ 1, wc);
        if (!ok) break;
        uint8_t* p = pring + s * PSTAGE;
        mbar_arrive_expect_tx(&pfull[s], bytes);
        tma_load_2d(p, &qx_map, &pfull[s], st * (kGemmKS / 2), m0);
        tma_load_2d(p + PA_BYTES, &qw_map, &pfull[s], st * (kGemmKS / 2), n0);
        tma_load_2d(p + PA_BYTES + PB_BYTES, &sx_map, &pfull[s], m0, st * gps);
        tma_load_2d(p + PA_BYTES + PB_BYTES + PSX_BYTES, &sw_map, &pfull[s], n0, st * gps);
      }
      // Let every issued load land before the CTA can exit.
      int never = 0;
      const WaitCtl dc{&never, a.err, globaltimer_ns() + a.timeout_ns};
      const int last = ok ? nst : 0;
      for (int j = (last > SP ? last - SP : 0); j < last; ++j) mbar_wait(&pfull[j % SP], (j / SP) & 1, dc);
      if (RP > 0) mbar_wait(bfull, 0, dc);
    }
  } else if (wid == 1) {
    // ------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      bool ok = true;
      constexpr uint32_t idesc = idesc_e4m3(kBM, kGemmBN);
      for (int st = 0; st < nst && ok; ++st) {
        const int x = st % SE;
        ok = mbar_wait(&xfull[x], (st / SE) & 1, wc);
        if (!ok) break;
        tc_fence_after();
        const uint32_t xa = smem_u32(xring + x * XSTAGE), xb = xa + XA_BYTES;
        for (int gi = 0; gi < gps && ok; ++gi) {
          const int g = st * gps + gi;
          if (g >= ngroups) break;
          const int b = g & 1;
          if (g >= 2) ok = mbar_wait(&tempty[b], ((g >> 1) & 1) ^ 1, wc);
          if (!ok) break;
          tc_fence_after();
          for (int kk = 0; kk < G / 32; ++kk) {
            const uint32_t off = static_cast<uint32_t>((gi * (G / 32) + kk) * 32);
            mma_f8f6f4(tmem + b * 128, smem_desc(xa + off, 16, 1024, kSw128), smem_desc(xb + off, 16, 1024, kSw128),
                       idesc, kk != 0);
          }
          mma_commit(&tfull[b]);
        }
        mma_commit(&xempty[x]);
      }
      if constexpr (RP > 0) {
        const int g = ngroups, b = g & 1;
        if (ok) ok = mbar_wait(bfull, 0, wc);
        if (ok && g >= 2) ok = mbar_wait(&tempty[b], ((g >> 1) & 1) ^ 1, wc);
        if (ok) {
          tc_fence_after();
          constexpr uint32_t idesc_br = idesc_f16(kBM, kGemmBN);
          const uint32_t pa = smem_u32(br), pb = pa + Cfg::BR_BYTES;
#pragma unroll
          for (int kk = 0; kk < RP / 16; ++kk)
            mma_f16(tmem + b * 128, smem_desc(pa + kk * 4096, 2048, 128, kSwNone),
                    smem_desc(pb + kk * 4096, 2048, 128, kSwNone), idesc_br, kk != 0);
          mma_commit(&tfull[b]);
        }
      }
      mma_commit(drain);
      int never = 0;
      const WaitCtl dc{&never, a.err, globaltimer_ns() + a.timeout_ns};
      mbar_wait(drain, 0, dc);
    }
    __syncwarp();
  } else if (wid < 6) {
    // ------------------------------------------------------------- expanders
    const int e = static_cast<int>(threadIdx.x) - 64;  // 0..127
    bool ok = true;
    for (int st = 0; st < nst && ok; ++st) {
      const int s = st % SP, x = st % SE;
      ok = mbar_wait(&pfull[s], (st / SP) & 1, wc);
      if (ok && st >= SE) ok = mbar_wait(&xempty[x], ((st / SE) & 1) ^ 1, wc);
      if (!ok) break;
      const uint8_t* p = pring + s * PSTAGE;
      uint8_t* xs = xring + x * XSTAGE;
#pragma unroll 4
      for (int i = 0; i < 16; ++i) {
        const int t = e + 128 * i;
        const int mat = t >> 10, tt = t & 1023, row = tt >> 3, j = tt & 7;
        const uint2 pk = *reinterpret_cast<const uint2*>(p + mat * PA_BYTES + row * 64 + j * 8);
        uint4 o;
        o.x = nibbles_to_e4m3(pk.x);
        o.y = nibbles_to_e4m3(pk.x >> 16);
        o.z = nibbles_to_e4m3(pk.y);
        o.w = nibbles_to_e4m3(pk.y >> 16);
        *reinterpret_cast<uint4*>(xs + mat * XA_BYTES + (row >> 3) * 1024 + (row & 7) * 128 + ((j ^ (row & 7)) << 4)) = o;
      }
      fence_proxy_async_smem();
      mbar_arrive(&xfull[x]);
      // group scales of this stage -> float32 slots for the epilogue
      const float* psx = reinterpret_cast<const float*>(p + PA_BYTES + PB_BYTES);
      const __half* psw = reinterpret_cast<const __half*>(p + PA_BYTES + PB_BYTES + PSX_BYTES);
      for (int gi = 0; gi < gps && ok; ++gi) {
        const int g = st * gps + gi;
        if (g >= ngroups) break;
        const int sl = g % NSL;
        if (g >= NSL) ok = mbar_wait(&sempty[sl], ((g / NSL) & 1) ^ 1, wc);
        if (!ok) break;
        float* slot = slots + sl * (kGemmBN + kBM);
        slot[e] = __half2float(psw[gi * kGemmBN + e]);
        slot[kGemmBN + e] = psx[gi * kBM + e];
        mbar_arrive(&sfull[sl]);
      }
      mbar_arrive(&pempty[s]);
    }
  } else {
    // ------------------------------------------------------------- epilogue
    // Warps 6..13: warp w reads TMEM lanes 32*(w%4).. (its quadrant of rows) and the 64
    // output columns [64*((w-6)/4), +64).
    const int quad = wid & 3;
    const int row = quad * 32 + static_cast<int>(lane);
    const int m = m0 + row;
    const int col0 = 64 * ((static_cast<int>(wid) - 6) >> 2);
    const uint32_t tlane = tmem + (static_cast<uint32_t>(quad * 32) << 16) + col0;
    float acc[64];
#pragma unroll
    for (int i = 0; i < 64; ++i) acc[i] = 0.0f;
    bool ok = true;
    const int ntot = ngroups + (RP > 0 ? 1 : 0);
    for (int g = 0; g < ntot; ++g) {
      const int b = g & 1;
      if (ok) ok = mbar_wait(&tfull[b], (g >> 1) & 1, wc);
      tc_fence_after();
      if (g < ngroups) {
        const int sl = g % NSL;
        if (ok) ok = mbar_wait(&sfull[sl], (g / NSL) & 1, wc);
        const float* slot = slots + sl * (kGemmBN + kBM);
        const float sxv = slot[kGemmBN + row];
#pragma unroll
        for (int c = 0; c < 2; ++c) {
          uint32_t v[32];
          tmem_ld32(tlane + b * 128 + c * 32, v);
          tmem_ld_wait();
          const float4* w4 = reinterpret_cast<const float4*>(slot + col0 + c * 32);
#pragma unroll
          for (int i4 = 0; i4 < 8; ++i4) {
            const float4 w = w4[i4];
            acc[c * 32 + 4 * i4 + 0] = fmaf(__uint_as_float(v[4 * i4 + 0]) * w.x, sxv, acc[c * 32 + 4 * i4 + 0]);
            acc[c * 32 + 4 * i4 + 1] = fmaf(__uint_as_float(v[4 * i4 + 1]) * w.y, sxv, acc[c * 32 + 4 * i4 + 1]);
            acc[c * 32 + 4 * i4 + 2] = fmaf(__uint_as_float(v[4 * i4 + 2]) * w.z, sxv, acc[c * 32 + 4 * i4 + 2]);
            acc[c * 32 + 4 * i4 + 3] = fmaf(__uint_as_float(v[4 * i4 + 3]) * w.w, sxv, acc[c * 32 + 4 * i4 + 3]);
          }
        }
        tc_fence_before();
        mbar_arrive(&tempty[b]);
        mbar_arrive(&sempty[sl]);
      } else {
#pragma unroll
        for (int c = 0; c < 2; ++c) {
          uint32_t v[32];
          tmem_ld32(tlane + b * 128 + c * 32, v);
          tmem_ld_wait();
#pragma unroll
          for (int i = 0; i < 32; ++i) acc[c * 32 + i] += __uint_as_float(v[i]);
        }
        tc_fence_before();
        mbar_arrive(&tempty[b]);
      }
    }
    if (ok && m < a.M) {
      const int nb = n0 + col0;
      if (a.y_f32) {
        float* yr = static_cast<float*>(a.Y) + static_cast<size_t>(m) * a.N + nb;
#pragma unroll
        for (int c8 = 0; c8 < 8; ++c8) {
          if (nb + c8 * 8 < a.N) {
            reinterpret_cast<float4*>(yr + c8 * 8)[0] =
                make_float4(acc[c8 * 8], acc[c8 * 8 + 1], acc[c8 * 8 + 2], acc[c8 * 8 + 3]);
            reinterpret_cast<float4*>(yr + c8 * 8)[1] =
                make_float4(acc[c8 * 8 + 4], acc[c8 * 8 + 5], acc[c8 * 8 + 6], acc[c8 * 8 + 7]);
          }
        }
      } else {
        __nv_bfloat16* yr = static_cast<__nv_bfloat16*>(a.Y) + static_cast<size_t>(m) * a.N + nb;
#pragma unroll
        for (int c8 = 0; c8 < 8; ++c8) {
          if (nb + c8 * 8 < a.N) {
            uint32_t w[4];
#pragma unroll
            for (int t = 0; t < 4; ++t) {
              __nv_bfloat162 h2 = __floats2bfloat162_rn(acc[c8 * 8 + 2 * t], acc[c8 * 8 + 2 * t + 1]);
              w[t] = *reinterpret_cast<uint32_t*>(&h2);
            }
            *reinterpret_cast<uint4*>(yr + c8 * 8) = make_uint4(w[0], w[1], w[2], w[3]);
          }
        }
      }
    }
  }

  __syncthreads();
  if (wid == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 256);
  }
}

template <int RP>
cudaError_t launch_rp(Handle& h, const ActMaps& am, int M, void* Y, bool y_f32, cudaStream_t s) {
  using Cfg = GemmCfg<RP>;
  GemmArgs a;
  a.M = M;
  a.N = h.N;
  a.K = h.K;
  a.G = h.G;
  a.Y = Y;
  a.y_f32 = y_f32 ? 1 : 0;
  a.err = h.err;
  a.timeout_ns = deadline_budget_ns(h);
  static bool attr_done = false;
  if (!attr_done) {
    cudaError_t e = cudaFuncSetAttribute(gemm_kernel<RP>, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::SMEM);
    if (e != cudaSuccess) return e;
    attr_done = true;
  }
  dim3 grid((h.N + kGemmBN - 1) / kGemmBN, (M + kBM - 1) / kBM, 1);
  const CUtensorMap& ph = (RP > 0) ? am.ph_map : am.qx_map;
  const CUtensorMap& bh = (RP > 0) ? h.Bh_map : am.qx_map;
  gemm_kernel<RP><<<grid, 448, Cfg::SMEM, s>>>(am.qx_map, h.qw_map, am.sx_map, h.sw_map, ph, bh, a);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_gemm(Handle& h, const ActMaps& am, const void* ws, int M, void* Y, bool y_f32, cudaStream_t s) {
  (void)ws;
  switch (h.r_pad) {
    case 0: return launch_rp<0>(h, am, M, Y, y_f32, s);
    case 16: return launch_rp<16>(h, am, M, Y, y_f32, s);
    case 32: return launch_rp<32>(h, am, M, Y, y_f32, s);
    case 48: return launch_rp<48>(h, am, M, Y, y_f32, s);
    case 64: return launch_rp<64>(h, am, M, Y, y_f32, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace qwam
