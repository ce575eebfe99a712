// gemm.cu -- kernel (b): the 4-bit deflated path of Eq. (asp) with the 16-bit branch fused into
// the epilogue (Sec. 3.2; App. B.1 describes the paper's GEMM as one that keeps the weights
// packed at 4 bits and adds the protected branch in its epilogue).
//
//   Y[m, n] = sum_g s_x[m, g] s_w[g, n] P_g[m, n]  +  sum_j p_hat[m, j] B_hat[n, j]
//   P_g[m, n] = sum_{k in group g} q_x[m, k] q_w[n, k]          (exact integers)
//
// sm_103a has no integer tensor-core MMA, so the codes are fed to tcgen05.mma.kind::f8f6f4 as
// E4M3 bit patterns of exact multiples of 2^-9 (E4M3 subnormals, which the tensor core keeps):
//   A: activation byte = sign | |c|      -> value c * 2^-9     (written so by kernel (a))
//   B: weight byte     = c + 8 in [1,15] -> value (c + 8) 2^-9 (expanded here from 4 bits)
// so one group's float32 accumulator holds D = 2^-18 sum_k c_a (c_b + 8) = 2^-18 (P + 8 S_a)
// exactly (S_a = the activation group's code sum, every partial sum an integer below 2^13 times
// 2^-18).  The epilogue forms s_x P = alpha D + beta with alpha = 2^18 s_x, beta = -8 s_x S_a
// (per row and group) and accumulates s_w * (s_x P) in float32 registers.  The 4-bit weights
// stay packed in HBM; a nibble becomes its byte with three logic ops per eight nibbles because
// the packing puts the codes of k = 8j..8j+3 in the low and of k = 8j+4..8j+7 in the high
// nibbles of the four bytes of word j.  Each group has its own TMEM accumulator (four buffers);
// after the last group one kind::f16 MMA of K = r_pad forms p_hat B_hat^T, added with scale 1.
//
// CTA tile 128 x 128 outputs, 384 threads: warp 0 TMA producer, warp 1 MMA issuer and TMEM
// owner, warps 2..3 expand weight nibbles and stage the group scales, warps 4..11 epilogue
// (thread = output row x 64 columns, float32 accumulators, packed f32x2 arithmetic).
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

constexpr int SO = 3;    // operand stages (A by TMA, B expanded)
constexpr int SP = 4;    // packed-weight stages
constexpr int NSL = 8;   // scale slots (one group each)
constexpr int NTB = 4;   // TMEM accumulator buffers (128 columns each)
constexpr int NEXP = 64; // expander threads
constexpr int NEPI = 256;// epilogue threads
constexpr int OA_BYTES = kBM * kGemmKS;          // 16 KB E4M3 A, 128-byte swizzle
constexpr int OB_BYTES = kGemmBN * kGemmKS;      // 16 KB E4M3 B, 128-byte swizzle
constexpr int OSTAGE = OA_BYTES + OB_BYTES;
constexpr int PB_BYTES = kGemmBN * kGemmKS / 2;  // 8 KB packed B
constexpr int PSX_BYTES = 4 * kBM * 4;           // up to 4 groups x 128 f32 activation scales
constexpr int PCS_BYTES = 4 * kBM * 4;           // up to 4 groups x 128 f32 activation code sums
constexpr int PSW_BYTES = 4 * kGemmBN * 2;       // up to 4 groups x 128 f16 weight scales
constexpr int PSTAGE = PB_BYTES + PSX_BYTES + PCS_BYTES + PSW_BYTES;
constexpr int SLOT_FLOATS = kGemmBN + 2 * kBM;   // s_w (f32) | s_x | code sums

template <int RP>
struct GemmCfg {
  static constexpr int BR_BYTES = RP * kBM * 2;  // p_hat tile (and the B_hat tile), RP/8 boxes of 2 KB
  static constexpr int NBAR = 2 * SO + 2 * SP + 2 * NSL + 2 * NTB + 2;
  static constexpr int SMEM =
      1024 + SO * OSTAGE + SP * PSTAGE + NSL * SLOT_FLOATS * 4 + 2 * BR_BYTES + NBAR * 8 + 16;
  static_assert(SMEM <= 232448, "kernel (b) shared memory above the 227 KB per-CTA limit");
};

typedef unsigned long long f2;  // two packed float32 (for the f32x2 instructions)

__device__ __forceinline__ f2 pk(float lo, float hi) {
  return static_cast<f2>(__float_as_uint(lo)) | (static_cast<f2>(__float_as_uint(hi)) << 32);
}
__device__ __forceinline__ f2 pku(uint32_t lo, uint32_t hi) {
  return static_cast<f2>(lo) | (static_cast<f2>(hi) << 32);
}
__device__ __forceinline__ float lo_f(f2 v) { return __uint_as_float(static_cast<uint32_t>(v)); }
__device__ __forceinline__ float hi_f(f2 v) { return __uint_as_float(static_cast<uint32_t>(v >> 32)); }
__device__ __forceinline__ f2 fma2(f2 a, f2 b, f2 c) {
  f2 d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ f2 add2(f2 a, f2 b) {
  f2 d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}

template <int RP>
__global__ void __launch_bounds__(384, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap qx_map, const __grid_constant__ CUtensorMap qw_map,
                const __grid_constant__ CUtensorMap sx_map, const __grid_constant__ CUtensorMap cs_map,
                const __grid_constant__ CUtensorMap sw_map, const __grid_constant__ CUtensorMap ph_map,
                const __grid_constant__ CUtensorMap bh_map, const GemmArgs a) {
  using Cfg = GemmCfg<RP>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* oring = smem;                          // SO x (A 16 KB | B 16 KB), 1024-aligned
  uint8_t* pring = oring + SO * OSTAGE;           // SP x (B packed | s_x | code sums | s_w)
  float* slots = reinterpret_cast<float*>(pring + SP * PSTAGE);
  uint8_t* br = reinterpret_cast<uint8_t*>(slots + NSL * SLOT_FLOATS);  // p_hat tile | B_hat tile
  uint64_t* bars = reinterpret_cast<uint64_t*>(br + 2 * Cfg::BR_BYTES);
  uint64_t* ofull = bars;
  uint64_t* oempty = ofull + SO;
  uint64_t* pfull = oempty + SO;
  uint64_t* pempty = pfull + SP;
  uint64_t* sfull = pempty + SP;
  uint64_t* sempty = sfull + NSL;
  uint64_t* tfull = sempty + NSL;
  uint64_t* tempty = tfull + NTB;
  uint64_t* bfull = tempty + NTB;
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
    for (int i = 0; i < SO; ++i) {
      mbar_init(&ofull[i], 1 + NEXP);
      mbar_init(&oempty[i], 1);
    }
    for (int i = 0; i < SP; ++i) {
      mbar_init(&pfull[i], 1);
      mbar_init(&pempty[i], NEXP);
    }
    for (int i = 0; i < NSL; ++i) {
      mbar_init(&sfull[i], NEXP);
      mbar_init(&sempty[i], NEPI);
    }
    for (int i = 0; i < NTB; ++i) {
      mbar_init(&tfull[i], 1);
      mbar_init(&tempty[i], NEPI);
    }
    mbar_init(bfull, 1);
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (wid == 1) {
    tmem_alloc(tmem_slot, 512);
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
      const uint32_t pbytes = PB_BYTES + gps * (kBM * 8 + kGemmBN * 2);
      for (int st = 0; st < nst; ++st) {
        const int sp = st % SP, so = st % SO;
        if (st >= SP) ok = mbar_wait(&pempty[sp], ((st / SP) & 1) ^ 1, wc);
        if (!ok) break;
        uint8_t* p = pring + sp * PSTAGE;
        mbar_arrive_expect_tx(&pfull[sp], pbytes);
        tma_load_2d(p, &qw_map, &pfull[sp], st * (kGemmKS / 2), n0);
        tma_load_2d(p + PB_BYTES, &sx_map, &pfull[sp], m0, st * gps);
        tma_load_2d(p + PB_BYTES + PSX_BYTES, &cs_map, &pfull[sp], m0, st * gps);
        tma_load_2d(p + PB_BYTES + PSX_BYTES + PCS_BYTES, &sw_map, &pfull[sp], n0, st * gps);
        if (st >= SO) ok = mbar_wait(&oempty[so], ((st / SO) & 1) ^ 1, wc);
        if (!ok) break;
        mbar_arrive_expect_tx(&ofull[so], OA_BYTES);
        tma_load_2d(oring + so * OSTAGE, &qx_map, &ofull[so], st * kGemmKS, m0);
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
        const int so = st % SO;
        ok = mbar_wait(&ofull[so], (st / SO) & 1, wc);
        if (!ok) break;
        tc_fence_after();
        const uint32_t xa = smem_u32(oring + so * OSTAGE), xb = xa + OA_BYTES;
        for (int gi = 0; gi < gps && ok; ++gi) {
          const int g = st * gps + gi;
          if (g >= ngroups) break;
          const int b = g % NTB;
          if (g >= NTB) ok = mbar_wait(&tempty[b], ((g / NTB) & 1) ^ 1, wc);
          if (!ok) break;
          tc_fence_after();
          for (int kk = 0; kk < G / 32; ++kk) {
            const uint32_t off = static_cast<uint32_t>((gi * (G / 32) + kk) * 32);
            mma_f8f6f4(tmem + b * 128, smem_desc(xa + off, 16, 1024, kSw128), smem_desc(xb + off, 16, 1024, kSw128),
                       idesc, kk != 0);
          }
          mma_commit(&tfull[b]);
        }
        mma_commit(&oempty[so]);
      }
      if constexpr (RP > 0) {
        const int g = ngroups, b = g % NTB;
        if (ok) ok = mbar_wait(bfull, 0, wc);
        if (ok && g >= NTB) ok = mbar_wait(&tempty[b], ((g / NTB) & 1) ^ 1, wc);
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
  } else if (wid < 4) {
    // ------------------------------------------------------------- weight expanders + scales
    const int e = static_cast<int>(threadIdx.x) - 64;  // 0..63
    const uint32_t kX8 = 0x88888888u;
    bool ok = true;
    for (int st = 0; st < nst && ok; ++st) {
      const int sp = st % SP, so = st % SO;
      ok = mbar_wait(&pfull[sp], (st / SP) & 1, wc);
      if (ok && st >= SO) ok = mbar_wait(&oempty[so], ((st / SO) & 1) ^ 1, wc);
      if (!ok) break;
      const uint8_t* p = pring + sp * PSTAGE;
      uint8_t* xb = oring + so * OSTAGE + OA_BYTES;
#pragma unroll 4
      for (int i = 0; i < 16; ++i) {
        const int t = e + NEXP * i;
        const int row = t >> 3, j = t & 7;
        const uint2 pkd = *reinterpret_cast<const uint2*>(p + row * 64 + j * 8);
        uint4 o;
        o.x = (pkd.x ^ kX8) & 0x0F0F0F0Fu;
        o.y = ((pkd.x >> 4) ^ kX8) & 0x0F0F0F0Fu;
        o.z = (pkd.y ^ kX8) & 0x0F0F0F0Fu;
        o.w = ((pkd.y >> 4) ^ kX8) & 0x0F0F0F0Fu;
        *reinterpret_cast<uint4*>(xb + (row >> 3) * 1024 + (row & 7) * 128 + ((j ^ (row & 7)) << 4)) = o;
      }
      fence_proxy_async_smem();
      mbar_arrive(&ofull[so]);
      // group scales of this stage -> float32 slots for the epilogue
      const float* psx = reinterpret_cast<const float*>(p + PB_BYTES);
      const float* pcs = reinterpret_cast<const float*>(p + PB_BYTES + PSX_BYTES);
      const __half* psw = reinterpret_cast<const __half*>(p + PB_BYTES + PSX_BYTES + PCS_BYTES);
      for (int gi = 0; gi < gps && ok; ++gi) {
        const int g = st * gps + gi;
        if (g >= ngroups) break;
        const int sl = g % NSL;
        if (g >= NSL) ok = mbar_wait(&sempty[sl], ((g / NSL) & 1) ^ 1, wc);
        if (!ok) break;
        float* slot = slots + sl * SLOT_FLOATS;
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int i = e + NEXP * h;
          slot[i] = __half2float(psw[gi * kGemmBN + i]);
          slot[kGemmBN + i] = psx[gi * kBM + i];
          slot[kGemmBN + kBM + i] = pcs[gi * kBM + i];
        }
        mbar_arrive(&sfull[sl]);
      }
      fence_proxy_async_smem();  // reads of the packed stage before the TMA refills it
      mbar_arrive(&pempty[sp]);
    }
  } else {
    // ------------------------------------------------------------- epilogue
    // Warps 4..11: warp w reads TMEM lanes 32*(w%4).. (its quadrant of rows) and the 64 output
    // columns [64*((w-4)/4), +64).
    const int quad = wid & 3;
    const int row = quad * 32 + static_cast<int>(lane);
    const int m = m0 + row;
    const int col0 = 64 * ((static_cast<int>(wid) - 4) >> 2);
    const uint32_t tlane = tmem + (static_cast<uint32_t>(quad * 32) << 16) + col0;
    f2 acc[32];
#pragma unroll
    for (int i = 0; i < 32; ++i) acc[i] = 0ull;
    bool ok = true;
    const int ntot = ngroups + (RP > 0 ? 1 : 0);
    for (int g = 0; g < ntot; ++g) {
      const int b = g % NTB;
      if (ok) ok = mbar_wait(&tfull[b], (g / NTB) & 1, wc);
      tc_fence_after();
      uint32_t v[64];
      tmem_ld32(tlane + b * 128, *reinterpret_cast<uint32_t(*)[32]>(&v[0]));
      tmem_ld32(tlane + b * 128 + 32, *reinterpret_cast<uint32_t(*)[32]>(&v[32]));
      tmem_ld_wait();
      tc_fence_before();
      mbar_arrive(&tempty[b]);
      if (g < ngroups) {
        const int sl = g % NSL;
        if (ok) ok = mbar_wait(&sfull[sl], (g / NSL) & 1, wc);
        const float* slot = slots + sl * SLOT_FLOATS;
        const float sxv = slot[kGemmBN + row];
        const float alpha = sxv * 262144.0f;                       // 2^18 s_x (exact)
        const float beta = -8.0f * sxv * slot[kGemmBN + kBM + row];  // -8 s_x S_a
        const f2 al2 = pk(alpha, alpha), be2 = pk(beta, beta);
        const float4* w4 = reinterpret_cast<const float4*>(slot + col0);
#pragma unroll
        for (int i4 = 0; i4 < 16; ++i4) {
          const float4 w = w4[i4];
          const f2 t0 = fma2(pku(v[4 * i4], v[4 * i4 + 1]), al2, be2);
          const f2 t1 = fma2(pku(v[4 * i4 + 2], v[4 * i4 + 3]), al2, be2);
          acc[2 * i4] = fma2(t0, pk(w.x, w.y), acc[2 * i4]);
          acc[2 * i4 + 1] = fma2(t1, pk(w.z, w.w), acc[2 * i4 + 1]);
        }
        mbar_arrive(&sempty[sl]);
      } else {
#pragma unroll
        for (int i = 0; i < 32; ++i) acc[i] = add2(acc[i], pku(v[2 * i], v[2 * i + 1]));
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
                make_float4(lo_f(acc[4 * c8]), hi_f(acc[4 * c8]), lo_f(acc[4 * c8 + 1]), hi_f(acc[4 * c8 + 1]));
            reinterpret_cast<float4*>(yr + c8 * 8)[1] = make_float4(lo_f(acc[4 * c8 + 2]), hi_f(acc[4 * c8 + 2]),
                                                                    lo_f(acc[4 * c8 + 3]), hi_f(acc[4 * c8 + 3]));
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
              __nv_bfloat162 h2 = __floats2bfloat162_rn(lo_f(acc[4 * c8 + t]), hi_f(acc[4 * c8 + t]));
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
    tmem_dealloc(tmem, 512);
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
  gemm_kernel<RP><<<grid, 384, Cfg::SMEM, s>>>(am.qx_map, h.qw_map, am.sx_map, am.cs_map, h.sw_map, ph, bh, a);
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
