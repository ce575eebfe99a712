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
// after the last group of a tile one kind::f16 MMA of K = r_pad forms p_hat B_hat^T, which the
// epilogue adds with scale 1.
//
// Persistent CTAs (one per SM) walk output tiles of 128 x 128 with a static stride; every ring
// (activation tiles, packed weights with the group scales, expanded weights, branch tiles, scale
// slots, TMEM accumulators) runs continuously across tiles, so loads for the next tile overlap
// the epilogue of the current one.  448 threads: warp 0 TMA producer, warp 1 MMA issuer and TMEM
// owner, warps 2..5 expand weight nibbles and stage the group scales (two teams taking alternate
// stages), warps 6..13 epilogue
// (thread = output row x 64 columns, packed f32x2).  Every ring has exactly one waiting role per
// side, which waits for each phase in turn.
#include "internal.h"
#include "ptx.cuh"

namespace qwam {
namespace {

struct GemmArgs {
  int M, N, K, G;
  int m_tiles, n_tiles;
  void* Y;
  int y_f32;
  int* err;
  uint64_t timeout_ns;
};

// Two expander teams take alternate stages.  Every ring a team touches therefore has an even
// number of slots, so each slot always belongs to the same team and every waiter sees each of its
// slot's phases in turn.
constexpr int SX = 2;     // expanded-weight stages (expanders -> MMA): one per team
constexpr int NSS = 2;    // scale slots, one per stage and team (up to 4 groups each)
constexpr int NTB = 2;    // TMEM accumulator buffers, one per unit (2 x 128 columns each)
constexpr int NBR = 2;    // branch-operand stages (one per tile)
constexpr int NTEAM = 64; // threads per expander team
constexpr int NTEAMW = 2; // warps per expander team
constexpr int NEPIW = 8;  // epilogue warps (2 per row quadrant, 64 columns each)
constexpr int A_BYTES = kBM * kGemmKS;            // 16 KB, 128-byte swizzle
constexpr int X_BYTES = kGemmBN * kGemmKS;        // 16 KB, 128-byte swizzle
constexpr int PB_BYTES = kGemmBN * kGemmKS / 2;   // 8 KB packed weights
constexpr int PSX_BYTES = 4 * kBM * 4;            // up to 4 groups x 128 f32 activation scales
constexpr int PCS_BYTES = 4 * kBM * 4;            // up to 4 groups x 128 f32 activation code sums
constexpr int PSW_BYTES = 4 * kGemmBN * 2;        // up to 4 groups x 128 f16 weight scales
constexpr int PSTAGE = PB_BYTES + PSX_BYTES + PCS_BYTES + PSW_BYTES;
constexpr int GSLOT = kGemmBN + 2 * kBM;         // per group: s_w (f32) | s_x | code sums
constexpr int SLOT_FLOATS = 4 * GSLOT;           // one stage (up to 4 groups)

template <int RP>
struct GemmCfg {
  static constexpr int SA = 4;                  // activation stages (TMA -> MMA)
  static constexpr int SP = RP <= 32 ? 6 : 4;   // packed-weight stages (even, see the teams)
  static constexpr int BR_BYTES = RP * kBM * 2;   // p_hat tile (and the B_hat tile), RP/8 boxes of 2 KB
  static constexpr int NBAR = 2 * SA + 2 * SX + 2 * SP + 2 * NSS + 2 * NTB + 2 * NBR + 1;
  static constexpr int SMEM = 1024 + SA * A_BYTES + SX * X_BYTES + SP * PSTAGE + NSS * SLOT_FLOATS * 4 +
                              NBR * 2 * BR_BYTES + NBAR * 8 + 16;
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
__global__ void __launch_bounds__(448, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap qx_map, const __grid_constant__ CUtensorMap qw_map,
                const __grid_constant__ CUtensorMap sx_map, const __grid_constant__ CUtensorMap cs_map,
                const __grid_constant__ CUtensorMap sw_map, const __grid_constant__ CUtensorMap ph_map,
                const __grid_constant__ CUtensorMap bh_map, const GemmArgs a) {
  using Cfg = GemmCfg<RP>;
  constexpr int SP = Cfg::SP;
  constexpr int SA = Cfg::SA;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* aring = smem;                           // SA x 16 KB, 1024-aligned
  uint8_t* xring = aring + SA * A_BYTES;           // SX x 16 KB, 1024-aligned
  uint8_t* pring = xring + SX * X_BYTES;           // SP x (weights packed | s_x | code sums | s_w)
  float* slots = reinterpret_cast<float*>(pring + SP * PSTAGE);
  uint8_t* br = reinterpret_cast<uint8_t*>(slots + NSS * SLOT_FLOATS);  // NBR x (p_hat | B_hat)
  uint64_t* bars = reinterpret_cast<uint64_t*>(br + NBR * 2 * Cfg::BR_BYTES);
  uint64_t* afull = bars;
  uint64_t* aempty = afull + SA;
  uint64_t* xfull = aempty + SA;
  uint64_t* xempty = xfull + SX;
  uint64_t* pfull = xempty + SX;
  uint64_t* pempty = pfull + SP;
  uint64_t* sfull = pempty + SP;
  uint64_t* sempty = sfull + NSS;
  uint64_t* tfull = sempty + NSS;
  uint64_t* tempty = tfull + NTB;
  uint64_t* bfull = tempty + NTB;
  uint64_t* bempty = bfull + NBR;
  uint64_t* drain = bempty + NBR;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + Cfg::NBAR);
  int* abort_flag = reinterpret_cast<int*>(tmem_slot + 1);

  const uint32_t wid = warp_id(), lane = lane_id();
  const int G = a.G;
  const int gps = kGemmKS / G;                    // groups per stage (2 or 4)
  const int ngroups = a.K / G;
  const int nst = (a.K + kGemmKS - 1) / kGemmKS;  // the last stage may be partly past K (zero-filled)
  const int ntiles = a.m_tiles * a.n_tiles;
  const int my_tiles = ntiles > static_cast<int>(blockIdx.x)
                           ? (ntiles - static_cast<int>(blockIdx.x) + static_cast<int>(gridDim.x) - 1) /
                                 static_cast<int>(gridDim.x)
                           : 0;
  auto tile_mn = [&](int i, int& m0, int& n0) {  // i-th tile of this CTA, m-major order
    const int t = static_cast<int>(blockIdx.x) + i * static_cast<int>(gridDim.x);
    m0 = (t / a.n_tiles) * kBM;
    n0 = (t % a.n_tiles) * kGemmBN;
  };

  if (threadIdx.x == 0) {
    for (int i = 0; i < SA; ++i) {
      mbar_init(&afull[i], 1);
      mbar_init(&aempty[i], 1);
    }
    for (int i = 0; i < SX; ++i) {
      mbar_init(&xfull[i], NTEAMW);
      mbar_init(&xempty[i], 1);
    }
    for (int i = 0; i < SP; ++i) {
      mbar_init(&pfull[i], 1);
      mbar_init(&pempty[i], NTEAMW);
    }
    for (int i = 0; i < NSS; ++i) {
      mbar_init(&sfull[i], NTEAMW);
      mbar_init(&sempty[i], NEPIW);
    }
    for (int i = 0; i < NTB; ++i) {
      mbar_init(&tfull[i], 1);
      mbar_init(&tempty[i], NEPIW);
    }
    for (int i = 0; i < NBR; ++i) {
      mbar_init(&bfull[i], 1);
      mbar_init(&bempty[i], 1);
    }
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
      const uint32_t pbytes = PB_BYTES + gps * (kBM * 8 + kGemmBN * 2);
      int sa = 0, sp = 0;  // running stage counters (the same sequence every role walks)
      for (int ti = 0; ti < my_tiles && ok; ++ti) {
        int m0, n0;
        tile_mn(ti, m0, n0);
        if constexpr (RP > 0) {
          const int bs = ti % NBR;
          if (ti >= NBR) ok = mbar_wait(&bempty[bs], ((ti / NBR) & 1) ^ 1, wc);
          if (!ok) break;
          uint8_t* b = br + bs * 2 * Cfg::BR_BYTES;
          mbar_arrive_expect_tx(&bfull[bs], 2 * Cfg::BR_BYTES);
          for (int q = 0; q < RP / 8; ++q) {
            tma_load_2d(b + q * 2048, &ph_map, &bfull[bs], q * 8, m0);
            tma_load_2d(b + Cfg::BR_BYTES + q * 2048, &bh_map, &bfull[bs], q * 8, n0);
          }
        }
        for (int st = 0; st < nst && ok; ++st) {
          // packed weights and the group scales of this stage
          const int ps = sp % SP;
          if (sp >= SP) ok = mbar_wait(&pempty[ps], ((sp / SP) & 1) ^ 1, wc);
          if (!ok) break;
          uint8_t* p = pring + ps * PSTAGE;
          mbar_arrive_expect_tx(&pfull[ps], pbytes);
          tma_load_2d(p, &qw_map, &pfull[ps], st * (kGemmKS / 2), n0);
          tma_load_2d(p + PB_BYTES, &sx_map, &pfull[ps], m0, st * gps);
          tma_load_2d(p + PB_BYTES + PSX_BYTES, &cs_map, &pfull[ps], m0, st * gps);
          tma_load_2d(p + PB_BYTES + PSX_BYTES + PCS_BYTES, &sw_map, &pfull[ps], n0, st * gps);
          ++sp;
          // activation codes of this stage
          const int as = sa % SA;
          if (sa >= SA) ok = mbar_wait(&aempty[as], ((sa / SA) & 1) ^ 1, wc);
          if (!ok) break;
          mbar_arrive_expect_tx(&afull[as], A_BYTES);
          tma_load_2d(aring + as * A_BYTES, &qx_map, &afull[as], st * kGemmKS, m0);
          ++sa;
        }
      }
      // Let every issued load land before the CTA can exit.
      int never = 0;
      const WaitCtl dc{&never, a.err, globaltimer_ns() + a.timeout_ns};
      for (int j = (sp > SP ? sp - SP : 0); j < sp; ++j) mbar_wait(&pfull[j % SP], (j / SP) & 1, dc);
      for (int j = (sa > SA ? sa - SA : 0); j < sa; ++j) mbar_wait(&afull[j % SA], (j / SA) & 1, dc);
    }
  } else if (wid == 1) {
    // ------------------------------------------------------------- MMA issuer
    // The epilogue consumes accumulators in units of two groups (one TMEM buffer of 2 x 128
    // columns); a unit never straddles a stage because a stage holds an even number of groups.
    // One tcgen05 fence per unit: fences and commits cost far more than an MMA issue.
    if (lane == 0) {
      bool ok = true;
      constexpr uint32_t idesc = idesc_e4m3(kBM, kGemmBN);
      int s = 0, u_all = 0;  // running stage and accumulator-unit counters
      for (int ti = 0; ti < my_tiles && ok; ++ti) {
        for (int st = 0; st < nst && ok; ++st, ++s) {
          const int gn = (st * gps + gps <= ngroups) ? gps : ngroups - st * gps;  // groups in this stage
          const int as = s % SA, xs = s % SX;
          ok = mbar_wait(&afull[as], (s / SA) & 1, wc);
          if (ok) ok = mbar_wait(&xfull[xs], (s / SX) & 1, wc);
          if (!ok) break;
          const uint32_t aa = smem_u32(aring + as * A_BYTES), xa = smem_u32(xring + xs * X_BYTES);
          for (int g0 = 0; g0 < gn && ok; g0 += 2, ++u_all) {
            const int ub = u_all % NTB;
            if (u_all >= NTB) ok = mbar_wait(&tempty[ub], ((u_all / NTB) & 1) ^ 1, wc);
            if (!ok) break;
            tc_fence_after();
            for (int gi = g0; gi < gn && gi < g0 + 2; ++gi)
              for (int kk = 0; kk < G / 32; ++kk) {
                const uint32_t off = static_cast<uint32_t>((gi * (G / 32) + kk) * 32);
                mma_f8f6f4(tmem + ub * 256 + (gi - g0) * 128, smem_desc(aa + off, 16, 1024, kSw128),
                           smem_desc(xa + off, 16, 1024, kSw128), idesc, kk != 0);
              }
            mma_commit(&tfull[ub]);
          }
          mma_commit(&aempty[as]);
          mma_commit(&xempty[xs]);
        }
        if constexpr (RP > 0) {
          const int bs = ti % NBR, ub = u_all % NTB;
          if (ok) ok = mbar_wait(&bfull[bs], (ti / NBR) & 1, wc);
          if (ok && u_all >= NTB) ok = mbar_wait(&tempty[ub], ((u_all / NTB) & 1) ^ 1, wc);
          if (ok) {
            tc_fence_after();
            constexpr uint32_t idesc_br = idesc_f16(kBM, kGemmBN);
            const uint32_t pa = smem_u32(br + bs * 2 * Cfg::BR_BYTES), pb = pa + Cfg::BR_BYTES;
#pragma unroll
            for (int kk = 0; kk < RP / 16; ++kk)
              mma_f16(tmem + ub * 256, smem_desc(pa + kk * 4096, 2048, 128, kSwNone),
                      smem_desc(pb + kk * 4096, 2048, 128, kSwNone), idesc_br, kk != 0);
            mma_commit(&tfull[ub]);
            mma_commit(&bempty[bs]);
            ++u_all;
          }
        }
      }
      mma_commit(drain);
      int never = 0;
      const WaitCtl dc{&never, a.err, globaltimer_ns() + a.timeout_ns};
      mbar_wait(drain, 0, dc);
    }
    __syncwarp();
  } else if (wid < 6) {
    // ------------------------------------------------------------- weight expanders + scales
    // Team t (warps 2+2t, 3+2t) takes the stages s with s % 2 == t.  Thread e (0..63) of a team
    // owns the 16-byte chunk j = e % 8 of rows e/8 + 8 i (i = 0..15): its source and destination
    // offsets only step by constants (512 and 1024 bytes).
    const int team = (static_cast<int>(wid) - 2) >> 1;
    const int e = (static_cast<int>(threadIdx.x) - 64) & (NTEAM - 1);
    const int r0 = e >> 3, j = e & 7;
    const int src0 = r0 * 64 + j * 8;
    const int dst0 = r0 * 128 + ((j ^ r0) << 4);
    const uint32_t kX8 = 0x88888888u;
    bool ok = true;
    int s = 0;
    for (int ti = 0; ti < my_tiles && ok; ++ti) {
      for (int st = 0; st < nst && ok; ++st, ++s) {
        if ((s & 1) != team) continue;
        const int gn = (st * gps + gps <= ngroups) ? gps : ngroups - st * gps;  // groups in this stage
        const int ps = s % SP, xs = team;
        ok = mbar_wait(&pfull[ps], (s / SP) & 1, wc);
        if (ok && s >= SX) ok = mbar_wait(&xempty[xs], ((s / SX) & 1) ^ 1, wc);
        if (!ok) break;
        const uint8_t* p = pring + ps * PSTAGE;
        uint8_t* xb = xring + xs * X_BYTES;
        uint2 pkd[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) pkd[i] = *reinterpret_cast<const uint2*>(p + src0 + i * 512);
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          uint4 o;
          o.x = (pkd[i].x ^ kX8) & 0x0F0F0F0Fu;
          o.y = ((pkd[i].x >> 4) ^ kX8) & 0x0F0F0F0Fu;
          o.z = (pkd[i].y ^ kX8) & 0x0F0F0F0Fu;
          o.w = ((pkd[i].y >> 4) ^ kX8) & 0x0F0F0F0Fu;
          *reinterpret_cast<uint4*>(xb + dst0 + i * 1024) = o;
        }
        fence_proxy_async_smem();
        warp_arrive(&xfull[xs]);
        // group scales of this stage -> the team's float32 scale slot for the epilogue
        const float* psx = reinterpret_cast<const float*>(p + PB_BYTES);
        const float* pcs = reinterpret_cast<const float*>(p + PB_BYTES + PSX_BYTES);
        const __half* psw = reinterpret_cast<const __half*>(p + PB_BYTES + PSX_BYTES + PCS_BYTES);
        const int ss = team;
        if (s >= NSS) ok = mbar_wait(&sempty[ss], ((s / NSS) & 1) ^ 1, wc);
        if (!ok) break;
        float* slot = slots + ss * SLOT_FLOATS;
        for (int gi = 0; gi < gn; ++gi) {
          float* sg = slot + gi * GSLOT;
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const int i = e + NTEAM * h;
            sg[i] = __half2float(psw[gi * kGemmBN + i]);
            sg[kGemmBN + i] = psx[gi * kBM + i];
            sg[kGemmBN + kBM + i] = pcs[gi * kBM + i];
          }
        }
        warp_arrive(&sfull[ss]);
        fence_proxy_async_smem();  // reads of the packed stage before the TMA refills it
        warp_arrive(&pempty[ps]);
      }
    }
  } else {
    // ------------------------------------------------------------- epilogue
    // Warps 6..13: warp w reads TMEM lanes 32*(w%4).. (its quadrant of rows) and the 64 output
    // columns [64*((w-6)/4), +64).
    const int quad = wid & 3;
    const int row = quad * 32 + static_cast<int>(lane);
    const int col0 = 64 * ((static_cast<int>(wid) - 6) >> 2);
    const uint32_t tlane = tmem + (static_cast<uint32_t>(quad * 32) << 16) + col0;
    bool ok = true;
    int u_all = 0, s = 0;  // accumulator-unit and stage counters
    for (int ti = 0; ti < my_tiles; ++ti) {
      int m0, n0;
      tile_mn(ti, m0, n0);
      f2 acc[32];
#pragma unroll
      for (int i = 0; i < 32; ++i) acc[i] = 0ull;
      for (int st = 0; st < nst; ++st, ++s) {
        const int gn = (st * gps + gps <= ngroups) ? gps : ngroups - st * gps;  // groups in this stage
        const int ss = s % NSS;
        if (ok) ok = mbar_wait(&sfull[ss], (s / NSS) & 1, wc);
        const float* slot = slots + ss * SLOT_FLOATS;
        for (int g0 = 0; g0 < gn; g0 += 2, ++u_all) {
          const int ub = u_all % NTB;
          const int nmem = (g0 + 1 < gn) ? 2 : 1;
          if (ok) ok = mbar_wait(&tfull[ub], (u_all / NTB) & 1, wc);
          tc_fence_after();
          for (int mi = 0; mi < nmem; ++mi) {
            const float* sg = slot + (g0 + mi) * GSLOT;
            const float sxv = sg[kGemmBN + row];
            const float alpha = sxv * 262144.0f;                       // 2^18 s_x (exact)
            const float beta = -8.0f * sxv * sg[kGemmBN + kBM + row];  // -8 s_x S_a
            const f2 al2 = pk(alpha, alpha), be2 = pk(beta, beta);
#pragma unroll
            for (int c = 0; c < 2; ++c) {
              uint32_t v[32];
              tmem_ld32(tlane + ub * 256 + mi * 128 + c * 32, v);
              tmem_ld_wait();
              if (mi == nmem - 1 && c == 1) {
                tc_fence_before();
                warp_arrive(&tempty[ub]);
              }
              const float4* w4 = reinterpret_cast<const float4*>(sg + col0 + c * 32);
#pragma unroll
              for (int i4 = 0; i4 < 8; ++i4) {
                const float4 w = w4[i4];
                const f2 t0 = fma2(pku(v[4 * i4], v[4 * i4 + 1]), al2, be2);
                const f2 t1 = fma2(pku(v[4 * i4 + 2], v[4 * i4 + 3]), al2, be2);
                acc[16 * c + 2 * i4] = fma2(t0, pk(w.x, w.y), acc[16 * c + 2 * i4]);
                acc[16 * c + 2 * i4 + 1] = fma2(t1, pk(w.z, w.w), acc[16 * c + 2 * i4 + 1]);
              }
            }
          }
        }
        warp_arrive(&sempty[ss]);
      }
      if constexpr (RP > 0) {
        const int ub = u_all % NTB;
        if (ok) ok = mbar_wait(&tfull[ub], (u_all / NTB) & 1, wc);
        tc_fence_after();
#pragma unroll
        for (int c = 0; c < 2; ++c) {
          uint32_t v[32];
          tmem_ld32(tlane + ub * 256 + c * 32, v);
          tmem_ld_wait();
#pragma unroll
          for (int i = 0; i < 16; ++i) acc[16 * c + i] = add2(acc[16 * c + i], pku(v[2 * i], v[2 * i + 1]));
        }
        tc_fence_before();
        warp_arrive(&tempty[ub]);
        ++u_all;
      }
      const int m = m0 + row;
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
  a.m_tiles = (M + kBM - 1) / kBM;
  a.n_tiles = (h.N + kGemmBN - 1) / kGemmBN;
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
  const int ntiles = a.m_tiles * a.n_tiles;
  const int grid = ntiles < h.num_sms ? ntiles : h.num_sms;
  const CUtensorMap& ph = (RP > 0) ? am.ph_map : am.qx_map;
  const CUtensorMap& bh = (RP > 0) ? h.Bh_map : am.qx_map;
  gemm_kernel<RP><<<grid, 448, Cfg::SMEM, s>>>(am.qx_map, h.qw_map, am.sx_map, am.cs_map, h.sw_map, ph, bh, a);
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
