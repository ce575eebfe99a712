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
// runs continuously across tiles, so loads for the next tile overlap the epilogue of the current
// one.  384 threads in three warpgroups (kEpiWarpsPerQuad = 2; 4 gives 640 threads):
//   warpgroup 0 (80 registers): warp 0 TMA producer, warp 1 MMA issuer and TMEM owner, warps 2-3
//     expand weight nibbles into the operand stage;
//   warpgroups 1-2 (208 registers): warps 4..11 epilogue.  A warp owns 32 rows x 64 columns of
//     the tile; TMEM is read with the 16x256b shape, so a thread holds 4 rows x 16 columns (as
//     packed f32x2 pairs) and, per group, loads 16 column scales s_w and the constants
//     (alpha, beta) of its 4 rows, which kernel (a) wrote.  With one row per
//     thread, moving the scales into registers cost as much as the arithmetic; here the floor is
//     the FMA pipe, two operations per output and group, and the issue of everything around it.
// Rings (each waiter waits for every phase of its slots in turn):
//   O  operand stage = activation codes (TMA) + expanded weights (expanders)  -> MMA     SO slots
//   P  packed weights of a stage  TMA -> expanders                                      SP slots
//   S  alpha, beta, s_w of eight groups  TMA -> epilogue                                SS slots
//   T  TMEM accumulators, units of two groups (2 x 128 columns)  MMA -> epilogue        NTB units
//   B  p_hat / B_hat tiles  TMA -> MMA, loaded after the tile's stages                   one per tile
// Every barrier operation costs on the order of 100 cycles, so each role touches as few as
// possible per stage: the MMA warp waits twice and commits twice, the expanders wait twice and
// arrive twice, the epilogue waits once and arrives once per unit, plus once each per S slot.
#include "internal.h"
#include "ptx.cuh"

namespace qwam {
namespace {

struct GemmArgs {
  int M, N, K, G;
  int m_tiles, n_tiles;
  void* Y;
  int y_f32;
  const float* bias;  // optional [N], added to the float32 result before it is stored
  int* err;
  uint64_t timeout_ns;
};

constexpr int kEpiWarpsPerQuad = 2;                 // epilogue warps per 32-row quadrant (2 or 4)
constexpr int CBW = 4 / kEpiWarpsPerQuad;           // 32-column blocks per epilogue warp
constexpr int kThreads = 128 + 128 * kEpiWarpsPerQuad;
constexpr int kLaunchRegs = kEpiWarpsPerQuad == 4 ? 96 : 168;  // 65536 / threads, multiple of 8
constexpr int kRegsCtl = kEpiWarpsPerQuad == 4 ? 56 : 80;     // warpgroup 0
constexpr int kRegsEpi = kEpiWarpsPerQuad == 4 ? 104 : 208;   // the epilogue warpgroups
static_assert(128 * kRegsCtl + (kThreads - 128) * kRegsEpi <= kThreads * kLaunchRegs,
              "register split above the launch allocation");
constexpr int SO = 3;     // operand stages
constexpr int SP = 6;     // packed-weight stages
constexpr int SS = 3;     // scale stages (kScaleGroups groups each)
constexpr int NTB = 2;    // TMEM accumulator units (2 x 128 columns each)
constexpr int NBR = 1;    // branch-operand stages (one per tile)
constexpr int NXW = 2;    // expander warps
constexpr int NEPIW = 4 * kEpiWarpsPerQuad;  // epilogue warps (32 * CBW columns each)
constexpr int A_BYTES = kBM * kGemmKS;            // 16 KB, 128-byte swizzle
constexpr int X_BYTES = kGemmBN * kGemmKS;        // 16 KB, 128-byte swizzle
constexpr int OSTAGE = A_BYTES + X_BYTES;
constexpr int PB_BYTES = kGemmBN * kGemmKS / 2;   // 8 KB packed weights
constexpr int PSTAGE = PB_BYTES;
constexpr int SAB_BYTES = kScaleGroups * 128 * 8;  // 8 groups x 128 rows x (alpha, beta)
constexpr int SSW_BYTES = kScaleGroups * 128 * 4;  // 8 groups x 128 f32 s_w
constexpr int SSTAGE = SAB_BYTES + SSW_BYTES;      // 12 KB

template <int RP>
struct GemmCfg {
  static constexpr int BR_BYTES = RP * kBM * 2;   // p_hat tile (and the B_hat tile), RP/8 boxes of 2 KB
  static constexpr int NBAR = 2 * SO + 2 * SP + 2 * SS + 2 * NTB + 2 * NBR + 1;
  static constexpr int SMEM = 1024 + SO * OSTAGE + SP * PSTAGE + SS * SSTAGE + NBR * 2 * BR_BYTES + NBAR * 8 + 16;
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
__global__ void __launch_bounds__(kThreads, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap qx_map, const __grid_constant__ CUtensorMap qw_map,
                const __grid_constant__ CUtensorMap ab_map, const __grid_constant__ CUtensorMap sw_map, const __grid_constant__ CUtensorMap ph_map,
                const __grid_constant__ CUtensorMap bh_map, const GemmArgs a) {
  using Cfg = GemmCfg<RP>;
  extern __shared__ uint8_t smem_raw[];
  pdl_launch_dependents();
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* oring = smem;                           // SO x (A 16 KB | X 16 KB), 1024-aligned
  uint8_t* pring = oring + SO * OSTAGE;            // SP x packed weights
  uint8_t* sring = pring + SP * PSTAGE;            // SS x ((alpha, beta) | s_w)
  uint8_t* br = sring + SS * SSTAGE;               // NBR x (p_hat | B_hat)
  uint64_t* bars = reinterpret_cast<uint64_t*>(br + NBR * 2 * Cfg::BR_BYTES);
  uint64_t* ofull = bars;
  uint64_t* oempty = ofull + SO;
  uint64_t* pfull = oempty + SO;
  uint64_t* pempty = pfull + SP;
  uint64_t* sfull = pempty + SP;
  uint64_t* sempty = sfull + SS;
  uint64_t* tfull = sempty + SS;
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
  auto groups_in = [&](int st) { return (st * gps + gps <= ngroups) ? gps : ngroups - st * gps; };
  // A scale stage starts with every K stage whose first group is a multiple of kScaleGroups
  // (gps divides kScaleGroups) and ends with the K stage that reaches the next one, or K.
  auto scale_starts = [&](int st) { return (st * gps) % kScaleGroups == 0; };
  auto scale_ends = [&](int st) { return ((st + 1) * gps) % kScaleGroups == 0 || st + 1 == nst; };

  if (threadIdx.x == 0) {
    for (int i = 0; i < SO; ++i) {
      mbar_init(&ofull[i], 1 + NXW);  // the producer's expect-tx arrival + one per expander warp
      mbar_init(&oempty[i], 1);
    }
    for (int i = 0; i < SP; ++i) {
      mbar_init(&pfull[i], 1);
      mbar_init(&pempty[i], NXW);
    }
    for (int i = 0; i < SS; ++i) {
      mbar_init(&sfull[i], 1);
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
  pdl_wait();  // every global access of this kernel comes after the previous kernel's

  if (wid < 4) {
    setmaxnreg_dec<kRegsCtl>();
    if (wid == 0) {
      // ----------------------------------------------------------- TMA producer
      // The whole warp walks the loop (so addresses, coordinates and barrier phases are
      // warp-uniform and stay in uniform registers); one elected lane issues each copy.
      bool ok = true;
      int s = 0, ss = 0;  // running K-stage and scale-stage counters (every role walks the same)
      for (int ti = 0; ti < my_tiles && ok; ++ti) {
        int m0, n0;
        tile_mn(ti, m0, n0);
        for (int st = 0; st < nst && ok; ++st, ++s) {
          if (scale_starts(st)) {
            // (alpha, beta) and s_w of the next kScaleGroups groups (zero-filled past K)
            const int sb = ss % SS;
            if (ss >= SS) ok = mbar_wait_inline(&sempty[sb], ((ss / SS) & 1) ^ 1, wc);
            if (!ok) break;
            uint8_t* q = sring + sb * SSTAGE;
            if (elect_one()) {
              mbar_arrive_expect_tx(&sfull[sb], SSTAGE);
              tma_load_2d(q, &ab_map, &sfull[sb], 2 * m0, st * gps);
              tma_load_2d(q + SAB_BYTES, &sw_map, &sfull[sb], n0, st * gps);
            }
            __syncwarp();
            ++ss;
          }
          // packed weights of this stage
          const int ps = s % SP;
          if (s >= SP) ok = mbar_wait_inline(&pempty[ps], ((s / SP) & 1) ^ 1, wc);
          if (!ok) break;
          uint8_t* p = pring + ps * PSTAGE;
          if (elect_one()) {
            mbar_arrive_expect_tx(&pfull[ps], PB_BYTES);
            tma_load_2d(p, &qw_map, &pfull[ps], st * (kGemmKS / 2), n0);
          }
          __syncwarp();
          // activation codes of this stage
          const int os = s % SO;
          if (s >= SO) ok = mbar_wait_inline(&oempty[os], ((s / SO) & 1) ^ 1, wc);
          if (!ok) break;
          if (elect_one()) {
            mbar_arrive_expect_tx(&ofull[os], A_BYTES);
            tma_load_2d(oring + os * OSTAGE, &qx_map, &ofull[os], st * kGemmKS, m0);
          }
          __syncwarp();
        }
        if constexpr (RP > 0) {
          // the branch operands are needed only after the tile's last stage
          const int bs = ti % NBR;
          if (ok && ti >= NBR) ok = mbar_wait_inline(&bempty[bs], ((ti / NBR) & 1) ^ 1, wc);
          if (!ok) break;
          uint8_t* b = br + bs * 2 * Cfg::BR_BYTES;
          if (elect_one()) {
            mbar_arrive_expect_tx(&bfull[bs], 2 * Cfg::BR_BYTES);
            for (int q = 0; q < RP / 8; ++q) {
              tma_load_2d(b + q * 2048, &ph_map, &bfull[bs], q * 8, m0);
              tma_load_2d(b + Cfg::BR_BYTES + q * 2048, &bh_map, &bfull[bs], q * 8, n0);
            }
          }
          __syncwarp();
        }
      }
      // Let every issued load land before the CTA can exit (these phases complete in the
      // normal course; after an abort the waits end at the deadline).
      int never = 0;
      const WaitCtl dc{&never, a.err, globaltimer_ns() + a.timeout_ns};
      for (int j = (s > SP ? s - SP : 0); j < s; ++j) mbar_wait_inline(&pfull[j % SP], (j / SP) & 1, dc);
      for (int j = (ss > SS ? ss - SS : 0); j < ss; ++j) mbar_wait_inline(&sfull[j % SS], (j / SS) & 1, dc);
      // An operand stage also needs the expanders' arrivals: in the normal course they come;
      // after an abort the wait ends at the deadline, long after the tile has landed.
      for (int j = (s > SO ? s - SO : 0); j < s; ++j) mbar_wait_inline(&ofull[j % SO], (j / SO) & 1, dc);
      if constexpr (RP > 0) {
        for (int t = (my_tiles > NBR ? my_tiles - NBR : 0); t < my_tiles; ++t)
          mbar_wait_inline(&bfull[t % NBR], (t / NBR) & 1, dc);
      }
    } else if (wid == 1) {
      // ----------------------------------------------------------- MMA issuer
      // The epilogue consumes accumulators in units of two groups (one TMEM buffer of 2 x 128
      // columns); a unit never straddles a stage because a full stage holds an even number of
      // groups.  The whole warp walks the loop and forms the descriptors (warp-uniform values);
      // one elected lane (the same one throughout, as the commits track its MMAs) issues.
      bool ok = true;
      constexpr uint32_t idesc = idesc_e4m3(kBM, kGemmBN);
      int s = 0, u_all = 0;  // running stage and accumulator-unit counters
      for (int ti = 0; ti < my_tiles && ok; ++ti) {
        for (int st = 0; st < nst && ok; ++st, ++s) {
          const int gn = groups_in(st);
          const int os = s % SO;
          ok = mbar_wait_inline(&ofull[os], (s / SO) & 1, wc);
          if (!ok) break;
          const uint32_t aa = smem_u32(oring + os * OSTAGE), xa = aa + A_BYTES;
          const uint64_t adesc0 = smem_desc(aa, 16, 1024, kSw128), xdesc0 = smem_desc(xa, 16, 1024, kSw128);
          for (int g0 = 0; g0 < gn && ok; g0 += 2, ++u_all) {
            const int ub = u_all % NTB;
            if (u_all >= NTB) ok = mbar_wait_inline(&tempty[ub], ((u_all / NTB) & 1) ^ 1, wc);
            if (!ok) break;
            tc_fence_after();
            const int g1 = (g0 + 2 < gn) ? g0 + 2 : gn;
            if (elect_one()) {
              for (int gi = g0; gi < g1; ++gi)
                for (int kk = 0; kk < G / 32; ++kk) {
                  const uint64_t off = static_cast<uint64_t>((gi * (G / 32) + kk) * 32) >> 4;  // 16-byte units
                  mma_f8f6f4(tmem + ub * 256 + (gi - g0) * 128, adesc0 + off, xdesc0 + off, idesc, kk != 0);
                }
              mma_commit(&tfull[ub]);
            }
            __syncwarp();
          }
          if (elect_one()) mma_commit(&oempty[os]);
          __syncwarp();
        }
        if constexpr (RP > 0) {
          const int bs = ti % NBR, ub = u_all % NTB;
          if (ok) ok = mbar_wait_inline(&bfull[bs], (ti / NBR) & 1, wc);
          if (ok && u_all >= NTB) ok = mbar_wait_inline(&tempty[ub], ((u_all / NTB) & 1) ^ 1, wc);
          if (ok) {
            tc_fence_after();
            constexpr uint32_t idesc_br = idesc_f16(kBM, kGemmBN);
            const uint32_t pa = smem_u32(br + bs * 2 * Cfg::BR_BYTES), pb = pa + Cfg::BR_BYTES;
            const uint64_t pdesc0 = smem_desc(pa, 2048, 128, kSwNone), bdesc0 = smem_desc(pb, 2048, 128, kSwNone);
            if (elect_one()) {
#pragma unroll
              for (int kk = 0; kk < RP / 16; ++kk)
                mma_f16(tmem + ub * 256, pdesc0 + kk * 256, bdesc0 + kk * 256, idesc_br, kk != 0);  // 4096 B
              mma_commit(&tfull[ub]);
              mma_commit(&bempty[bs]);
            }
            __syncwarp();
            ++u_all;
          }
        }
      }
      if (elect_one()) mma_commit(drain);
      __syncwarp();
      int never = 0;
      const WaitCtl dc{&never, a.err, globaltimer_ns() + a.timeout_ns};
      mbar_wait_inline(drain, 0, dc);
    } else {
      // ----------------------------------------------------------- weight expanders
      // Thread e (0..63) owns the 16-byte chunk j = e % 8 of rows e/8 + 8 i (i = 0..15): its source
      // and destination offsets only step by constants (512 and 1024 bytes).
      const int e = static_cast<int>(threadIdx.x) - 64;
      const int r0 = e >> 3, j = e & 7;
      const int src0 = r0 * 64 + j * 8;
      const int dst0 = r0 * 128 + ((j ^ r0) << 4);
      const uint32_t kX8 = 0x88888888u;
      bool ok = true;
      int s = 0;
      for (int ti = 0; ti < my_tiles && ok; ++ti) {
        for (int st = 0; st < nst && ok; ++st, ++s) {
          const int ps = s % SP, os = s % SO;
          ok = mbar_wait_inline(&pfull[ps], (s / SP) & 1, wc);
          if (ok && s >= SO) ok = mbar_wait_inline(&oempty[os], ((s / SO) & 1) ^ 1, wc);
          if (!ok) break;
          const uint8_t* p = pring + ps * PSTAGE;
          uint8_t* xb = oring + os * OSTAGE + A_BYTES;
#pragma unroll
          for (int h8 = 0; h8 < 16; h8 += 8) {
            uint2 pkd[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) pkd[i] = *reinterpret_cast<const uint2*>(p + src0 + (h8 + i) * 512);
#pragma unroll
            for (int i = 0; i < 8; ++i) {
              uint4 o;
              o.x = (pkd[i].x ^ kX8) & 0x0F0F0F0Fu;
              o.y = ((pkd[i].x >> 4) ^ kX8) & 0x0F0F0F0Fu;
              o.z = (pkd[i].y ^ kX8) & 0x0F0F0F0Fu;
              o.w = ((pkd[i].y >> 4) ^ kX8) & 0x0F0F0F0Fu;
              *reinterpret_cast<uint4*>(xb + dst0 + (h8 + i) * 1024) = o;
            }
          }
          // Orders the generic writes of the expanded weights before the MMA reads them, and the
          // generic reads of the packed stage before TMA refills it.
          fence_proxy_async_smem();
          warp_arrive(&ofull[os]);
          if (lane == 0) mbar_arrive(&pempty[ps]);
        }
      }
    }
  } else {
    setmaxnreg_inc<kRegsEpi>();
    // ------------------------------------------------------------- epilogue
    // Warp w reads TMEM lanes 32*(w%4).. (its quadrant of rows) and the 32 CBW output columns
    // from 32 CBW ((w-4)/4).  Thread t holds rows rq + 8k (k = 0..3, rq = t/4 within the
    // quadrant) and, in each 32-column block cb, columns 8j + 2 cq + {0, 1} (j = 0..3,
    // cq = t % 4): acc[16 cb + 4k + j] is that pair.
    const int quad = wid & 3;
    const int col0 = 32 * CBW * ((static_cast<int>(wid) - 4) >> 2);
    const int rq = static_cast<int>(lane) >> 2, cq = static_cast<int>(lane) & 3;
    const int rbase = quad * 32 + rq;
    const uint32_t tq = tmem + (static_cast<uint32_t>(quad * 32) << 16) + col0;
    bool ok = true;
    int u_all = 0, s = 0, ss = 0;  // accumulator-unit, K-stage and scale-stage counters
    for (int ti = 0; ti < my_tiles; ++ti) {
      int m0, n0;
      tile_mn(ti, m0, n0);
      f2 acc[16 * CBW];
#pragma unroll
      for (int i = 0; i < 16 * CBW; ++i) acc[i] = 0ull;
      for (int st = 0; st < nst; ++st, ++s) {
        const int gn = groups_in(st);
        const int sb = ss % SS;
        if (scale_starts(st) && ok) ok = mbar_wait_inline(&sfull[sb], (ss / SS) & 1, wc);
        const int gl0 = (st * gps) % kScaleGroups;  // the stage's first group within the scale stage
        const float2* pab = reinterpret_cast<const float2*>(sring + sb * SSTAGE) + gl0 * 128;
        const float* psw = reinterpret_cast<const float*>(sring + sb * SSTAGE + SAB_BYTES) + gl0 * 128;
        for (int g0 = 0; g0 < gn; g0 += 2, ++u_all) {
          const int ub = u_all % NTB;
          const int nmem = (g0 + 1 < gn) ? 2 : 1;
          if (ok) ok = mbar_wait_inline(&tfull[ub], (u_all / NTB) & 1, wc);
          tc_fence_after();
          for (int mi = 0; mi < nmem; ++mi) {
            const int gi = g0 + mi;
            uint32_t v0[CBW][16], v1[CBW][16];
#pragma unroll
            for (int cb = 0; cb < CBW; ++cb) {
              tmem_ld16x256_x4(tq + ub * 256 + mi * 128 + 32 * cb, v0[cb]);
              tmem_ld16x256_x4(tq + (16u << 16) + ub * 256 + mi * 128 + 32 * cb, v1[cb]);
            }
            float2 abr[4];  // (alpha, beta) of rows rbase + 8k
#pragma unroll
            for (int k = 0; k < 4; ++k) abr[k] = pab[gi * 128 + rbase + 8 * k];
            f2 sw2[4 * CBW];
#pragma unroll
            for (int j = 0; j < 4 * CBW; ++j)
              sw2[j] = *reinterpret_cast<const f2*>(psw + gi * 128 + col0 + 8 * j + 2 * cq);
            f2 d[CBW][16];  // d[cb][8h + 2j + rr] = columns (8j + 2cq, +1) of row rq + 16h + 8rr
#pragma unroll
            for (int cb = 0; cb < CBW; ++cb) tmem_ld_wait_pairs(v0[cb], v1[cb], d[cb]);
            if (mi == nmem - 1) {
              tc_fence_before();
              warp_arrive(&tempty[ub]);  // every load of the unit has landed
            }
            // acc += (alpha D + beta) * s_w, alpha = 2^18 s_x, beta = -8 s_x S_a (from kernel (a))
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              const f2 al2 = dup2(abr[k].x), be2 = dup2(abr[k].y);
#pragma unroll
              for (int cb = 0; cb < CBW; ++cb)
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                  const f2 t = fma2(d[cb][8 * (k >> 1) + 2 * j + (k & 1)], al2, be2);
                  acc[16 * cb + 4 * k + j] = fma2(t, sw2[4 * cb + j], acc[16 * cb + 4 * k + j]);
                }
            }
          }
        }
        if (scale_ends(st)) {
          fence_proxy_async_smem();  // reads of the TMA-written scales before the slot is refilled
          warp_arrive(&sempty[sb]);
          ++ss;
        }
      }
      if constexpr (RP > 0) {
        const int ub = u_all % NTB;
        if (ok) ok = mbar_wait_inline(&tfull[ub], (u_all / NTB) & 1, wc);
        tc_fence_after();
#pragma unroll
        for (int cb = 0; cb < CBW; ++cb) {
          uint32_t v0[16], v1[16];
          tmem_ld16x256_x4(tq + ub * 256 + 32 * cb, v0);
          tmem_ld16x256_x4(tq + (16u << 16) + ub * 256 + 32 * cb, v1);
          f2 d[16];
          tmem_ld_wait_pairs(v0, v1, d);
#pragma unroll
          for (int k = 0; k < 4; ++k)
#pragma unroll
            for (int j = 0; j < 4; ++j)
              acc[16 * cb + 4 * k + j] = add2(acc[16 * cb + 4 * k + j], d[8 * (k >> 1) + 2 * j + (k & 1)]);
        }
        tc_fence_before();
        warp_arrive(&tempty[ub]);
        ++u_all;
      }
      if (ok) {
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const int m = m0 + rbase + 8 * k;
          if (m >= a.M) continue;
#pragma unroll
          for (int cb = 0; cb < CBW; ++cb)
#pragma unroll
            for (int j = 0; j < 4; ++j) {
              const int n = n0 + col0 + 32 * cb + 8 * j + 2 * cq;  // even; N is a multiple of 8
              if (n >= a.N) continue;
              const size_t off = static_cast<size_t>(m) * a.N + n;
              const f2 y = acc[16 * cb + 4 * k + j];
              float y0 = lo_f(y), y1 = hi_f(y);
              if (a.bias) {
                const float2 bb = *reinterpret_cast<const float2*>(a.bias + n);
                y0 += bb.x;
                y1 += bb.y;
              }
              if (a.y_f32) {
                *reinterpret_cast<float2*>(static_cast<float*>(a.Y) + off) = make_float2(y0, y1);
              } else {
                *reinterpret_cast<__nv_bfloat162*>(static_cast<__nv_bfloat16*>(a.Y) + off) =
                    __floats2bfloat162_rn(y0, y1);
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
  a.bias = h.bias;
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
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = Cfg::SMEM;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, gemm_kernel<RP>, am.qx_map, h.qw_map, am.ab_map, h.sw32_map, ph, bh, a);
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
