// gemm.cu -- kernel (b): the 4-bit deflated path of Eq. (asp) with the 16-bit branch fused into
// the same kernel (Sec. 4.2; App. B.1 describes the paper's GEMM as one that keeps the weights
// packed at 4 bits and adds the protected branch in its epilogue).
//
//   Y[m, n] = sum_g s_x[m, g] s_w[g, n] P_g[m, n]  +  sum_j p_hat[m, j] B_hat[n, j]
//   P_g[m, n] = sum_{k in group g} q_x[m, k] q_w[n, k]          (exact integers)
//
// sm_103a has no integer tensor-core MMA, so both operands go to tcgen05.mma.kind::f8f6f4 as
// E4M3 bytes of c * 2^-9 (sign | |c|: E4M3 subnormals, which the tensor core keeps exactly).  One
// group's float32 accumulator then holds D = 2^-18 P_g exactly (every partial sum is an integer
// below 2^13 times 2^-18).  The epilogue accumulates s_x s_w P_g as (D s_x) sigma, where
// sigma = 2^18 s_w is the handle's float32 copy of the weight scale: two float32 roundings per
// output and group, the float32 running sum a third.
//
// Both operands stay packed at 4 bits in HBM (SM4 words, see sm4_pack) and are expanded to bytes
// in shared memory: lo = w & 0x87878787 (k = 8j..8j+3), hi = rotr(w, 4) & 0x87878787 (k = 8j+4..).
//
// Persistent CTAs (one per SM) walk output tiles of 128 x 128 with a static stride (row-block
// major, so the CTAs working at one time share the activation rows in L2).  Every ring runs
// continuously across tiles.  384 threads:
//   warp 0        TMA producer: packed codes of both operands per stage, scale slots;
//   warp 1        MMA issuer and TMEM owner;
//   warps 2, 3    expanders: packed stage -> byte operand stage (128-byte swizzle);
//   warps 4..11   epilogue: warp 4 + 4h + q reads TMEM lane quadrant q, columns 64h .. 64h + 63.
// Stages cover 128 K (two groups of 64 or four of 32).  After a tile's K stages come r_pad / 32
// branch stages: the producer brings 32 columns of p_hat and B_hat (float16) through the same
// packed ring, the expanders copy them into the operand layout, and the MMA issuer runs two
// kind::f16 MMAs (K = 16 each); the branch accumulates in its own TMEM unit, which the epilogue
// adds with scale 1.  Any r_pad works.
// TMEM holds four units of 128 columns, one group each (unit g mod 4), so the MMA issuer runs up
// to four groups ahead of the epilogue.  An mbarrier wait costs on the order of a hundred cycles
// even when its phase has completed, so each role waits as little as possible: the MMA issuer
// once per stage for its operands and once for the last TMEM unit the stage writes (the epilogue
// releases units in order); each epilogue warp once per group, for the unit after the one it is
// about to compute (its TMEM loads are double-buffered across groups, so a group's load latency
// overlaps the arithmetic of the previous one).
// Rings (every wait is bounded):
//   P  packed stage (A and B codes, or p_hat / B_hat)   TMA -> expanders          SP slots
//   O  operand stage (A and B bytes)                    expanders -> MMA          SO slots
//   S  scale slot: s_x and sigma of kSG groups           TMA -> epilogue           SS slots
//   T  TMEM units                                       MMA -> epilogue           4 units
#include "internal.h"
#include "ptx.cuh"

namespace qwam {
namespace {

struct GemmArgs {
  int M, N, K;
  int nbs;  // branch stages per tile (r_pad / 32, rounded up)
  int m_tiles, n_tiles;
  void* Y;
  int y_f32;
  const float* bias;  // optional [N], added to the float32 result before it is stored
  int* err;
  uint64_t timeout_ns;
};

constexpr int kBN = 128;       // output columns per tile
constexpr int kKS = 128;       // K per stage (128 codes: 64 packed bytes, 128 operand bytes per row)
constexpr int kSG = 8;         // groups per scale slot
constexpr int kNX = 2;         // expander warps
constexpr int kThreads = 384;  // 12 warps
constexpr int kLaunchRegs = 168;
constexpr int kRegsCtl = 48;   // warpgroup 0 (producer, MMA, expanders)
constexpr int kRegsEpi = 224;  // warpgroups 1-2 (epilogue)
static_assert(128 * kRegsCtl + 256 * kRegsEpi <= kThreads * kLaunchRegs, "register split above the launch allocation");
constexpr int SO = 4;  // operand stages
constexpr int SP = 4;  // packed stages
constexpr int SS = 2;  // scale slots
constexpr int A_PK = kBM * 64;                // packed A rows (64 bytes each), then B rows
constexpr int PSTAGE = (kBM + kBN) * 64;      // 16 KB
constexpr int A_OP = kBM * 128;               // byte operands, 128-byte rows, 128-byte swizzle
constexpr int OSTAGE = (kBM + kBN) * 128;     // 32 KB
constexpr int SX_BYTES = kSG * kBM * 4;       // s_x [kSG][128]
constexpr int SSLOT = kSG * (kBM + kBN) * 4;  // then sigma [kSG][128]
constexpr int ONES_BYTES = 512;               // 128 floats of 1.0: the branch group's scales
constexpr int NBAR = 2 * (SO + SP + SS + 4) + 1;
constexpr int SMEM = 1024 + SO * OSTAGE + SP * PSTAGE + SS * SSLOT + ONES_BYTES + NBAR * 8 + 16;
static_assert(SMEM <= 232448, "kernel (b) shared memory above the 227 KB per-CTA limit");

typedef unsigned long long f2;  // two packed float32 (for the f32x2 instructions)

__device__ __forceinline__ float lo_f(f2 v) { return __uint_as_float(static_cast<uint32_t>(v)); }
__device__ __forceinline__ float hi_f(f2 v) { return __uint_as_float(static_cast<uint32_t>(v >> 32)); }
__device__ __forceinline__ f2 fma2(f2 a, f2 b, f2 c) {
  f2 d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ f2 mul2(f2 a, f2 b) {
  f2 d;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ f2 add2(f2 a, f2 b) {
  f2 d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ f2 pk2u(uint32_t a, uint32_t b) {
  f2 d;
  asm("mov.b64 %0, {%1, %2};" : "=l"(d) : "r"(a), "r"(b));
  return d;
}
__device__ __forceinline__ f2 pk4(float a, float b) {
  f2 d;
  asm("mov.b64 %0, {%1, %2};" : "=l"(d) : "f"(a), "f"(b));
  return d;
}

// SM4 word -> the E4M3 bytes of its eight codes (k order).
__device__ __forceinline__ uint2 sm4_expand(uint32_t w) {
  return make_uint2(w & 0x87878787u, __funnelshift_r(w, w, 4) & 0x87878787u);
}

// Everything one epilogue warp needs to process a group (see the epilogue in gemm_kernel).
struct EpiCtx {
  const uint8_t* sring;   // scale slots
  const float* ones;      // 128 floats of 1.0 (the branch group's scales)
  uint64_t* sfull;
  uint64_t* sempty;
  uint64_t* tfull;
  uint64_t* tempty;
  WaitCtl wc;
  uint32_t tq;            // TMEM address of this warp's lane quadrant and column half
  int quad, h, rq, cq;
  int ngk, ngt, total;    // K groups per tile, groups per tile, groups of this CTA
};

// One group of the epilogue: g is the CTA's running group index (TMEM unit g % 4), gi its index in
// the tile, sl the running index of the scale slot it reads.  Its TMEM loads sit in v[CUR] (issued
// while the previous group was computed); the loads of group g + 1 go to v[CUR ^ 1] block by block.
template <int CUR>
__device__ __forceinline__ void epi_group(const EpiCtx& c, f2 (&acc)[32], uint32_t (&v)[2][4][16], int& g, int& gi,
                                          int& sl, bool& ok) {
  const bool more = g + 1 < c.total;
  const bool kgroup = gi < c.ngk;
  const int gi_n = gi + 1 == c.ngt ? 0 : gi + 1;
  const bool slot_n = gi_n < c.ngk && (gi_n & (kSG - 1)) == 0;  // group g + 1 starts a scale slot
  const int gl = gi & (kSG - 1);
  // v[CUR][2b + rh][4j + 2rr + {0, 1}] = columns (32b + 8j + 2cq, +1) of row rq + 16 rh + 8 rr
  tmem_ld_wait_dep4(v[CUR]);
  tc_fence_before();
  // Every load of the unit has landed: release it before waiting for the next group (whose stage
  // the MMA issuer may only start once this unit is free).
  warp_arrive(&c.tempty[g & 3]);
  // The next group's phases, tested now and used after the first block: the test's latency
  // overlaps the arithmetic.
  const bool ready_n = !more || ((!slot_n || mbar_test_wait(&c.sfull[(sl + 1) & (SS - 1)], ((sl + 1) / SS) & 1)) &&
                                 mbar_test_wait(&c.tfull[(g + 1) & 3], ((g + 1) >> 2) & 1));
  const uint8_t* slot = c.sring + (sl & (SS - 1)) * SSLOT;
  const float* sxb = kgroup ? reinterpret_cast<const float*>(slot) + gl * kBM : c.ones;
  const float* sgb = kgroup ? reinterpret_cast<const float*>(slot + SX_BYTES) + gl * kBN : c.ones;
  float sx[4];
#pragma unroll
  for (int k = 0; k < 4; ++k) sx[k] = sxb[c.quad * 32 + c.rq + 8 * k];
  const uint32_t tn = c.tq + static_cast<uint32_t>(((g + 1) & 3) * kBN);
#pragma unroll
  for (int b = 0; b < 2; ++b) {
    const float4* sgp = reinterpret_cast<const float4*>(sgb + 64 * c.h + 32 * b + c.cq * 8);
    const float4 s0 = sgp[0], s1 = sgp[1];
    const f2 sg[4] = {pk4(s0.x, s0.y), pk4(s0.z, s0.w), pk4(s1.x, s1.y), pk4(s1.z, s1.w)};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const f2 sx2 = dup2(sx[k]);
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const uint32_t* dv = &v[CUR][2 * b + (k >> 1)][4 * j + 2 * (k & 1)];
        const f2 t = mul2(pk2u(dv[0], dv[1]), sx2);
        acc[16 * b + 4 * k + j] = fma2(t, sg[j], acc[16 * b + 4 * k + j]);
      }
    }
    if (b == 0) {
      if (!ready_n && ok) {
        if (slot_n) ok = mbar_wait_inline(&c.sfull[(sl + 1) & (SS - 1)], ((sl + 1) / SS) & 1, c.wc);
        if (ok) ok = mbar_wait_inline(&c.tfull[(g + 1) & 3], ((g + 1) >> 2) & 1, c.wc);
      }
      tc_fence_after();
    }
    // Issued on every path (after the CTA's last group it reads a unit nobody uses any more), so
    // that each wait's registers come from the loads just before it.
    tmem_ld16x256_x4(tn + 32 * b, v[CUR ^ 1][2 * b]);
    tmem_ld16x256_x4(tn + (16u << 16) + 32 * b, v[CUR ^ 1][2 * b + 1]);
  }
  if (kgroup && (gl == kSG - 1 || gi == c.ngk - 1)) {
    fence_proxy_async_smem();  // reads of the TMA-written scales before the slot is refilled
    warp_arrive(&c.sempty[sl & (SS - 1)]);
  }
  if (slot_n) ++sl;
  ++g;
  gi = gi_n;
}

template <int G>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap qa_map, const __grid_constant__ CUtensorMap qw_map,
                const __grid_constant__ CUtensorMap sx_map, const __grid_constant__ CUtensorMap sw_map,
                const __grid_constant__ CUtensorMap ph_map, const __grid_constant__ CUtensorMap bh_map,
                const GemmArgs a) {
  constexpr int GPS = kKS / G;  // groups per K stage
  static_assert(kSG % GPS == 0, "a scale slot covers whole stages");
  extern __shared__ uint8_t smem_raw[];
  pdl_launch_dependents();
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* oring = smem;                 // SO x (A bytes | B bytes)
  uint8_t* pring = oring + SO * OSTAGE;  // SP x (A packed | B packed)
  uint8_t* sring = pring + SP * PSTAGE;  // SS x (s_x | sigma)
  float* ones = reinterpret_cast<float*>(sring + SS * SSLOT);
  uint64_t* bars = reinterpret_cast<uint64_t*>(sring + SS * SSLOT + ONES_BYTES);
  uint64_t* pfull = bars;
  uint64_t* pempty = pfull + SP;
  uint64_t* ofull = pempty + SP;
  uint64_t* oempty = ofull + SO;
  uint64_t* sfull = oempty + SO;
  uint64_t* sempty = sfull + SS;
  uint64_t* tfull = sempty + SS;
  uint64_t* tempty = tfull + 4;
  uint64_t* drain = tempty + 4;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + NBAR);
  int* abort_flag = reinterpret_cast<int*>(tmem_slot + 1);

  const uint32_t wid = warp_id(), lane = lane_id();
  const int ngk = a.K / G;     // K groups per tile
  const int nks = (a.K + kKS - 1) / kKS;  // K stages per tile (the last is half past K when K % 128 == 64:
                                          // TMA zero-fills it and its missing groups are skipped)
  const int nbs = a.nbs;       // branch stages per tile
  const int nst = nks + nbs;
  const int ngt = ngk + (nbs > 0 ? 1 : 0);  // groups per tile, the branch included
  const int nsl = (ngk + kSG - 1) / kSG;    // scale slots per tile
  const int ntiles = a.m_tiles * a.n_tiles;
  const int my_tiles = ntiles > static_cast<int>(blockIdx.x)
                           ? (ntiles - static_cast<int>(blockIdx.x) + static_cast<int>(gridDim.x) - 1) /
                                 static_cast<int>(gridDim.x)
                           : 0;
  auto tile_mn = [&](int i, int& m0, int& n0) {
    const int t = static_cast<int>(blockIdx.x) + i * static_cast<int>(gridDim.x);
    m0 = (t / a.n_tiles) * kBM;
    n0 = (t % a.n_tiles) * kBN;
  };

  if (threadIdx.x == 0) {
    for (int i = 0; i < SP; ++i) {
      mbar_init(&pfull[i], 1);
      mbar_init(&pempty[i], kNX);
    }
    for (int i = 0; i < SO; ++i) {
      mbar_init(&ofull[i], kNX);
      mbar_init(&oempty[i], 1);
    }
    for (int i = 0; i < SS; ++i) {
      mbar_init(&sfull[i], 1);
      mbar_init(&sempty[i], 8);
    }
    for (int i = 0; i < 4; ++i) {
      mbar_init(&tfull[i], 1);
      mbar_init(&tempty[i], 8);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (threadIdx.x < 128) ones[threadIdx.x] = 1.0f;
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
      // The whole warp walks the loop (warp-uniform state); one elected lane issues each copy.
      bool ok = true;
      int s = 0, ss = 0;
      for (int ti = 0; ti < my_tiles && ok; ++ti) {
        int m0, n0;
        tile_mn(ti, m0, n0);
        for (int st = 0; st < nst && ok; ++st, ++s) {
          if (st < nks && (st * GPS) % kSG == 0) {
            // s_x and sigma of the next kSG groups (zero-filled past K)
            const int sb = ss % SS;
            if (ss >= SS) ok = mbar_wait_inline(&sempty[sb], ((ss / SS) & 1) ^ 1, wc);
            if (!ok) break;
            uint8_t* q = sring + sb * SSLOT;
            if (elect_one()) {
              mbar_arrive_expect_tx(&sfull[sb], SSLOT);
              tma_load_2d(q, &sx_map, &sfull[sb], m0, st * GPS);
              tma_load_2d(q + SX_BYTES, &sw_map, &sfull[sb], n0, st * GPS);
            }
            __syncwarp();
            ++ss;
          }
          const int ps = s % SP;
          if (s >= SP) ok = mbar_wait_inline(&pempty[ps], ((s / SP) & 1) ^ 1, wc);
          if (!ok) break;
          uint8_t* p = pring + ps * PSTAGE;
          if (elect_one()) {
            mbar_arrive_expect_tx(&pfull[ps], PSTAGE);
            if (st < nks) {
              tma_load_2d(p, &qa_map, &pfull[ps], st * (kKS / 2), m0);
              tma_load_2d(p + A_PK, &qw_map, &pfull[ps], st * (kKS / 2), n0);
            } else {
              const int bs = st - nks;
              tma_load_2d(p, &ph_map, &pfull[ps], bs * 32, m0);
              tma_load_2d(p + A_PK, &bh_map, &pfull[ps], bs * 32, n0);
            }
          }
          __syncwarp();
        }
      }
      // Let every issued load land before the CTA can exit (these phases complete in the normal
      // course; after an abort the waits end at the deadline).
      int never = 0;
      const WaitCtl dc{&never, a.err, globaltimer_ns() + a.timeout_ns};
      for (int j = (s > SP ? s - SP : 0); j < s; ++j) mbar_wait_inline(&pfull[j % SP], (j / SP) & 1, dc);
      for (int j = (ss > SS ? ss - SS : 0); j < ss; ++j) mbar_wait_inline(&sfull[j % SS], (j / SS) & 1, dc);
    } else if (wid == 1) {
      // ----------------------------------------------------------- MMA issuer
      // The whole warp walks the loop and forms the descriptors; one elected lane (the same one
      // throughout, as the commits track its MMAs) issues a stage's MMAs and commits together.
      bool ok = true;
      constexpr uint32_t idesc = idesc_e4m3(kBM, kBN);
      constexpr uint32_t idesc_br = idesc_f16(kBM, kBN);
      int s = 0, gr = 0;  // running stage and group counters
      for (int ti = 0; ti < my_tiles && ok; ++ti) {
        for (int st = 0; st < nst && ok; ++st, ++s) {
          const int os = s % SO;
          const bool kst = st < nks;
          const int gn = kst ? min(GPS, ngk - st * GPS) : 1;  // groups this stage writes
          ok = mbar_wait_inline(&ofull[os], (s / SO) & 1, wc);
          // the last TMEM unit this stage writes: its release (four groups back) implies the
          // earlier ones (the epilogue releases units in order)
          const int glast = gr + gn - 1;
          if (ok && glast >= 4 && (kst || st == nks))
            ok = mbar_wait_inline(&tempty[glast & 3], ((glast >> 2) & 1) ^ 1, wc);
          if (!ok) break;
          tc_fence_after();
          const uint32_t aa = smem_u32(oring + os * OSTAGE);
          const uint64_t adesc = smem_desc(aa, 16, 1024, kSw128), bdesc = smem_desc(aa + A_OP, 16, 1024, kSw128);
          if (elect_one()) {
            if (kst) {
#pragma unroll
              for (int gi = 0; gi < GPS; ++gi) {
                if (gi >= gn) break;
                const uint32_t d = tmem + static_cast<uint32_t>(((gr + gi) & 3) * kBN);
#pragma unroll
                for (int kk = 0; kk < G / 32; ++kk) {
                  const uint64_t off = static_cast<uint64_t>((gi * G + kk * 32) >> 4);  // 16-byte units
                  mma_f8f6f4(d, adesc + off, bdesc + off, idesc, kk != 0);
                }
                mma_commit(&tfull[(gr + gi) & 3]);
              }
            } else {
              const int bs = st - nks;
              const uint32_t d = tmem + static_cast<uint32_t>((gr & 3) * kBN);
              mma_f16(d, adesc, bdesc, idesc_br, bs != 0);
              mma_f16(d, adesc + 2, bdesc + 2, idesc_br, 1);
              if (bs == nbs - 1) mma_commit(&tfull[gr & 3]);
            }
            mma_commit(&oempty[os]);
          }
          __syncwarp();
          if (kst)
            gr += gn;
          else if (st == nst - 1)
            ++gr;
        }
      }
      if (elect_one()) mma_commit(drain);
      __syncwarp();
      int never = 0;
      const WaitCtl dc{&never, a.err, globaltimer_ns() + a.timeout_ns};
      mbar_wait_inline(drain, 0, dc);
    } else {
      // ----------------------------------------------------------- expanders
      // Thread e (0..63) takes the 16-byte piece q = e % 4 of packed rows r0 + 16 i (r0 = e / 4,
      // i = 0..15; rows 0..127 are A, 128..255 B): a K stage expands it to the operand chunks
      // 2q, 2q + 1 of the row, a branch stage copies it to chunk q.  Operand rows are 128 bytes with
      // the 128-byte swizzle (chunk c of row r at c ^ (r % 8)); r % 8 = r0 % 8 for all of this
      // thread's rows, so every offset below is a constant.
      const int e = static_cast<int>(threadIdx.x) - 64;
      const int r0 = e >> 2, q = e & 3, sw = r0 & 7;
      const int src0 = r0 * 64 + q * 16;
      const int dlo = r0 * 128 + (((2 * q) ^ sw) << 4), dhi = r0 * 128 + (((2 * q + 1) ^ sw) << 4);
      const int dcp = r0 * 128 + ((q ^ sw) << 4);
      bool ok = true;
      int s = 0;
      for (int ti = 0; ti < my_tiles && ok; ++ti) {
        for (int st = 0; st < nst && ok; ++st, ++s) {
          const int ps = s % SP, os = s % SO;
          ok = mbar_wait_inline(&pfull[ps], (s / SP) & 1, wc);
          if (ok && s >= SO) ok = mbar_wait_inline(&oempty[os], ((s / SO) & 1) ^ 1, wc);
          if (!ok) break;
          const uint8_t* src = pring + ps * PSTAGE + src0;
          uint8_t* dst = oring + os * OSTAGE;
          // Four loads, then four expansions and their stores: the stores may alias the loads as far
          // as the compiler knows, so written in this order the loads are in flight together.
          if (st < nks) {
#pragma unroll 1
            for (int i0 = 0; i0 < 16; i0 += 4) {
              uint4 v[4];
#pragma unroll
              for (int i = 0; i < 4; ++i) v[i] = *reinterpret_cast<const uint4*>(src + (i0 + i) * 1024);
#pragma unroll
              for (int i = 0; i < 4; ++i) {
                const uint2 x = sm4_expand(v[i].x), y = sm4_expand(v[i].y), z = sm4_expand(v[i].z),
                            w = sm4_expand(v[i].w);
                *reinterpret_cast<uint4*>(dst + dlo + (i0 + i) * 2048) = make_uint4(x.x, x.y, y.x, y.y);
                *reinterpret_cast<uint4*>(dst + dhi + (i0 + i) * 2048) = make_uint4(z.x, z.y, w.x, w.y);
              }
            }
          } else {
#pragma unroll 1
            for (int i0 = 0; i0 < 16; i0 += 4) {
              uint4 v[4];
#pragma unroll
              for (int i = 0; i < 4; ++i) v[i] = *reinterpret_cast<const uint4*>(src + (i0 + i) * 1024);
#pragma unroll
              for (int i = 0; i < 4; ++i) *reinterpret_cast<uint4*>(dst + dcp + (i0 + i) * 2048) = v[i];
            }
          }
          // Orders the generic writes of the operand stage before the MMA reads them, and the
          // generic reads of the packed stage before TMA refills it.
          fence_proxy_async_smem();
          warp_arrive(&ofull[os]);
          warp_arrive(&pempty[ps]);
        }
      }
    }
  } else {
    setmaxnreg_inc<kRegsEpi>();
    // ------------------------------------------------------------- epilogue
    // Warp 4 + 4h + q reads TMEM lanes 32q.. (its quadrant of rows), columns 64h .. 64h + 63 of
    // each unit.  With the 16x256b load shape, thread t holds rows rq + 8k (k = 0..3, rq = t / 4)
    // and, in each 32-column block b, columns 8j + 2cq + {0, 1} (j = 0..3, cq = t % 4):
    // acc[16b + 4k + j] is that pair.  Per group and output: t = D s_x, acc += t sigma.  Sigma is
    // stored permuted within each 32-column block, so the thread's eight scales of a block are
    // contiguous (two 16-byte loads).
    const int quad = static_cast<int>(wid & 3), h = (static_cast<int>(wid) - 4) >> 2;
    const int rq = static_cast<int>(lane) >> 2, cq = static_cast<int>(lane) & 3;
    EpiCtx c;
    c.sring = sring;
    c.ones = ones;
    c.sfull = sfull;
    c.sempty = sempty;
    c.tfull = tfull;
    c.tempty = tempty;
    c.wc = wc;
    c.tq = tmem + (static_cast<uint32_t>(quad * 32) << 16) + static_cast<uint32_t>(64 * h);
    c.quad = quad;
    c.h = h;
    c.rq = rq;
    c.cq = cq;
    c.ngk = ngk;
    c.ngt = ngt;
    c.total = my_tiles * ngt;  // groups this CTA's epilogue walks (branch included)
    bool ok = true;
    uint32_t v[2][4][16];  // TMEM loads of two groups: [buffer][block b * 2 + row half][16]
    f2 acc[32];
    if (c.total > 0) {
      if (ok) ok = mbar_wait_inline(&sfull[0], 0, wc);
      if (ok) ok = mbar_wait_inline(&tfull[0], 0, wc);
      tc_fence_after();
#pragma unroll
      for (int b = 0; b < 2; ++b) {
        tmem_ld16x256_x4(c.tq + 32 * b, v[0][2 * b]);
        tmem_ld16x256_x4(c.tq + (16u << 16) + 32 * b, v[0][2 * b + 1]);
      }
    }
    // Group g of the CTA lands in buffer g % 2.  A tile's groups run in pairs from a buffer parity
    // fixed at compile time (one copy of the loop per parity, chosen by the tile's first group), so
    // the accumulator is zeroed and stored outside the per-group code.  The branch group takes the
    // same arithmetic with unit scales (D * 1 * 1 + acc = D + acc exactly).
    int g = 0, sl = 0;
    for (int ti = 0; ti < my_tiles; ++ti) {
#pragma unroll
      for (int i = 0; i < 32; ++i) acc[i] = 0ull;
      // (gi is advanced by epi_group and wraps to 0 after the tile's last group; the loops below
      // count the tile's groups with their own index)
      int gi = 0;
      if ((g & 1) == 0) {
        for (int j = 0; j + 2 <= ngt; j += 2) {
          epi_group<0>(c, acc, v, g, gi, sl, ok);
          epi_group<1>(c, acc, v, g, gi, sl, ok);
        }
        if (ngt & 1) epi_group<0>(c, acc, v, g, gi, sl, ok);
      } else {
        for (int j = 0; j + 2 <= ngt; j += 2) {
          epi_group<1>(c, acc, v, g, gi, sl, ok);
          epi_group<0>(c, acc, v, g, gi, sl, ok);
        }
        if (ngt & 1) epi_group<1>(c, acc, v, g, gi, sl, ok);
      }
      // the tile's output: Y (plus the bias)
      int m0, n0;
      tile_mn(ti, m0, n0);
      if (ok) {
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const int m = m0 + quad * 32 + rq + 8 * k;
          if (m >= a.M) continue;
#pragma unroll
          for (int b = 0; b < 2; ++b)
#pragma unroll
            for (int j = 0; j < 4; ++j) {
              const int n = n0 + 64 * h + 32 * b + 8 * j + 2 * cq;  // even; N is a multiple of 8
              if (n >= a.N) continue;
              const size_t off = static_cast<size_t>(m) * a.N + n;
              const f2 y = acc[16 * b + 4 * k + j];
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
    tmem_ld_wait();  // the loads issued after the last group land before TMEM is released
  }

  __syncthreads();
  if (wid == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

template <int G>
cudaError_t launch_g(Handle& h, const ActMaps& am, int M, void* Y, bool y_f32, cudaStream_t s) {
  GemmArgs a;
  a.M = M;
  a.N = h.N;
  a.K = h.K;
  a.nbs = (h.r_pad + 31) / 32;
  a.m_tiles = (M + kBM - 1) / kBM;
  a.n_tiles = (h.N + kBN - 1) / kBN;
  a.Y = Y;
  a.y_f32 = y_f32 ? 1 : 0;
  a.bias = h.bias;
  a.err = h.err;
  a.timeout_ns = deadline_budget_ns(h);
  static bool attr_done = false;
  if (!attr_done) {
    cudaError_t e = cudaFuncSetAttribute(gemm_kernel<G>, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM);
    if (e != cudaSuccess) return e;
    attr_done = true;
  }
  const int ntiles = a.m_tiles * a.n_tiles;
  const int grid = ntiles < h.num_sms ? ntiles : h.num_sms;
  // Without a branch the p_hat / B_hat maps are never used; any valid map fills the slots.
  const CUtensorMap& ph = (h.r_pad > 0) ? am.ph32_map : am.qa_map;
  const CUtensorMap& bh = (h.r_pad > 0) ? h.bh32_map : am.qa_map;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = SMEM;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, gemm_kernel<G>, am.qa_map, h.qw_map, am.sx_map, h.sw32_map, ph, bh, a);
}

}  // namespace

cudaError_t launch_gemm(Handle& h, const ActMaps& am, const void* ws, int M, void* Y, bool y_f32, cudaStream_t s) {
  (void)ws;
  return h.G == 32 ? launch_g<32>(h, am, M, Y, y_f32, s) : launch_g<64>(h, am, M, Y, y_f32, s);
}

}  // namespace qwam
