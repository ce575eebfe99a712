// gemm.cu -- kernel (b): the 4-bit deflated path of Eq. (asp) with the 16-bit branch fused into
// the same kernel (Sec. 4.2; App. B.1 describes the paper's GEMM as one that keeps the weights
// packed at 4 bits and adds the protected branch in its epilogue).
//
//   Y[m, n] = sum_g s_x[m, g] s_w[g, n] P_g[m, n]  +  sum_j p_hat[m, j] B_hat[n, j]
//   P_g[m, n] = sum_{k in group g} q_x[m, k] q_w[n, k]
//
// Both scales are bfloat16 (8 significant bits) and the codes lie in [-7, 7] (3 bits), so every
// dequantized operand s q has at most 11 significant bits: it is exact in float16.  The layer is
// then one contraction over K + r_pad columns,
//
//   Y = [s_x q_x | p_hat] [s_w q_w | B_hat]^T,
//
// which this kernel runs on tcgen05.mma.kind::f16 (float16 operands, float32 accumulation in TMEM)
// with the operands dequantized from the packed 4-bit codes on the fly.  No per-group rescale is
// left for the epilogue: the tensor cores apply both scales, and the branch is r_pad more K
// columns of the same accumulator.
//
// Range.  float16 holds s q exactly while it stays in [2^-14, 2^16) (and down to 2^-24 when its
// low bits allow).  Row m of the activation operand is therefore scaled by 2^e_m and column n of
// the weight operand by 2^e_n, powers of two chosen so that the largest dequantized value of the
// row (7 max_g s_x, or max |p_hat|) and of the column (7 max_g s_w, or max |B_hat|) lies in
// [2^10, 2^11) (so that 16 s and the dequantization's other constants stay finite); the
// epilogue multiplies by 2^-e_n and then 2^-e_m, which is exact unless the result is a float32
// subnormal.  Only values below 2^-24 of their row's or column's largest can lose bits, which is
// at the float32 accumulator's own resolution.  The weight side is done
// once, at pack time (the handle's swh, Bhs, fcol); the row factors are formed here from s_x and
// p_hat by the epilogue warps.
//
// Tiles are 128 tokens x 256 outputs (one tcgen05 MMA of M = 128, N = 256, K = 16 per 16 columns),
// K stages of 64.  The activation operand lives in TMEM (tcgen05.mma with A from tensor memory:
// lane m holds row m, column c the float16 pair k = 2c, 2c + 1), written by tcgen05.st from the
// expanders' registers; the weight operand lives in shared memory in the 128-byte swizzled K-major
// layout.  (An A operand in TMEM takes the shared-memory bandwidth of the MMA down by a third.)
// Persistent CTAs, one per SM, walk the tiles with a static stride.  896 threads:
//   warp 0        TMA producer: per K stage the packed codes of both operands and their scales
//   warp 1        MMA issuer and TMEM owner
//   warp 2        idle
//   warp 3        with PREB (below): TMA producer of the float16 weight stages; else idle
//   warps 4..19   expanders, two groups of eight that take alternate stages (group x the stages
//                 whose running index is x mod 2), so that each warp has two stage times for its
//                 work.  Warp e of a group takes the activation codes k = 32h .. 32h + 31
//                 (h = e / 4) of the 32 token rows in TMEM lane quadrant q = e % 4 (16 columns
//                 stored with tcgen05.st) and weight rows 32e .. 32e + 31 of the stage's 256
//                 (float16 into the shared-memory operand)
//   warps 20..27  epilogue: warp 20 + 4h + q reads lanes 32q.., columns 128h..128h+127; between
//                 tiles the same warps form the row scales 2^e_m, 2^-e_m of the tile after next
//                 (two threads per row) and stage their columns' 2^-e_n and bias in shared memory
// Branch stages (after the K stages, r_pad / 64 rounded up): the expanders load p_hat by TMA (one
// buffer per group) and scale it by 2^e_m into TMEM, and B_hat 2^e_n comes by TMA straight into the
// operand stage.  Every wait is bounded.
// Layers with several 128-row tiles (kPreExpandMinTiles) would convert every weight stage once per
// row tile; for them the float16 weights [s_w 2^e_n c | B_hat 2^e_n] are written once per call into
// the workspace (the PREB instantiation): by kernel (a) inside qwam_asp_linear when r > 0, else by
// `dequant_weights_kernel` just before this kernel.  The producer loads each weight stage by TMA
// straight into the operand ring, and the expanders convert the activations only.
// Rings:
//   P  packed stage: A and B codes, s_x and s_w 2^e_n of its groups   TMA -> expanders   SP slots
//   O  operand stage: A (TMEM, 32 columns) and B (shared memory)  expanders -> MMA   SO slots
//   R  row-scale slot                          epilogue warps -> expanders, epilogue   2 slots
//   the accumulator (TMEM columns 0..255)     MMA -> epilogue             1
#include "dequant.cuh"
#include "internal.h"
#include "ptx.cuh"

namespace qwam {
namespace {

struct GemmArgs {
  int M, N, K, r_pad, M_pad;
  int nbs;  // branch stages per tile
  int m_tiles, n_tiles;
  const __nv_bfloat16* sx;  // workspace s_x [K/G, M_pad] (row-scale warp)
  const __half* phat;       // workspace p_hat [M, r_pad] (row-scale warp; null when r_pad == 0)
  const float* fcol;        // handle: 2^-e_n [N_pad]
  void* Y;
  int y_f32;
  const float* bias;        // optional [N], added to the float32 result before it is stored
  int splits;               // > 1: split-K over a cluster of `splits` CTAs per tile (below)
  float* part;              // splits > 1: float32 [splits, M, N] partial results (workspace)
  int* err;
  uint64_t timeout_ns;
};

constexpr int BM = kBM;        // 128 token rows
constexpr int BN = kGemm16BN;  // 256 output columns
constexpr int KS = 64;         // K per stage
constexpr int kThreads = 896;
constexpr int SP = 4, SO = 4;
constexpr int PA = BM * KS / 2;          // packed A bytes per stage (4 KB)
constexpr int PB = BN * KS / 2;          // packed B bytes per stage (8 KB)
constexpr int PSX = 2 * BM * 2;          // s_x [GPS][128] bf16 (room for two groups)
constexpr int PSTAGE = PA + PSX + 2 * BN * 2;  // packed A, s_x, then s_w 2^e_n [GPS][256] f16
constexpr int BSTAGE = BN * KS * 2;      // float16 weight operand, 128-byte rows (32 KB)
constexpr int PHB = BM * KS * 2;         // p_hat stage [128][64] f16, 128-byte swizzle (one per group)
constexpr int RSB = BM * 8;              // {2^e_m, 2^-e_m} per row
constexpr int EFB = 2 * 128 * 4;         // per epilogue warp: 2^-e_n and bias of its 128 columns
constexpr int NBAR = 2 * SP + 2 * SO + 2 + 2 * 2 + 2 * 2 + 1;
constexpr int OFF_B = 0;
constexpr int OFF_PH = OFF_B + SO * BSTAGE;
constexpr int OFF_PB = OFF_PH + 2 * PHB;  // packed B of each stage [SP][PB]; PREB: the output staging
constexpr int OFF_P = OFF_PB + SP * PB;
constexpr int OFF_R = OFF_P + SP * PSTAGE;
constexpr int OFF_E = OFF_R + 2 * RSB;
constexpr int OFF_BAR = OFF_E + 8 * EFB;
constexpr int SMEM = 1024 + OFF_BAR + NBAR * 8 + 16;
static_assert(SMEM <= 232448, "kernel (b) shared memory above the 227 KB per-CTA limit");
// PREB: each epilogue warp stages 32 rows x 128 bytes of output (128-byte swizzle, 1024-byte
// aligned) in the packed-B slots, which that mode does not use, and stores them by TMA.
constexpr int YSTG = 4096;
static_assert(8 * YSTG <= SP * PB && OFF_PB % 1024 == 0 && PB % 1024 == 0, "output staging");
static_assert(SMEM <= 232448, "kernel (b) shared memory above the 227 KB per-CTA limit");
constexpr uint32_t TMEM_COLS = 512;  // accumulator 0..255, A ring 256 + 32 i
constexpr uint32_t TMEM_A = 256;

__device__ __forceinline__ void mma_f16_tmem_a(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc, uint32_t idesc,
                                               uint32_t accumulate) {
  asm volatile(
      "{\n.reg .pred p;\nsetp.ne.b32 p, %4, 0;\n"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

__device__ __forceinline__ void tmem_st_wait() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

__device__ __forceinline__ uint32_t f32x2_to_bf16x2(float lo, float hi) {
  uint32_t d;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(hi), "f"(lo));
  return d;
}
// Global stores and read-only loads named as such: a generic store could alias the shared-memory
// reads around it as far as the compiler knows, which would serialize the epilogue.
__device__ __forceinline__ void st_global_v4(void* p, uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
  asm volatile("st.global.v4.b32 [%0], {%1, %2, %3, %4};" ::"l"(p), "r"(a), "r"(b), "r"(c), "r"(d));
}
__device__ __forceinline__ void st_global_v8(void* p, const uint32_t* v) {
  asm volatile("st.global.v8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"l"(p), "r"(v[0]), "r"(v[1]), "r"(v[2]),
               "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]));
}
__device__ __forceinline__ uint32_t ld_nc_u16(const void* p) {
  unsigned short v;
  asm volatile("ld.global.nc.u16 %0, [%1];" : "=h"(v) : "l"(p));
  return v;
}
__device__ __forceinline__ uint4 ld_nc_v4(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.v4.b32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
  return v;
}
__device__ __forceinline__ float f16_lo(uint32_t u) { return __half2float(__ushort_as_half(static_cast<unsigned short>(u))); }
__device__ __forceinline__ float f16_hi(uint32_t u) { return __half2float(__ushort_as_half(static_cast<unsigned short>(u >> 16))); }


// s (bfloat16) times 2^e, rounded to float16 (exact while in range), as dequantization constants.
__device__ __forceinline__ DqScale scale_consts(__nv_bfloat16 s, float mul) {
  return dq_scale(__half2float(__float2half_rn(__bfloat162float(s) * mul)));
}

// 32 TMEM lanes x 16 consecutive 32-bit columns from registers.
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
      "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]),
      "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
      : "memory");
}

// Transaction bytes expected on a barrier, without an arrival.
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.expect_tx.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes) : "memory");
}

// The weights of one call in float16 (expand_w16), for layers with several row tiles.  Each thread
// takes eight pieces a grid stride apart per round.
__global__ void __launch_bounds__(256) dequant_weights_kernel(const W16Args w) {
  pdl_launch_dependents();
  pdl_wait();  // the workspace may still be read by the stream's previous GEMM until then
  expand_w16<8>(w, static_cast<int>(blockIdx.x * blockDim.x + threadIdx.x), static_cast<int>(gridDim.x * blockDim.x));
}

template <int G, bool PREB>
__global__ void __launch_bounds__(kThreads, 1)
    gemm16_kernel(const __grid_constant__ CUtensorMap qa_map, const __grid_constant__ CUtensorMap qw_map,
                  const __grid_constant__ CUtensorMap sx_map, const __grid_constant__ CUtensorMap sw_map,
                  const __grid_constant__ CUtensorMap ph_map, const __grid_constant__ CUtensorMap bh_map,
                  const __grid_constant__ CUtensorMap y_map, const GemmArgs a) {
  constexpr int GPS = KS / G;   // groups per K stage (1 or 2)
  extern __shared__ uint8_t smem_raw[];
  pdl_launch_dependents();
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* bring = smem + OFF_B;
  uint8_t* phbuf = smem + OFF_PH;
  uint8_t* pring = smem + OFF_P;
  uint8_t* pbring = smem + OFF_PB;
  float2* rslot = reinterpret_cast<float2*>(smem + OFF_R);
  float* efb = reinterpret_cast<float*>(smem + OFF_E);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + OFF_BAR);
  uint64_t* pfull = bars;
  uint64_t* pempty = pfull + SP;
  uint64_t* ofull = pempty + SP;
  uint64_t* oempty = ofull + SO;
  uint64_t* accfull = oempty + SO;
  uint64_t* accempty = accfull + 1;
  uint64_t* rfull = accempty + 1;
  uint64_t* rempty = rfull + 2;
  uint64_t* phfull = rempty + 2;   // one per expander group
  uint64_t* phempty = phfull + 2;
  uint64_t* drain = phempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + NBAR);
  int* abort_flag = reinterpret_cast<int*>(tmem_slot + 1);

  const uint32_t wid = warp_id(), lane = lane_id();
  // Split-K (few tiles, many idle SMs): the `splits` CTAs of a cluster share one tile, CTA `rank`
  // taking K stages [kb, kb + nks) and, the last one, the branch stages; each writes its float32
  // partial tile (without the bias) to the workspace, and after one cluster barrier each sums a
  // 1/splits slice of the tile's columns over the partials in rank order and stores the output.
  const bool split = !PREB && a.splits > 1;  // (the float16-weight GEMM never splits)
  const int rank = split ? static_cast<int>(cluster_ctarank()) : 0;
  const int nks_all = a.K / KS;
  const int kb = rank * nks_all / a.splits;
  const int nks = (rank + 1) * nks_all / a.splits - kb;
  const int nbs = rank == a.splits - 1 ? a.nbs : 0;
  const int nst = nks + nbs;
  const int ntiles = a.m_tiles * a.n_tiles;
  const int my_tiles = split ? 1
                       : ntiles > static_cast<int>(blockIdx.x)
                           ? (ntiles - static_cast<int>(blockIdx.x) + static_cast<int>(gridDim.x) - 1) /
                                 static_cast<int>(gridDim.x)
                           : 0;
  auto tile_mn = [&](int i, int& m0, int& n0) {
    const int t = split ? static_cast<int>(blockIdx.x) / a.splits
                        : static_cast<int>(blockIdx.x) + i * static_cast<int>(gridDim.x);
    m0 = (t / a.n_tiles) * BM;
    n0 = (t % a.n_tiles) * BN;
  };
  // where the epilogue writes: the output, or (split-K) this CTA's partial slice, float32, no bias
  void* const yout = split ? static_cast<void*>(a.part + static_cast<size_t>(rank) * a.M * a.N) : a.Y;
  const int yf32 = split ? 1 : a.y_f32;
  const float* const ybias = split ? nullptr : a.bias;

  if (threadIdx.x == 0) {
    for (int i = 0; i < SP; ++i) {
      mbar_init(&pfull[i], 1);
      mbar_init(&pempty[i], 8);
    }
    for (int i = 0; i < SO; ++i) {
      mbar_init(&ofull[i], PREB ? 9 : 8);  // the group's eight expanders (and, with PREB, the producer)
      mbar_init(&oempty[i], 1);
    }
    mbar_init(accfull, 1);
    mbar_init(accempty, 8);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&rfull[i], 8);
      mbar_init(&rempty[i], 24);
      mbar_init(&phfull[i], 1);
      mbar_init(&phempty[i], 8);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (wid == 1) {
    tmem_alloc(tmem_slot, TMEM_COLS);
    tmem_relinquish();
  }
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const WaitCtl wc{abort_flag, a.err, globaltimer_ns() + a.timeout_ns};
  // Every global access of this kernel that reads what the previous kernel of the stream wrote
  // comes after this wait (the producer's first weight stages, which it did not write, go before).
  if (wid != 0 || PREB) pdl_wait();

  if (wid == 0) {
    // ------------------------------------------------------------- TMA producer (activations)
    // Per K stage: the packed codes of both operands and their scales (with PREB: the activation
    // codes and s_x; warp 3 brings the float16 weights).
    bool ok = true;
    int s = 0;
    int pre = 0;  // stages of the first tile whose weight part was requested before the wait
    if (!PREB) {
      if (my_tiles > 0) {
        int m0, n0;
        tile_mn(0, m0, n0);
        pre = nks < SP ? nks : SP;
        if (elect_one())
          for (int st = 0; st < pre; ++st) {
            uint8_t* p = pring + st * PSTAGE;
            mbar_arrive_expect_tx(&pfull[st], PA + PB + GPS * (BM + BN) * 2);
            tma_load_2d(pbring + st * PB, &qw_map, &pfull[st], (kb + st) * (KS / 2), n0);
            tma_load_2d(p + PA + PSX, &sw_map, &pfull[st], n0, (kb + st) * GPS);
          }
        __syncwarp();
      }
      pdl_wait();
    }
    for (int ti = 0; ti < my_tiles && ok; ++ti) {
      int m0, n0;
      tile_mn(ti, m0, n0);
      for (int st = 0; st < nks && ok; ++st, ++s) {
        const int ps = s % SP;
        if (s >= SP) ok = mbar_wait_inline(&pempty[ps], ((s / SP) & 1) ^ 1, wc);
        if (!ok) break;
        uint8_t* p = pring + ps * PSTAGE;
        if (elect_one()) {
          if (PREB) {
            mbar_arrive_expect_tx(&pfull[ps], PA + GPS * BM * 2);
            tma_load_2d(p, &qa_map, &pfull[ps], (kb + st) * (KS / 2), m0);
            tma_load_2d(p + PA, &sx_map, &pfull[ps], m0, (kb + st) * GPS);
          } else if (s < pre) {  // the weight part is on its way
            tma_load_2d(p, &qa_map, &pfull[ps], (kb + st) * (KS / 2), m0);
            tma_load_2d(p + PA, &sx_map, &pfull[ps], m0, (kb + st) * GPS);
          } else {
            mbar_arrive_expect_tx(&pfull[ps], PA + PB + GPS * (BM + BN) * 2);
            tma_load_2d(p, &qa_map, &pfull[ps], (kb + st) * (KS / 2), m0);
            tma_load_2d(pbring + ps * PB, &qw_map, &pfull[ps], (kb + st) * (KS / 2), n0);
            tma_load_2d(p + PA, &sx_map, &pfull[ps], m0, (kb + st) * GPS);
            tma_load_2d(p + PA + PSX, &sw_map, &pfull[ps], n0, (kb + st) * GPS);
          }
        }
        __syncwarp();
      }
    }
    // every issued load lands before the CTA can exit
    int never = 0;
    const WaitCtl dc{&never, a.err, globaltimer_ns() + a.timeout_ns};
    for (int j = (s > SP ? s - SP : 0); j < s; ++j) mbar_wait_inline(&pfull[j % SP], (j / SP) & 1, dc);
  } else if (wid == 3 && PREB) {
    // ------------------------------------------------------------- TMA producer (weights, PREB)
    // Every stage's float16 weights (W_perp, or B_hat in a branch stage) into the operand ring.
    bool ok = true;
    int so = 0;
    for (int ti = 0; ti < my_tiles && ok; ++ti) {
      int m0, n0;
      tile_mn(ti, m0, n0);
      for (int st = 0; st < nst && ok; ++st, ++so) {
        const int os = so % SO;
        if (so >= SO) ok = mbar_wait_inline(&oempty[os], ((so / SO) & 1) ^ 1, wc);
        if (!ok) break;
        if (elect_one()) {
          mbar_arrive_expect_tx(&ofull[os], BSTAGE);
          tma_load_2d(bring + os * BSTAGE, &bh_map, &ofull[os], st * KS, n0);
        }
        __syncwarp();
      }
    }
    int never = 0;
    const WaitCtl dc{&never, a.err, globaltimer_ns() + a.timeout_ns};
    for (int j = (so > SO ? so - SO : 0); j < so; ++j) mbar_wait_inline(&ofull[j % SO], (j / SO) & 1, dc);
  } else if (wid == 1) {
    // ------------------------------------------------------------- MMA issuer
    constexpr uint32_t idesc = idesc_f16(BM, BN);
    bool ok = true;
    int so = 0;
    for (int ti = 0; ti < my_tiles && ok; ++ti) {
      if (ti > 0) ok = mbar_wait_inline(accempty, (ti - 1) & 1, wc);  // the epilogue has read the last tile
      for (int st = 0; st < nst && ok; ++st, ++so) {
        const int os = so % SO;
        ok = mbar_wait_inline(&ofull[os], (so / SO) & 1, wc);
        if (!ok) break;
        tc_fence_after();
        const uint64_t bdesc = smem_desc(smem_u32(bring + os * BSTAGE), 16, 1024, kSw128);
        const uint32_t at = tmem + TMEM_A + static_cast<uint32_t>(os * 32);
        if (elect_one()) {
#pragma unroll
          for (int kk = 0; kk < KS / 16; ++kk)
            mma_f16_tmem_a(tmem, at + 8 * kk, bdesc + 2 * kk, idesc, (st | kk) != 0 ? 1u : 0u);
          mma_commit(&oempty[os]);
          if (st == nst - 1) mma_commit(accfull);
        }
        __syncwarp();
      }
    }
    if (elect_one()) mma_commit(drain);
    __syncwarp();
    int never = 0;
    const WaitCtl dc{&never, a.err, globaltimer_ns() + a.timeout_ns};
    mbar_wait_inline(drain, 0, dc);
  } else if (wid >= 4 && wid < 20) {
    // ------------------------------------------------------------- expanders
    // Activation part: row r = 32q + lane (TMEM lane), codes k = 32h .. 32h + 31 of the stage
    // (packed words 4h .. 4h+3), to TMEM columns 16h .. 16h + 15 of the stage's slot.
    // Weight part: rows R = 32e + 16i + lane/2 (i = 0, 1), half hh = lane % 2 of the row (words
    // 4hh .. 4hh+3, codes 32hh ..), written as the 16-byte chunks 4hh + jj of row R at their
    // swizzled places (chunk c of row R at c ^ (R % 8); R % 8 = (lane / 2) % 8 for every i).
    const int gx = (static_cast<int>(wid) - 4) >> 3;  // expander group
    const int e = (static_cast<int>(wid) - 4) & 7;
    const int q = e & 3, h = e >> 2;
    const int r = 32 * q + static_cast<int>(lane);
    const int hh = static_cast<int>(lane) & 1;
    const int Rb = 32 * e + (static_cast<int>(lane) >> 1);
    const uint32_t tlane = tmem + (static_cast<uint32_t>(32 * q) << 16) + TMEM_A + static_cast<uint32_t>(16 * h);
    uint8_t* phb = phbuf + gx * PHB;
    uint32_t xo[4];  // swizzled chunk offsets of this thread's weight chunks within a row
#pragma unroll
    for (int jj = 0; jj < 4; ++jj) xo[jj] = static_cast<uint32_t>(((4 * hh + jj) ^ (Rb & 7)) << 4);
    bool ok = true;
    int s = 0, so = 0, ph = 0;
    for (int ti = 0; ti < my_tiles && ok; ++ti) {
      int m0, n0;
      tile_mn(ti, m0, n0);
      ok = mbar_wait_inline(&rfull[ti & 1], (ti >> 1) & 1, wc);
      if (!ok) break;
      const float mul = rslot[(ti & 1) * BM + r].x;
      for (int st = 0; st < nst && ok; ++st, ++so) {
        const bool kst = st < nks;
        const int ps = s % SP;
        const int pphase = (s / SP) & 1;
        if (kst) ++s;
        if ((so & 1) != gx) continue;  // the other group's stage
        const int os = so % SO;
        if (so >= SO) ok = mbar_wait_inline(&oempty[os], ((so / SO) & 1) ^ 1, wc);
        if (!ok) break;
        tc_fence_after();
        uint8_t* dst = bring + os * BSTAGE;
        uint32_t v[16];
        if (kst) {
          ok = mbar_wait_inline(&pfull[ps], pphase, wc);
          if (!ok) break;
          const uint8_t* pk = pring + ps * PSTAGE;
          // every load of the stage first (the operand stores may alias them as far as the
          // compiler knows), then the conversions and stores
          const uint4 wa = *reinterpret_cast<const uint4*>(pk + r * (KS / 2) + 16 * h);
          const __nv_bfloat16 sxa = reinterpret_cast<const __nv_bfloat16*>(pk + PA)[(GPS == 2 ? h : 0) * BM + r];
          uint4 wb[2];
          __half swb[2];
          if (!PREB) {
#pragma unroll
            for (int i = 0; i < 2; ++i) {
              const int R = Rb + 16 * i;
              wb[i] = *reinterpret_cast<const uint4*>(pbring + ps * PB + R * (KS / 2) + 16 * hh);
              swb[i] = reinterpret_cast<const __half*>(pk + PA + PSX)[(GPS == 2 ? hh : 0) * BN + R];
            }
          }
          const DqScale da = scale_consts(sxa, mul);
          dequant_word(wa.x, da, v + 0);
          dequant_word(wa.y, da, v + 4);
          dequant_word(wa.z, da, v + 8);
          dequant_word(wa.w, da, v + 12);
#pragma unroll
          for (int i = 0; i < (PREB ? 0 : 2); ++i) {
            const DqScale db = dq_scale(__half2float(swb[i]));
            uint8_t* row = dst + (Rb + 16 * i) * 128;
            const uint32_t wv[4] = {wb[i].x, wb[i].y, wb[i].z, wb[i].w};
#pragma unroll
            for (int jj = 0; jj < 4; ++jj) {
              uint32_t o[4];
              dequant_word(wv[jj], db, o);
              *reinterpret_cast<uint4*>(row + xo[jj]) = make_uint4(o[0], o[1], o[2], o[3]);
            }
          }
          // orders the operand writes before the MMA reads them, and the packed reads before TMA
          // refills the stage
          fence_proxy_async_smem();
          warp_arrive(&pempty[ps]);
        } else {
          // branch stage: p_hat 2^e_m into TMEM (exact unless p_hat itself is zero: then 0), and
          // B_hat 2^e_n by TMA straight into the operand stage (its bytes complete the stage's
          // barrier together with the eight arrivals)
          if (ph > 0) ok = mbar_wait_inline(&phempty[gx], (ph - 1) & 1, wc);  // the group's last p_hat was read
          if (!ok) break;
          if (e == 0) {
            if (elect_one()) {
              if (!PREB) {  // (with PREB the producer brings B_hat with the other weight stages)
                mbar_expect_tx(&ofull[os], BSTAGE);
                tma_load_2d(dst, &bh_map, &ofull[os], (st - nks) * KS, n0);
              }
              mbar_arrive_expect_tx(&phfull[gx], PHB);
              tma_load_2d(phb, &ph_map, &phfull[gx], (st - nks) * KS, m0);
            }
            __syncwarp();
          }
          ok = mbar_wait_inline(&phfull[gx], ph & 1, wc);
          ++ph;
          if (!ok) break;
#pragma unroll
          for (int c = 0; c < 4; ++c) {
            const uint4 u = *reinterpret_cast<const uint4*>(phb + r * 128 + (((4 * h + c) ^ (r & 7)) << 4));
            const uint32_t w4[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
            for (int t = 0; t < 4; ++t) v[4 * c + t] = f32x2_to_f16x2(f16_lo(w4[t]) * mul, f16_hi(w4[t]) * mul);
          }
          fence_proxy_async_smem();
          warp_arrive(&phempty[gx]);
        }
        tmem_st16(tlane + static_cast<uint32_t>(os * 32), v);
        tmem_st_wait();
        tc_fence_before();
        warp_arrive(&ofull[os]);
      }
      warp_arrive(&rempty[ti & 1]);
    }
    // the last TMA loads this warp issued have landed (they have, unless the kernel aborted first)
    int never = 0;
    const WaitCtl dc{&never, a.err, globaltimer_ns() + a.timeout_ns};
    if (ph > 0) mbar_wait_inline(&phfull[gx], (ph - 1) & 1, dc);
    if (!PREB && e == 0 && nbs > 0) {
      // this group's last branch stage: its B_hat load completed the stage's barrier
      int lb = -1;
      for (int j = so - 1; j >= 0 && j >= so - nbs; --j)
        if ((j & 1) == gx) {
          lb = j;
          break;
        }
      if (lb >= 0) mbar_wait_inline(&ofull[lb % SO], (lb / SO) & 1, dc);
    }
  } else if (wid >= 20) {
    // ------------------------------------------------------------- epilogue and row scales
    const int ew = static_cast<int>(wid) - 20;
    const int q = ew & 3, hf = ew >> 2;
    const int r = 32 * q + static_cast<int>(lane);
    const uint32_t tbase = tmem + (static_cast<uint32_t>(32 * q) << 16) + static_cast<uint32_t>(128 * hf);
    float* fcb = efb + ew * (EFB / 4);  // [0, 128): 2^-e_n, [128, 256): bias of columns n0 + 128 hf ..
    // Row scales of tile tt into slot tt % 2: thread u takes row u / 2 and every other group from
    // u % 2 (and that half of p_hat); the pair combines by a shuffle.  a_m = max(7 max_g s_x[m, g],
    // max_j |p_hat[m, j]|) gives e_m = 10 - floor(log2 a_m).
    const int u = 32 * ew + static_cast<int>(lane);
    const int rr = u >> 1, hs = u & 1;
    const int ng = a.K / G;
    auto rowscale = [&](int tt) -> bool {
      int m0t, n0t;
      tile_mn(tt, m0t, n0t);
      const int sl = tt & 1;
      if (tt >= 2 && !mbar_wait_inline(&rempty[sl], ((tt >> 1) & 1) ^ 1, wc)) return false;
      const int m = m0t + rr;  // < M_pad (a multiple of 128)
      const __nv_bfloat16* sp = a.sx + m;
      // (the workspace was written by the previous kernel of the stream, complete before pdl_wait)
      auto sx_at = [&](int g) { return __uint_as_float(ld_nc_u16(sp + static_cast<size_t>(g) * a.M_pad) << 16); };
      // the first p_hat pieces are loaded ahead of the scales, so that both are in flight together
      const bool has_ph = a.r_pad > 0 && m < a.M;
      const uint4* pr = has_ph ? reinterpret_cast<const uint4*>(a.phat + static_cast<size_t>(m) * a.r_pad) + hs * (a.r_pad / 16)
                               : nullptr;
      const int nph = has_ph ? a.r_pad / 16 : 0;  // 16-byte pieces of this thread's half row
      uint4 ph4[2];
#pragma unroll
      for (int j = 0; j < 2; ++j) ph4[j] = j < nph ? ld_nc_v4(pr + j) : make_uint4(0u, 0u, 0u, 0u);
      float s0 = 0.0f, s1 = 0.0f, s2 = 0.0f, s3 = 0.0f;
      int g = hs;
#pragma unroll 4
      for (; g + 6 < ng; g += 8) {  // up to 16 independent loads in flight
        s0 = fmaxf(s0, sx_at(g));
        s1 = fmaxf(s1, sx_at(g + 2));
        s2 = fmaxf(s2, sx_at(g + 4));
        s3 = fmaxf(s3, sx_at(g + 6));
      }
      for (; g < ng; g += 2) s0 = fmaxf(s0, sx_at(g));
      float am = 7.0f * fmaxf(fmaxf(s0, s1), fmaxf(s2, s3));  // exact: 8 + 3 significant bits
      auto ph_max = [&](const uint4& u4) {
        const uint32_t w4[4] = {u4.x, u4.y, u4.z, u4.w};
#pragma unroll
        for (int t = 0; t < 4; ++t) am = fmaxf(am, fmaxf(fabsf(f16_lo(w4[t])), fabsf(f16_hi(w4[t]))));
      };
#pragma unroll
      for (int j = 0; j < 2; ++j) ph_max(ph4[j]);  // (zero pieces past nph leave am as it is)
#pragma unroll 4
      for (int j = 2; j < nph; ++j) ph_max(ld_nc_v4(pr + j));
      am = fmaxf(am, __shfl_xor_sync(0xFFFFFFFFu, am, 1));
      int e = 0;
      if (am > 0.0f) {
        int ex;
        frexpf(am, &ex);  // am in [2^(ex-1), 2^ex)
        e = min(126, max(-126, 11 - ex));
      }
      if (hs == 0) rslot[sl * BM + rr] = make_float2(ldexpf(1.0f, e), ldexpf(1.0f, -e));
      warp_arrive(&rfull[sl]);
      return true;
    };
    bool ok = true;
    if (my_tiles > 0) ok = rowscale(0);
    if (ok && my_tiles > 1) ok = rowscale(1);
    for (int ti = 0; ti < my_tiles && ok; ++ti) {
      int m0, n0;
      tile_mn(ti, m0, n0);
      {  // this warp's columns' 2^-e_n and bias, staged while the tile's MMAs run
        const int n = n0 + 128 * hf + 4 * static_cast<int>(lane);  // < N_pad
        reinterpret_cast<float4*>(fcb)[lane] = *reinterpret_cast<const float4*>(a.fcol + n);
        float4 b = make_float4(0.f, 0.f, 0.f, 0.f);
        if (ybias && n < a.N) b = *reinterpret_cast<const float4*>(ybias + n);
        reinterpret_cast<float4*>(fcb + 128)[lane] = b;
        __syncwarp();
      }
      ok = mbar_wait_inline(&rfull[ti & 1], (ti >> 1) & 1, wc);
      if (ok) ok = mbar_wait_inline(accfull, ti & 1, wc);
      if (!ok) break;
      tc_fence_after();
      const float fm = rslot[(ti & 1) * BM + r].y;
      warp_arrive(&rempty[ti & 1]);
      const int m = m0 + r;
      if constexpr (PREB) {
        // Output through the staging buffer: this warp's 32 rows x 32 columns of a chunk (fp32), or
        // of two chunks (bf16), 128 bytes per row in the 128-byte swizzle, then one TMA store of
        // the box (rows >= M and columns >= N are not written).
        uint8_t* stg = pbring + (ew >> 1) * PB + (ew & 1) * YSTG;
        uint8_t* srow = stg + lane * 128;
        const uint32_t sw = lane & 7u;
        auto cols8p = [&](int cb, const uint32_t* av, float (&y)[8]) {  // cb: column within the warp's 128
          const float4 f0 = reinterpret_cast<const float4*>(fcb)[cb / 4];
          const float4 f1 = reinterpret_cast<const float4*>(fcb)[cb / 4 + 1];
          const float fn[8] = {f0.x, f0.y, f0.z, f0.w, f1.x, f1.y, f1.z, f1.w};
#pragma unroll
          for (int t = 0; t < 8; ++t) y[t] = (__uint_as_float(av[t]) * fn[t]) * fm;
          if (ybias) {
            const float4 b0 = reinterpret_cast<const float4*>(fcb + 128)[cb / 4];
            const float4 b1 = reinterpret_cast<const float4*>(fcb + 128)[cb / 4 + 1];
            y[0] += b0.x; y[1] += b0.y; y[2] += b0.z; y[3] += b0.w;
            y[4] += b1.x; y[5] += b1.y; y[6] += b1.z; y[7] += b1.w;
          }
        };
#pragma unroll 1
        for (int c = 0; c < 4; ++c) {
          uint32_t acc[32];
          tmem_ld32(tbase + 32 * c, acc);
          tmem_ld_wait_dep(acc);
          if (c == 3) {
            // the tile's accumulator has been read: the MMA may start the next tile
            tc_fence_before();
            warp_arrive(accempty);
          }
          if (yf32 || (c & 1) == 0) {  // the buffer is free once the last store has read it
            if (lane == 0) bulk_wait_read();
            __syncwarp();
          }
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            float y[8];
            cols8p(32 * c + 8 * j, acc + 8 * j, y);
            if (yf32) {
              *reinterpret_cast<float4*>(srow + (((2u * j) ^ sw) << 4)) = make_float4(y[0], y[1], y[2], y[3]);
              *reinterpret_cast<float4*>(srow + (((2u * j + 1u) ^ sw) << 4)) = make_float4(y[4], y[5], y[6], y[7]);
            } else {
              *reinterpret_cast<uint4*>(srow + ((static_cast<uint32_t>(4 * (c & 1) + j) ^ sw) << 4)) =
                  make_uint4(f32x2_to_bf16x2(y[0], y[1]), f32x2_to_bf16x2(y[2], y[3]), f32x2_to_bf16x2(y[4], y[5]),
                             f32x2_to_bf16x2(y[6], y[7]));
            }
          }
          if (yf32 || (c & 1) == 1) {
            fence_proxy_async_smem();  // the staged rows, before the async proxy reads them
            __syncwarp();
            if (lane == 0) {
              tma_store_2d(&y_map, stg, n0 + 128 * hf + (yf32 ? 32 * c : 64 * (c >> 1)), m0 + 32 * q);
              bulk_commit();
            }
          }
        }
      } else if (split && m0 + 32 * q >= a.M) {
        // Split-K, a lane quadrant with no row of the layer: nothing to write
        tc_fence_before();
        warp_arrive(accempty);
      } else if (split && a.M - m0 > 32) {
        // Split-K: this warp's scaled partial (no bias), 32 rows x 32 columns a chunk, through a
        // staging buffer in the operand ring (idle once the item's MMAs have completed) and a TMA
        // store into the CTA's slice of the workspace (rows >= M and columns >= N not written).
        // (With one quadrant of rows the direct stores below finish sooner: the store's
        // completion is waited for before the cluster barrier.)
        uint8_t* stg = bring + ew * YSTG;
        uint8_t* srow = stg + lane * 128;
        const uint32_t sw = lane & 7u;
#pragma unroll 1
        for (int c = 0; c < 4; ++c) {
          uint32_t acc[32];
          tmem_ld32(tbase + 32 * c, acc);
          tmem_ld_wait_dep(acc);
          if (c == 3) {
            tc_fence_before();
            warp_arrive(accempty);
          }
          if (lane == 0) bulk_wait_read();  // the buffer's last store has read it
          __syncwarp();
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const int cb = 32 * c + 8 * j;  // column within the warp's 128
            const float4 f0 = reinterpret_cast<const float4*>(fcb)[cb / 4];
            const float4 f1 = reinterpret_cast<const float4*>(fcb)[cb / 4 + 1];
            *reinterpret_cast<float4*>(srow + (((2u * j) ^ sw) << 4)) =
                make_float4((__uint_as_float(acc[8 * j]) * f0.x) * fm, (__uint_as_float(acc[8 * j + 1]) * f0.y) * fm,
                            (__uint_as_float(acc[8 * j + 2]) * f0.z) * fm, (__uint_as_float(acc[8 * j + 3]) * f0.w) * fm);
            *reinterpret_cast<float4*>(srow + (((2u * j + 1u) ^ sw) << 4)) =
                make_float4((__uint_as_float(acc[8 * j + 4]) * f1.x) * fm, (__uint_as_float(acc[8 * j + 5]) * f1.y) * fm,
                            (__uint_as_float(acc[8 * j + 6]) * f1.z) * fm, (__uint_as_float(acc[8 * j + 7]) * f1.w) * fm);
          }
          fence_proxy_async_smem();  // the staged rows, before the async proxy reads them
          __syncwarp();
          if (lane == 0) {
            tma_store_3d(&y_map, stg, n0 + 128 * hf + 32 * c, m0 + 32 * q, rank);
            bulk_commit();
          }
        }
        if (lane == 0) {  // the partial is written before this CTA reaches the cluster barrier
          bulk_wait_all();
          fence_proxy_async_all();
        }
        __syncwarp();
      } else {
  #pragma unroll 1
        for (int c = 0; c < 4; ++c) {
          uint32_t acc[32];
          tmem_ld32(tbase + 32 * c, acc);
          tmem_ld_wait_dep(acc);
          if (c == 3) {
            // the tile's accumulator has been read: the MMA may start the next tile
            tc_fence_before();
            warp_arrive(accempty);
          }
          const int nb = n0 + 128 * hf + 32 * c;
          if (m < a.M) {
  #pragma unroll
            for (int j2 = 0; j2 < 2; ++j2) {  // 16 columns at a time: one 32-byte store per row (bf16)
              const int n = nb + 16 * j2;
              if (n >= a.N) continue;
              // results of columns n + 8 h8 .. + 7: (acc 2^-e_n) 2^-e_m (+ bias)
              auto cols8 = [&](int h8, float (&y)[8]) {
                const int cb = 32 * c + 16 * j2 + 8 * h8;  // column within the warp's 128
                const float4 f0 = reinterpret_cast<const float4*>(fcb)[cb / 4];
                const float4 f1 = reinterpret_cast<const float4*>(fcb)[cb / 4 + 1];
                const float fn[8] = {f0.x, f0.y, f0.z, f0.w, f1.x, f1.y, f1.z, f1.w};
  #pragma unroll
                for (int t = 0; t < 8; ++t) y[t] = (__uint_as_float(acc[16 * j2 + 8 * h8 + t]) * fn[t]) * fm;
                if (ybias) {
                  const float4 b0 = reinterpret_cast<const float4*>(fcb + 128)[cb / 4];
                  const float4 b1 = reinterpret_cast<const float4*>(fcb + 128)[cb / 4 + 1];
                  y[0] += b0.x; y[1] += b0.y; y[2] += b0.z; y[3] += b0.w;
                  y[4] += b1.x; y[5] += b1.y; y[6] += b1.z; y[7] += b1.w;
                }
              };
              const size_t off = static_cast<size_t>(m) * a.N + n;
              const bool two = n + 16 <= a.N;  // N is a multiple of 8: the second 8 may lie past it
              if (yf32) {
                float* yp = static_cast<float*>(yout) + off;
  #pragma unroll
                for (int h8 = 0; h8 < 2; ++h8) {
                  if (h8 == 1 && !two) break;
                  float y[8];
                  cols8(h8, y);
                  uint32_t u[8];
  #pragma unroll
                  for (int t = 0; t < 8; ++t) u[t] = __float_as_uint(y[t]);
                  if ((off & 7) == 0) {
                    st_global_v8(yp + 8 * h8, u);
                  } else {
                    st_global_v4(yp + 8 * h8, u[0], u[1], u[2], u[3]);
                    st_global_v4(yp + 8 * h8 + 4, u[4], u[5], u[6], u[7]);
                  }
                }
              } else {
                __nv_bfloat16* yp = static_cast<__nv_bfloat16*>(yout) + off;
                uint32_t u[8];
                {
                  float y[8];
                  cols8(0, y);
  #pragma unroll
                  for (int t = 0; t < 4; ++t) u[t] = f32x2_to_bf16x2(y[2 * t], y[2 * t + 1]);
                }
                if (two) {
                  float y[8];
                  cols8(1, y);
  #pragma unroll
                  for (int t = 0; t < 4; ++t) u[4 + t] = f32x2_to_bf16x2(y[2 * t], y[2 * t + 1]);
                }
                if (two && (off & 15) == 0) {
                  st_global_v8(yp, u);
                } else {
                  st_global_v4(yp, u[0], u[1], u[2], u[3]);
                  if (two) st_global_v4(yp + 8, u[4], u[5], u[6], u[7]);
                }
              }
            }
          }
        }
      }
      __syncwarp();  // every lane's reads of the staged columns are done before the next tile's
      if (ti + 2 < my_tiles) ok = rowscale(ti + 2);
    }
    if (PREB) {  // every output store is complete before the CTA exits
      if (lane == 0) bulk_wait_all();
      __syncwarp();
    }
    tmem_ld_wait();
  }

  if (!PREB && split) {
    // Every thread of the cluster arrives here once its role is done; the barrier's release /
    // acquire orders the partial tiles written above before the reads below.
    cluster_sync();
    int m0, n0;
    tile_mn(0, m0, n0);
    const int W = BN / a.splits;  // this CTA's columns of the tile
    const int c0 = n0 + rank * W;
    const int rows = min(BM, a.M - m0);
    const int w4 = W / 4;
    const size_t slice = static_cast<size_t>(a.M) * a.N;
    for (int i = static_cast<int>(threadIdx.x); i < rows * w4; i += kThreads) {
      const int m = m0 + i / w4, n = c0 + 4 * (i % w4);
      if (n >= a.N) continue;  // N is a multiple of 8, so n < N covers n .. n + 3
      const float* pp = a.part + static_cast<size_t>(m) * a.N + n;
      float4 v[8];  // every split's partial in flight at once (splits <= 8), summed in rank order
#pragma unroll
      for (int q = 0; q < 8; ++q)
        v[q] = q < a.splits ? *reinterpret_cast<const float4*>(pp + q * slice) : make_float4(0.f, 0.f, 0.f, 0.f);
      float4 y = v[0];
#pragma unroll
      for (int q = 1; q < 8; ++q) {
        if (q >= a.splits) break;
        y.x += v[q].x;
        y.y += v[q].y;
        y.z += v[q].z;
        y.w += v[q].w;
      }
      if (a.bias) {
        const float4 b = *reinterpret_cast<const float4*>(a.bias + n);
        y.x += b.x;
        y.y += b.y;
        y.z += b.z;
        y.w += b.w;
      }
      const size_t off = static_cast<size_t>(m) * a.N + n;
      if (a.y_f32) {
        *reinterpret_cast<float4*>(static_cast<float*>(a.Y) + off) = y;
      } else {
        *reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(a.Y) + off) =
            make_uint2(f32x2_to_bf16x2(y.x, y.y), f32x2_to_bf16x2(y.z, y.w));
      }
    }
  }

  __syncthreads();
  if (wid == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}

template <int G, bool PREB>
cudaError_t launch_g(Handle& h, const ActMaps& am, const ActLayout& L, const void* ws, int M, void* Y, bool y_f32,
                     cudaStream_t s, bool w16_ready) {
  const uint8_t* base = static_cast<const uint8_t*>(ws);
  GemmArgs a;
  a.M = M;
  a.N = h.N;
  a.K = h.K;
  a.r_pad = h.r_pad;
  a.M_pad = L.M_pad;
  a.nbs = (h.r_pad + KS - 1) / KS;
  a.m_tiles = (M + BM - 1) / BM;
  a.n_tiles = (h.N + BN - 1) / BN;
  a.sx = reinterpret_cast<const __nv_bfloat16*>(base + L.scales_off);
  a.phat = h.r_pad > 0 ? reinterpret_cast<const __half*>(base + L.phat_off) : nullptr;
  a.fcol = h.fcol;
  a.Y = Y;
  a.y_f32 = y_f32 ? 1 : 0;
  a.bias = h.bias;
  a.splits = L.gsplit_off ? gemm_split(M, h.N, h.K, h.num_sms) : 1;
  a.part = L.gsplit_off ? reinterpret_cast<float*>(const_cast<uint8_t*>(base) + L.gsplit_off) : nullptr;
  a.err = h.err;
  a.timeout_ns = deadline_budget_ns(h);
  static bool attr_done = false;
  if (!attr_done) {
    cudaError_t e = cudaFuncSetAttribute(gemm16_kernel<G, PREB>, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM);
    if (e != cudaSuccess) return e;
    attr_done = true;
  }
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;  // split-K: the splits of a tile form a cluster
  attr[1].val.clusterDim.x = a.splits;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (PREB && !w16_ready) {
    const long long pieces = static_cast<long long>(h.N_pad) * ((h.K + h.r_pad) / 8);
    const long long blocks = (pieces + 8 * 256 - 1) / (8 * 256);  // eight pieces a thread
    cfg.gridDim = dim3(static_cast<unsigned>(blocks < 8 * h.num_sms ? blocks : 8 * h.num_sms), 1, 1);
    cfg.blockDim = dim3(256, 1, 1);
    cfg.dynamicSmemBytes = 0;
    cudaError_t e = cudaLaunchKernelEx(&cfg, dequant_weights_kernel, w16_args(h, L, base));
    if (e != cudaSuccess) return e;
  }
  const int ntiles = a.m_tiles * a.n_tiles;
  const int grid = a.splits > 1 ? ntiles * a.splits : (ntiles < h.num_sms ? ntiles : h.num_sms);
  cfg.numAttrs = a.splits > 1 ? 2 : 1;
  // With PREB every weight stage comes through the expanded-weight map; without a branch the
  // p_hat / B_hat maps are never used and any valid map fills the slots.
  const CUtensorMap& ph = (h.r_pad > 0) ? am.ph64_map : am.qa_map;
  const CUtensorMap& bh = PREB ? am.w16_map : ((h.r_pad > 0) ? h.bhs_map : am.qa_map);
  // PREB stores the output by TMA (the map of Y), the split-K GEMM its partials (their map);
  // otherwise any valid map fills the slot.
  const CUtensorMap* ym = PREB ? get_y_map(h, Y, M, y_f32)
                               : (a.splits > 1 ? get_part_map(h, a.part, M, a.splits) : &am.qa_map);
  if (!ym) return cudaErrorInvalidValue;
  cfg.gridDim = dim3(grid, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = SMEM;
  return cudaLaunchKernelEx(&cfg, gemm16_kernel<G, PREB>, am.qa_map, h.qw_map, am.sx_map, h.swh_map, ph, bh, *ym, a);
}

}  // namespace

W16Args w16_args(const Handle& h, const ActLayout& L, const void* ws) {
  W16Args w;
  w.qw = reinterpret_cast<const uint32_t*>(h.qw);
  w.swh = h.swh;
  w.bhs = h.Bhs;
  w.w16 = L.w16_off ? reinterpret_cast<__half*>(static_cast<uint8_t*>(const_cast<void*>(ws)) + L.w16_off) : nullptr;
  w.K = h.K;
  w.r_pad = h.r_pad;
  w.N_pad = h.N_pad;
  w.gshift = h.G == 32 ? 2 : 3;
  return w;
}

cudaError_t launch_gemm(Handle& h, const ActMaps& am, const void* ws, int M, void* Y, bool y_f32, cudaStream_t s,
                        bool lean, bool w16_ready) {
  const ActLayout L = act_layout(h, M, lean);
  if (L.w16_off)
    return h.G == 32 ? launch_g<32, true>(h, am, L, ws, M, Y, y_f32, s, w16_ready)
                     : launch_g<64, true>(h, am, L, ws, M, Y, y_f32, s, w16_ready);
  return h.G == 32 ? launch_g<32, false>(h, am, L, ws, M, Y, y_f32, s, false)
                   : launch_g<64, false>(h, am, L, ws, M, Y, y_f32, s, false);
}

}  // namespace qwam
