// gemm_nvfp4.cu -- kernel (b) of the NVFP4 variant (App. B.1: on Blackwell the paper stores
// E2M1 values with an E4M3 scale for every 16 elements, for weights and activations, and one
// float32 scale per weight tensor), with the 16-bit branch of Eq. (asp) in the epilogue:
//
//   Y[m, n] = s_g * sum_b s_a[m, b] s_b[n, b] sum_{k in b} qa[m, k] qb[n, k]  +  p_hat[m, :] B_hat[n, :]
//
// The block scales are applied by the tensor cores: tcgen05.mma.kind::mxf4nvf4.block_scale with
// scale_vec::4X multiplies each 16-wide block's partial product by its row's and column's UE4M3
// scales and accumulates in float32 in TMEM, so there is no per-block work outside the MMA.  The
// epilogue runs once per output tile: Y = s_g D + branch.
//
// Persistent CTAs (one per SM) walk 128 x 128 output tiles with a static stride.  192 threads:
//   warp 0   TMA producer: per stage of 256 K, the two 16 KB code tiles (128-byte swizzle) and
//            the two 2 KB scale-atom blocks (plain bulk copies; see internal.h for the atom);
//   warp 1   MMA issuer and TMEM owner (warp-wide loop, one elected lane issues): copies a
//            stage's scale atoms into TMEM
//            (tcgen05.cp.32x128b.warpx4, which puts the 32 x 16 bytes of an atom into all four
//            lane quarters, where the MMA reads them), then issues four 128x128x64 MMAs;
//            tcgen05 operations of one thread run in issue order, so a scale slot is rewritten
//            only after the MMAs that read it;
//   warps 2-5 epilogue: one TMEM lane quarter each (thread = output row), 32x32b loads; warp 2
//            also issues each tile's branch MMA, so the MMA issuer never waits on the branch.
// TMEM: two accumulators (columns 0..255), the branch accumulator (256..383), four scale slots
// of 32 columns (384..511: A at +0, B at +16, four columns per MMA).
#include "internal.h"
#include "ptx.cuh"

namespace qwam {
namespace {

struct Gemm4Args {
  int M, N, K;
  int m_tiles, n_tiles;
  const uint8_t* sfa;  // activation scale atoms (workspace), M_pad rows
  const uint8_t* sfb;  // weight scale atoms (handle), N_pad rows
  float sg;            // per-tensor weight scale
  void* Y;
  int y_f32;
  const float* bias;  // optional [N], added to the float32 result before it is stored
  int* err;
  uint64_t timeout_ns;
};

constexpr int kThreads4 = 192;
constexpr int NS4 = 5;                                       // operand stages
constexpr int A4_BYTES = kBM * kFp4KS / 2;                   // 16 KB
constexpr int B4_BYTES = kGemmBN * kFp4KS / 2;               // 16 KB
constexpr int SF4_BYTES = (kFp4KS / 64) * kSfAtom;           // 2 KB per operand
constexpr int STAGE4 = A4_BYTES + B4_BYTES + 2 * SF4_BYTES;  // 36 KB
constexpr int NSF = 4;                                       // TMEM scale slots
constexpr uint32_t kColBranch = 256, kColScale = 384;

template <int RP>
struct Gemm4Cfg {
  static constexpr int BR_BYTES = RP * kBM * 2;  // p_hat tile (and the B_hat tile): RP/8 boxes of 2 KB
  static constexpr int NBAR = 2 * NS4 + 4 + 4 + 1;
  static constexpr int SMEM = 1024 + NS4 * STAGE4 + 2 * BR_BYTES + NBAR * 8 + 16;
  static_assert(SMEM <= 232448, "NVFP4 GEMM shared memory above the 227 KB per-CTA limit");
};

template <int RP>
__global__ void __launch_bounds__(kThreads4, 1)
    gemm_nvfp4_kernel(const __grid_constant__ CUtensorMap qa_map, const __grid_constant__ CUtensorMap qb_map,
                      const __grid_constant__ CUtensorMap ph_map, const __grid_constant__ CUtensorMap bh_map,
                      const Gemm4Args a) {
  using Cfg = Gemm4Cfg<RP>;
  extern __shared__ uint8_t smem_raw[];
  pdl_launch_dependents();
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* stages = smem;                       // NS4 x (A | B | SF_A | SF_B)
  uint8_t* br = stages + NS4 * STAGE4;          // p_hat | B_hat
  uint64_t* bars = reinterpret_cast<uint64_t*>(br + 2 * Cfg::BR_BYTES);
  uint64_t* full = bars;
  uint64_t* empty = full + NS4;
  uint64_t* tfull = empty + NS4;      // [2]
  uint64_t* tempty = tfull + 2;       // [2]
  uint64_t* bfull = tempty + 2;       // branch operands landed
  uint64_t* bempty = bfull + 1;       // branch operands consumed by the MMA
  uint64_t* brfull = bempty + 1;      // branch accumulator ready
  uint64_t* brempty = brfull + 1;     // branch accumulator read by the epilogue
  uint64_t* drain = brempty + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + Cfg::NBAR);
  int* abort_flag = reinterpret_cast<int*>(tmem_slot + 1);

  const uint32_t wid = warp_id(), lane = lane_id();
  const int nst = a.K / kFp4KS;
  const int nkc = a.K / 64;
  const int ntiles = a.m_tiles * a.n_tiles;
  const int my_tiles = ntiles > static_cast<int>(blockIdx.x)
                           ? (ntiles - static_cast<int>(blockIdx.x) + static_cast<int>(gridDim.x) - 1) /
                                 static_cast<int>(gridDim.x)
                           : 0;
  auto tile_mn = [&](int i, int& m0, int& n0) {
    const int t = static_cast<int>(blockIdx.x) + i * static_cast<int>(gridDim.x);
    m0 = (t / a.n_tiles) * kBM;
    n0 = (t % a.n_tiles) * kGemmBN;
  };
  auto stage = [&](int slot) { return stages + slot * STAGE4; };

  if (threadIdx.x == 0) {
    for (int i = 0; i < NS4; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&tfull[i], 1);
      mbar_init(&tempty[i], 4);
    }
    mbar_init(bfull, 1);
    mbar_init(bempty, 1);
    mbar_init(brfull, 1);
    mbar_init(brempty, 4);
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

  if (wid == 0) {
    // ------------------------------------------------------------- TMA producer
    bool ok = true;
    int s = 0;
    for (int ti = 0; ti < my_tiles && ok; ++ti) {
      int m0, n0;
      tile_mn(ti, m0, n0);
      const uint8_t* sfa = a.sfa + static_cast<size_t>(m0 / kBM) * nkc * kSfAtom;
      const uint8_t* sfb = a.sfb + static_cast<size_t>(n0 / kGemmBN) * nkc * kSfAtom;
      for (int st = 0; st < nst && ok; ++st, ++s) {
        const int slot = s % NS4;
        if (s >= NS4) ok = mbar_wait_inline(&empty[slot], ((s / NS4) & 1) ^ 1, wc);
        if (!ok) break;
        uint8_t* p = stage(slot);
        if (elect_one()) {
          mbar_arrive_expect_tx(&full[slot], STAGE4);
          tma_load_2d(p, &qa_map, &full[slot], st * (kFp4KS / 2), m0);
          tma_load_2d(p + A4_BYTES, &qb_map, &full[slot], st * (kFp4KS / 2), n0);
          bulk_load_1d(p + A4_BYTES + B4_BYTES, sfa + static_cast<size_t>(st) * SF4_BYTES, SF4_BYTES, &full[slot]);
          bulk_load_1d(p + A4_BYTES + B4_BYTES + SF4_BYTES, sfb + static_cast<size_t>(st) * SF4_BYTES, SF4_BYTES,
                       &full[slot]);
        }
        __syncwarp();
      }
      if constexpr (RP > 0) {
        if (ok && ti >= 1) ok = mbar_wait_inline(bempty, (ti & 1) ^ 1, wc);
        if (!ok) break;
        if (elect_one()) {
          mbar_arrive_expect_tx(bfull, 2 * Cfg::BR_BYTES);
          for (int q = 0; q < RP / 8; ++q) {
            tma_load_2d(br + q * 2048, &ph_map, bfull, q * 8, m0);
            tma_load_2d(br + Cfg::BR_BYTES + q * 2048, &bh_map, bfull, q * 8, n0);
          }
        }
        __syncwarp();
      }
    }
    // Let every issued load land before the CTA can exit.
    int never = 0;
    const WaitCtl dc{&never, a.err, globaltimer_ns() + a.timeout_ns};
    for (int j = (s > NS4 ? s - NS4 : 0); j < s; ++j) mbar_wait_inline(&full[j % NS4], (j / NS4) & 1, dc);
    if constexpr (RP > 0) {
      if (my_tiles > 0) mbar_wait_inline(bfull, (my_tiles - 1) & 1, dc);
    }
  } else if (wid == 1) {
    // ------------------------------------------------------------- MMA issuer
    // The whole warp walks the loop (warp-uniform counters and descriptors); one elected lane
    // issues.  The tensor pipe queues little ahead of the issuing thread, so the work between
    // MMAs is kept small: counters advance by increments, descriptors are offsets from
    // precomputed bases, and the 16-bit branch MMA is issued by an epilogue warp instead.
    bool ok = true;
    constexpr uint32_t idesc = idesc_nvf4(kBM, kGemmBN);
    const uint32_t s0 = smem_u32(stages);
    const uint64_t adesc_base = smem_desc(s0, 16, 1024, kSw128);
    const uint64_t bdesc_base = smem_desc(s0 + A4_BYTES, 16, 1024, kSw128);
    const uint64_t sadesc_base = smem_desc(s0 + A4_BYTES + B4_BYTES, 128, 128, kSwNone);
    const uint64_t sbdesc_base = smem_desc(s0 + A4_BYTES + B4_BYTES + SF4_BYTES, 128, 128, kSwNone);
    int slot = 0, phase = 0, sfs = 0;  // operand slot, its phase bit, scale slot
    for (int ti = 0; ti < my_tiles && ok; ++ti) {
      const uint32_t d = tmem + 128u * static_cast<uint32_t>(ti & 1);
      if (ti >= 2) {
        ok = mbar_wait_inline(&tempty[ti & 1], ((ti >> 1) & 1) ^ 1, wc);
        if (!ok) break;
        tc_fence_after();
      }
      for (int st = 0; st < nst; ++st) {
        ok = mbar_wait_inline(&full[slot], phase, wc);
        if (!ok) break;
        tc_fence_after();
        const uint64_t soff = static_cast<uint64_t>(slot) * (STAGE4 >> 4);
        const uint32_t ta = tmem + kColScale + 32u * static_cast<uint32_t>(sfs), tb = ta + 16;
        if (elect_one()) {
#pragma unroll
          for (int kk = 0; kk < 4; ++kk) {
            tc_cp_32x128b_x4(ta + 4 * kk, sadesc_base + soff + kk * (kSfAtom >> 4));
            tc_cp_32x128b_x4(tb + 4 * kk, sbdesc_base + soff + kk * (kSfAtom >> 4));
          }
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)  // 32 bytes (64 codes) of each row per MMA
            mma_nvf4(d, adesc_base + soff + 2 * kk, bdesc_base + soff + 2 * kk, idesc, ta + 4 * kk, tb + 4 * kk,
                     (st | kk) != 0);
          mma_commit(&empty[slot]);
        }
        __syncwarp();
        if (++slot == NS4) {
          slot = 0;
          phase ^= 1;
        }
        sfs = (sfs + 1) & (NSF - 1);
      }
      if (!ok) break;
      if (elect_one()) mma_commit(&tfull[ti & 1]);
      __syncwarp();
    }
    if (elect_one()) mma_commit(drain);
    __syncwarp();
    int never = 0;
    const WaitCtl dc{&never, a.err, globaltimer_ns() + a.timeout_ns};
    mbar_wait_inline(drain, 0, dc);
  } else {
    // ------------------------------------------------------------- epilogue (thread = row)
    const int quad = static_cast<int>(wid & 3);
    const int row = quad * 32 + static_cast<int>(lane);
    const uint32_t tq = tmem + (static_cast<uint32_t>(quad * 32) << 16);
    bool ok = true;
    // Warp 2 issues the branch MMA p_hat B_hat^T of tile t (kind::f16, K = RP) into the branch
    // accumulator once the four epilogue warps have read tile t - 1's and the operands have landed.
    auto issue_branch = [&](int t) {
      if constexpr (RP > 0) {
        if (ok && t >= 1) ok = mbar_wait_inline(brempty, (t - 1) & 1, wc);
        if (ok) ok = mbar_wait_inline(bfull, t & 1, wc);
        tc_fence_after();
        if (ok && lane == 0) {
          constexpr uint32_t idesc_br = idesc_f16(kBM, kGemmBN);
          const uint32_t pp = smem_u32(br), pw = pp + Cfg::BR_BYTES;
          const uint64_t pdesc0 = smem_desc(pp, 2048, 128, kSwNone), wdesc0 = smem_desc(pw, 2048, 128, kSwNone);
#pragma unroll
          for (int kk = 0; kk < RP / 16; ++kk)
            mma_f16(tmem + kColBranch, pdesc0 + kk * 256, wdesc0 + kk * 256, idesc_br, kk != 0);  // 4096 B
          mma_commit(brfull);
          mma_commit(bempty);
        }
        __syncwarp();
      }
    };
    if (wid == 2 && my_tiles > 0) issue_branch(0);
    for (int ti = 0; ti < my_tiles; ++ti) {
      int m0, n0;
      tile_mn(ti, m0, n0);
      const int ub = ti & 1;
      if (ok) ok = mbar_wait_inline(&tfull[ub], (ti >> 1) & 1, wc);
      if constexpr (RP > 0) {
        if (ok) ok = mbar_wait_inline(brfull, ti & 1, wc);
      }
      tc_fence_after();
      const int m = m0 + row;
#pragma unroll 1
      for (int c = 0; c < 4; ++c) {
        uint32_t v[32], b[32];
        tmem_ld32(tq + 128u * ub + 32 * c, v);
        if constexpr (RP > 0) tmem_ld32(tq + kColBranch + 32 * c, b);
        tmem_ld_wait();
        if (c == 3) {
          tc_fence_before();
          warp_arrive(&tempty[ub]);
          if constexpr (RP > 0) warp_arrive(brempty);
        }
        if (!ok || m >= a.M) continue;
        float y[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) y[i] = fmaf(a.sg, __uint_as_float(v[i]), RP > 0 ? __uint_as_float(b[i]) : 0.0f);
        if (a.bias) {
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const int n = n0 + 32 * c + 8 * j;
            if (n >= a.N) continue;
            const float4 b0 = reinterpret_cast<const float4*>(a.bias + n)[0];
            const float4 b1 = reinterpret_cast<const float4*>(a.bias + n)[1];
            y[8 * j] += b0.x; y[8 * j + 1] += b0.y; y[8 * j + 2] += b0.z; y[8 * j + 3] += b0.w;
            y[8 * j + 4] += b1.x; y[8 * j + 5] += b1.y; y[8 * j + 6] += b1.z; y[8 * j + 7] += b1.w;
          }
        }
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const int n = n0 + 32 * c + 8 * j;  // N is a multiple of 8
          if (n >= a.N) continue;
          const size_t off = static_cast<size_t>(m) * a.N + n;
          if (a.y_f32) {
            float4* d = reinterpret_cast<float4*>(static_cast<float*>(a.Y) + off);
            d[0] = make_float4(y[8 * j], y[8 * j + 1], y[8 * j + 2], y[8 * j + 3]);
            d[1] = make_float4(y[8 * j + 4], y[8 * j + 5], y[8 * j + 6], y[8 * j + 7]);
          } else {
            uint32_t w[4];
#pragma unroll
            for (int t = 0; t < 4; ++t) {
              const __nv_bfloat162 h = __floats2bfloat162_rn(y[8 * j + 2 * t], y[8 * j + 2 * t + 1]);
              w[t] = *reinterpret_cast<const uint32_t*>(&h);
            }
            *reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(a.Y) + off) = make_uint4(w[0], w[1], w[2], w[3]);
          }
        }
      }
      if (wid == 2 && ti + 1 < my_tiles) issue_branch(ti + 1);
    }
  }

  __syncthreads();
  if (wid == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// Ranks above kMaxRank: the 16-bit branch added to the 4-bit part (float32, no bias) after the GEMM,
// one thread per output, float32 sums over j ascending:  Y = Y4 + p_hat B_hat^T (+ bias).
__global__ void __launch_bounds__(128) branch_finalize_kernel(const float* __restrict__ y4,
                                                              const __half* __restrict__ ph,
                                                              const __half* __restrict__ bh, const float* bias, int M,
                                                              int N, int rp, void* Y, int y_f32) {
  pdl_launch_dependents();
  pdl_wait();
  const int n = blockIdx.x * blockDim.x + threadIdx.x, m = blockIdx.y;
  if (n >= N || m >= M) return;
  float acc = 0.0f;
  for (int j = 0; j < rp; ++j)
    acc = fmaf(__half2float(ph[static_cast<size_t>(m) * rp + j]), __half2float(bh[static_cast<size_t>(n) * rp + j]), acc);
  float y = y4[static_cast<size_t>(m) * N + n] + acc;
  if (bias) y += bias[n];
  const size_t off = static_cast<size_t>(m) * N + n;
  if (y_f32)
    static_cast<float*>(Y)[off] = y;
  else
    static_cast<__nv_bfloat16*>(Y)[off] = __float2bfloat16_rn(y);
}

template <int RP>
cudaError_t launch_rp(Handle& h, const ActMaps& am, const void* ws, int M, void* Y, bool y_f32, cudaStream_t s,
                      bool with_bias = true) {
  using Cfg = Gemm4Cfg<RP>;
  const ActLayout L = act_layout(h, M);
  Gemm4Args a;
  a.M = M;
  a.N = h.N;
  a.K = h.K;
  a.m_tiles = (M + kBM - 1) / kBM;
  a.n_tiles = (h.N + kGemmBN - 1) / kGemmBN;
  a.sfa = static_cast<const uint8_t*>(ws) + L.scales_off;
  a.sfb = h.sfw;
  a.sg = h.sg;
  a.Y = Y;
  a.y_f32 = y_f32 ? 1 : 0;
  a.bias = with_bias ? h.bias : nullptr;
  a.err = h.err;
  a.timeout_ns = deadline_budget_ns(h);
  static bool attr_done = false;
  if (!attr_done) {
    cudaError_t e = cudaFuncSetAttribute(gemm_nvfp4_kernel<RP>, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::SMEM);
    if (e != cudaSuccess) return e;
    attr_done = true;
  }
  const int ntiles = a.m_tiles * a.n_tiles;
  const int grid = ntiles < h.num_sms ? ntiles : h.num_sms;
  const CUtensorMap& ph = (RP > 0) ? am.ph_map : am.qx4_map;
  const CUtensorMap& bh = (RP > 0) ? h.Bh_map : am.qx4_map;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid, 1, 1);
  cfg.blockDim = dim3(kThreads4, 1, 1);
  cfg.dynamicSmemBytes = Cfg::SMEM;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, gemm_nvfp4_kernel<RP>, am.qx4_map, h.qw4_map, ph, bh, a);
}

}  // namespace

cudaError_t launch_gemm_nvfp4(Handle& h, const ActMaps& am, const void* ws, int M, void* Y, bool y_f32, cudaStream_t s) {
  switch (h.r_pad) {
    case 0: return launch_rp<0>(h, am, ws, M, Y, y_f32, s);
    case 16: return launch_rp<16>(h, am, ws, M, Y, y_f32, s);
    case 32: return launch_rp<32>(h, am, ws, M, Y, y_f32, s);
    case 48: return launch_rp<48>(h, am, ws, M, Y, y_f32, s);
    case 64: return launch_rp<64>(h, am, ws, M, Y, y_f32, s);
    default: break;
  }
  if (h.r_pad <= kMaxRank) return cudaErrorInvalidValue;
  // larger ranks: the 4-bit part in float32 into the workspace, then the branch and the bias
  const ActLayout L = act_layout(h, M);
  uint8_t* base = static_cast<uint8_t*>(const_cast<void*>(ws));
  float* y4 = reinterpret_cast<float*>(base + L.ytmp_off);
  cudaError_t e = launch_rp<0>(h, am, ws, M, y4, true, s, false);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((h.N + 127) / 128, M, 1);
  cfg.blockDim = dim3(128, 1, 1);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, branch_finalize_kernel, static_cast<const float*>(y4),
                            reinterpret_cast<const __half*>(base + L.phat_off), static_cast<const __half*>(h.Bh),
                            static_cast<const float*>(h.bias), M, h.N, h.r_pad, Y, y_f32 ? 1 : 0);
}

}  // namespace qwam
