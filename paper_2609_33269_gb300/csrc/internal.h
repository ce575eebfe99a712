// internal.h -- handle layout and kernel launchers shared by the translation units of the
// library (never by the oracle).
#pragma once
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "../../include/qwam_asp.h"
#include "dequant.cuh"

namespace qwam {

constexpr int kBM = 128;        // token rows per CTA tile (one TMEM lane per row)
constexpr int kChunk = 64;      // K columns per activation chunk (bf16: one 128-byte row)
constexpr int kMaxRank = 64;    // largest rank of kernel (a)'s tensor-core path (above: the general-rank path)
constexpr int kGemmBN = 128;    // output columns per NVFP4 GEMM CTA tile
constexpr int kGemm16BN = 256;  // output columns per INT4 GEMM CTA tile (float16 tensor-core kernel)
// INT4 layers with at least this many 128-row tiles have their weights expanded to float16 once per
// call (into the workspace) instead of once per tile inside the GEMM.
constexpr int kPreExpandMinTiles = 4;

// NVFP4 variant (App. B.1): E2M1 codes, one E4M3 scale per 16 consecutive K, one float32 scale per
// weight tensor.  Block scales are stored in 512-byte atoms, one per 128 rows x 64 K: the four
// scales of row r (r = row % 128) sit at bytes (r % 32) * 16 + (r / 32) * 4 .. +3, K order, and
// atom (row / 128, k / 64) starts at ((row / 128) * (K / 64) + k / 64) * 512.
constexpr int kFp4Block = 16;   // K entries per E4M3 scale
constexpr int kFp4KS = 256;     // K entries per NVFP4 GEMM stage (128 bytes of codes per row)
constexpr int kSfAtom = 512;    // bytes per scale atom (128 rows x 64 K)
enum Format : int { kFmtInt4 = 0, kFmtNvfp4 = 1 };

inline int round_up(int a, int b) { return (a + b - 1) / b * b; }

// INT4 codes are stored packed at four bits in OB4 words (offset binary): word j of a row holds
// k = 8j .. 8j+7 as nibbles c + 8 in [1, 15], k = 8j + 2p in bits 4p .. 4p+3 and k = 8j + 2p + 1
// in bits 16 + 4p .. 16 + 4p + 3 (p = 0..3).  Pair p then becomes the float16 pair
// (c_{8j+2p}, c_{8j+2p+1}) in one 32-bit register with one shift, one and-or with
// 0x000F000F / 0x64006400 (0x6400 | n is the float16 value 1024 + n) and one float16 subtraction of
// 1032.  A zero word (TMA fill outside the tensor) decodes to -8 everywhere, and its scale to 0.
__host__ __device__ inline uint32_t ob4_word(const int (&c)[8]) {
  uint32_t w = 0;
  for (int p = 0; p < 4; ++p)
    w |= (static_cast<uint32_t>(c[2 * p] + 8) << (4 * p)) | (static_cast<uint32_t>(c[2 * p + 1] + 8) << (16 + 4 * p));
  return w;
}
// Code k (0..7) of an OB4 word.
__host__ __device__ inline int ob4_code(uint32_t w, int k) {
  return static_cast<int>((w >> ((k & 1) * 16 + (k >> 1) * 4)) & 0xFu) - 8;
}

// Activation-side tensor maps for one (workspace, X, M) triple.
struct ActMaps {
  const void* ws = nullptr;
  const void* x = nullptr;
  int M = -1;
  CUtensorMap x_map;    // X bf16 [M, K], box {64, 128}, 128-byte swizzle
  CUtensorMap qa_map;   // INT4: packed OB4 codes [M, K/2] bytes, box {32, 128}
  CUtensorMap sx_map;   // INT4: s_x bf16 [K/G, M] (row pitch M_pad), box {128, 64/G}: one GEMM stage's groups
  CUtensorMap ph_map;   // p_hat f16 [M, r_pad], box {8, 128} (NVFP4 GEMM)
  CUtensorMap ph64_map; // p_hat f16 [M, r_pad], box {64, 128}, 128-byte swizzle (INT4 GEMM)
  CUtensorMap qx4_map;  // NVFP4 codes [M, K/2] bytes, box {128, 128}, 128-byte swizzle
  CUtensorMap w16_map;  // INT4, large M: float16 weights [N_pad, K + r_pad], box {64, 256}, 128-byte swizzle
  bool lean = false;    // the layout without the expanded-weight region
};

struct Handle {
  int fmt = kFmtInt4;
  int K = 0, N = 0, r = 0, G = 0, r_pad = 0, N_pad = 0, ku3 = 0;
  int device = 0;
  int num_sms = 148;
  void* block = nullptr;             // one device allocation holding every buffer below
  uint8_t* qw = nullptr;             // INT4: [N_pad, K/2] OB4 words (word j of a row: k = 8j..8j+7,
                                     // see ob4_word); NVFP4: E2M1 codes, low nibble = even k
  __nv_bfloat16* sw = nullptr;       // INT4: s_w [K/G, N_pad], bfloat16
  // The INT4 GEMM's copies, scaled per output column n by 2^e_n (e_n chosen so that the column's
  // largest dequantized value 7 s_w, or its largest |B_hat|, lies in [2^10, 2^11)): float16
  // s_w 2^e_n [K/G, N_pad] and B_hat 2^e_n [N_pad, r_pad], and the float32 factor 2^-e_n [N_pad].
  __half* swh = nullptr;
  __half* Bhs = nullptr;
  float* fcol = nullptr;
  __half* Bh = nullptr;              // [N_pad, r_pad]
  __nv_bfloat16* ucat_t = nullptr;   // [2 r_pad, K]: rows 0..r_pad-1 = U_hi^T, then U_lo^T
  __nv_bfloat16* ucat3 = nullptr;    // [K, ku3]: row k = U_hi[k,:], U_lo[k,:], U_hi[k,:], zeros
  uint8_t* sfw = nullptr;            // NVFP4: E4M3 block scales of W_perp in atoms (N_pad rows)
  float sg = 0.0f;                   // NVFP4: float32 per-tensor weight scale
  int* err = nullptr;                // device error word (first error kept until read)
  // qwam_asp_get_error waits for the handle's last launch, not for the device: an event
  // recorded after each launch outside a stream capture, read through a stream of its own
  cudaEvent_t done = nullptr;
  bool done_valid = false;
  cudaStream_t err_stream = nullptr;
  int* err_host = nullptr;           // pinned host copy of the word
  // Smoothing and block Hadamard rotation in front of the layer (Sec. 3 Eq. (pair)): the packed
  // weight is W~ = H diag(s) W, the activations are rotated at run time, x~ = H diag(s)^-1 x.
  // ucat_t then holds diag(s)^-1 H U (the projection x~ U = x (diag(s)^-1 H U)) and ucat3 holds
  // diag(s) H U (the remainder x - diag(s) H U p, which H diag(s)^-1 maps to x~ - U p).
  bool rot = false;
  int hb = 0;                        // Hadamard block: largest power of two dividing K, <= 1024
  float* inv_s = nullptr;            // [K]: RN_f32(1 / (sqrt(hb) s_k)) (s_k = 1 without smoothing)
  float* bias = nullptr;             // optional float32 [N], added in the GEMM epilogue (own allocation)
  float* up32 = nullptr;             // [r_pad, K] float32 projection basis (U, or diag(s)^-1 H U), transposed
  float* ur32 = nullptr;             // [r_pad, K] float32 reconstruction basis (U, or diag(s) H U), transposed
  int small_m = 256;                 // token counts up to this take the small-M activation kernel
  double timeout_s = 2.0;
  CUtensorMap qw_map;                // INT4 weight codes [N_pad, K/2] bytes, box {32, 256}
  CUtensorMap swh_map;               // s_w 2^e_n f16 [K/G, N_pad], box {256, 64/G}: one GEMM stage's groups
  CUtensorMap Bh_map;                // B_hat [N, r_pad] f16, box {8, 128} (NVFP4 GEMM)
  CUtensorMap bhs_map;               // B_hat 2^e_n [N_pad, r_pad] f16, box {64, 256}, 128-byte swizzle
  CUtensorMap ucat_t_map, ucat3_map;
  CUtensorMap qw4_map;               // NVFP4 weight codes [N, K/2], box {128, 128}, 128-byte swizzle
  ActMaps act_cache[4];
  int act_next = 0;
  // Output maps of the INT4 GEMM's TMA-store epilogue: Y [M, N] (bf16 or float32), box 128 bytes
  // x 32 rows, 128-byte swizzle; the last few (Y, M, dtype) triples.
  struct YMap {
    const void* y = nullptr;
    int M = -1;
    bool f32 = false;
    int S = 0;  // > 0: the split-K GEMM's partial outputs [S, M, N] (float32, box 32 x 32 x 1)
    CUtensorMap map;
  };
  YMap y_cache[4];
  int y_next = 0;
};

// Workspace of M tokens.  INT4: packed OB4 codes [M, K/2], s_x bf16 [K/G, M_pad], p_hat f16
// [M, r_pad]; NVFP4: E2M1 codes [M, K/2], scale atoms, p_hat.  ab_off = phat_off (no region).
// Kernel (a)'s split of K over the CTAs of a cluster (C = 1, 2, 4 or 8) for `tiles` row tiles:
// as many CTAs as the SMs allow, each with an even number of 64-wide chunks.
inline int act_split(int K, int tiles, int sms) {
  const int chunks = K / kChunk;
  int C = 1;
  while (C < 8 && chunks % (2 * C) == 0 && tiles * 2 * C <= sms) C *= 2;
  if (C == 1 && chunks % 2 == 0 && tiles < sms) C = 2;
  return C;
}

// The INT4 GEMM's split of K over a cluster of CTAs per output tile (1, 2, 4 or 8) for layers
// whose 128 x kGemm16BN tiles would leave most SMs idle: CTAs on at most half the SMs (the
// clusters are then placed at once, beside the activation kernel's), each with at least two
// 64-wide K stages, and float32 partials of at most 8 MiB.
inline int gemm_split(int M, int N, int K, int sms) {
  // (layers of kPreExpandMinTiles row tiles or more take the float16-weight GEMM, unsplit, so that
  // the workspace-free call, which converts the weights tile by tile, gives the same sums)
  if ((M + kBM - 1) / kBM >= kPreExpandMinTiles) return 1;
  const int tiles = ((M + kBM - 1) / kBM) * ((N + kGemm16BN - 1) / kGemm16BN);
  const int nks = K / kChunk;
  int S = 1;
  while (S < 8 && tiles * 4 * S <= sms && nks >= 4 * S &&
         static_cast<size_t>(2 * S) * M * N * 4 <= (size_t{8} << 20))
    S *= 2;
  return S;
}

struct ActLayout {
  size_t codes_off, scales_off, ab_off, phat_off, bytes;
  size_t gsplit_off;  // INT4 with a split-K GEMM: float32 [S, M, N] partial outputs (0: none)
  size_t part_off;   // r_pad <= kMaxRank: float32 [C, M_pad, r_pad], kernel (a)'s partial projections
                     // of its C CTAs per row tile (C = act_split), exchanged through L2 (0: none)
  size_t resid_off;  // rotated handles with r > 0: float32 [M, K] remainder before the rotation
  size_t ytmp_off;   // NVFP4 with r_pad > kMaxRank: float32 [M, N] 4-bit part before the branch
  size_t w16_off;    // INT4 with >= kPreExpandMinTiles row tiles: float16 [N_pad, K + r_pad], the
                     // dequantized W_perp (s_w 2^e_n c) and B_hat 2^e_n of the call (0: none)
  int M_pad;
};
// `lean`: without the expanded-weight region (the GEMM then expands the weights tile by tile).
ActLayout act_layout(const Handle& h, int M, bool lean = false);

// Tensor-map encoder (driver entry point fetched through the runtime).
bool encode_2d(CUtensorMap* map, CUtensorMapDataType dt, const void* base, uint64_t inner, uint64_t outer,
               uint64_t row_stride_bytes, uint32_t box_inner, uint32_t box_outer, CUtensorMapSwizzle sw);
// The output map of Y [M, N] for the INT4 GEMM's TMA-store epilogue (cached per handle).
const CUtensorMap* get_y_map(Handle& h, const void* Y, int M, bool y_f32);
// The map of the split-K GEMM's float32 partial outputs [S, M, N], box 32 x 32 x 1, 128-byte swizzle.
const CUtensorMap* get_part_map(Handle& h, const void* part, int M, int S);
bool encode_3d(CUtensorMap* map, CUtensorMapDataType dt, const void* base, const uint64_t dims[3],
               const uint64_t strides_bytes[2], const uint32_t box[3],
               CUtensorMapSwizzle sw = CU_TENSOR_MAP_SWIZZLE_NONE);
const ActMaps* get_act_maps(Handle& h, const void* x, const void* ws, int M, bool lean = false);

uint64_t deadline_budget_ns(const Handle& h);

// The layer on a workspace of act_layout(h, M, lean) (api.cu).
qwam_status linear_impl(const void* X_bf16, int M, qwam_asp_handle h, void* Y, int y_dtype, void* act_ws,
                        struct CUstream_st* stream, bool lean);

// Launchers (return cudaSuccess or the launch error).
cudaError_t launch_pack(Handle& h, const __nv_bfloat16* W, const float* U, cudaStream_t s);
cudaError_t launch_pack_nvfp4(Handle& h, const __nv_bfloat16* W, const float* U, cudaStream_t s);
cudaError_t launch_pack_rotated(Handle& h, const __nv_bfloat16* W, const float* s, const float* U, cudaStream_t st);
// expand_w16: kernel (a) also writes the call's float16 weights into the workspace's expanded-weight
// region when it is the activation kernel of an INT4 layer whose GEMM takes them (act_layout(h, M)
// has the region); *expanded tells whether it did, and the GEMM launch then skips its own expansion
// (w16_ready).
cudaError_t launch_actquant(Handle& h, const ActMaps& am, const void* ws, int M, float* dump, cudaStream_t s,
                            bool expand_w16 = false, bool* expanded = nullptr);
cudaError_t launch_gemm(Handle& h, const ActMaps& am, const void* ws, int M, void* Y, bool y_f32, cudaStream_t s,
                        bool lean = false, bool w16_ready = false);
// The arguments of expand_w16 for the handle's weights and the expanded-weight region of layout L.
W16Args w16_args(const Handle& h, const ActLayout& L, const void* ws);
cudaError_t launch_gemm_nvfp4(Handle& h, const ActMaps& am, const void* ws, int M, void* Y, bool y_f32, cudaStream_t s);
cudaError_t launch_wait_probe(Handle& h, int timeout_us, cudaStream_t s);
cudaError_t launch_debug_quantize_lanes(const float* R, int M, int K, bool nvfp4, int G, uint8_t* codes,
                                        uint8_t* scales, int M_pad, cudaStream_t s);
cudaError_t launch_debug_quantize_rows(const float* R, int M, int K, bool nvfp4, int G, uint8_t* codes,
                                       void* scales, cudaStream_t s);
// The offline choice of what to protect (subspace.cu).
int subspace_width(int d, int r);
size_t subspace_workspace_bytes(int d, int r);
cudaError_t launch_smoothing(const float* xmax, const __nv_bfloat16* W, int K, int N, double alpha, float* s,
                             cudaStream_t st);
cudaError_t launch_rotated_gramian(const float* G, const float* gamma, int d, float* Gt, float* work, cudaStream_t st);
cudaError_t gramian_trace(const float* A, int d, double* host_out, cudaStream_t st);
cudaError_t action_subspace(const float* Gt, int d, int r, int iters, float* V_out, float* lambda, void* work,
                            cudaStream_t st);

}  // namespace qwam

struct qwam_asp_handle_s {
  qwam::Handle h;
};
