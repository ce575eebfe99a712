// api.cu -- the C ABI declared in include/qwam_asp.h: argument validation, the handle's device
// buffers, TMA tensor maps, and the launches.  No entry point on the run-time path allocates
// device memory.
#include <cudaTypedefs.h>

#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <new>
#include <vector>

#include "internal.h"
#include "ptx.cuh"

namespace qwam {
namespace {

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::once_flag g_encode_once;

bool ensure_encoder() {
  std::call_once(g_encode_once, [] {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  });
  return g_encode != nullptr;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

size_t up256(size_t b) { return (b + 255) & ~size_t(255); }

__global__ void wait_probe_kernel(int* err, uint64_t timeout_ns) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    const WaitCtl wc{&abort_flag, err, globaltimer_ns() + timeout_ns};
    mbar_wait(&bar, 0, wc);  // nothing arrives: the bound runs out and records kErrTimeout
    mbar_arrive(&bar);       // complete the phase so the barrier is left consistent
  }
}

}  // namespace

bool encode_2d(CUtensorMap* map, CUtensorMapDataType dt, const void* base, uint64_t inner, uint64_t outer,
               uint64_t row_stride_bytes, uint32_t box_inner, uint32_t box_outer, CUtensorMapSwizzle sw) {
  if (!ensure_encoder()) return false;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {row_stride_bytes};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = g_encode(map, dt, 2, const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        sw, CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

bool encode_3d(CUtensorMap* map, CUtensorMapDataType dt, const void* base, const uint64_t dims[3],
               const uint64_t strides_bytes[2], const uint32_t box[3], CUtensorMapSwizzle sw) {
  if (!ensure_encoder()) return false;
  cuuint64_t d[3] = {dims[0], dims[1], dims[2]};
  cuuint64_t st[2] = {strides_bytes[0], strides_bytes[1]};
  cuuint32_t b[3] = {box[0], box[1], box[2]};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = g_encode(map, dt, 3, const_cast<void*>(base), d, st, b, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, sw,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

const CUtensorMap* get_part_map(Handle& h, const void* part, int M, int S) {
  for (auto& c : h.y_cache)
    if (c.y == part && c.M == M && c.S == S) return &c.map;
  Handle::YMap& c = h.y_cache[h.y_next];
  c.y = nullptr;
  const uint64_t dims[3] = {static_cast<uint64_t>(h.N), static_cast<uint64_t>(M), static_cast<uint64_t>(S)};
  const uint64_t strides[2] = {static_cast<uint64_t>(h.N) * 4, static_cast<uint64_t>(M) * h.N * 4};
  const uint32_t box[3] = {32, 32, 1};
  if (!encode_3d(&c.map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, part, dims, strides, box, CU_TENSOR_MAP_SWIZZLE_128B))
    return nullptr;
  c.y = part;
  c.M = M;
  c.f32 = true;
  c.S = S;
  h.y_next = (h.y_next + 1) % 4;
  return &c.map;
}

const CUtensorMap* get_y_map(Handle& h, const void* Y, int M, bool y_f32) {
  for (auto& c : h.y_cache)
    if (c.y == Y && c.M == M && c.f32 == y_f32 && c.S == 0) return &c.map;
  Handle::YMap& c = h.y_cache[h.y_next];
  c.y = nullptr;
  const uint32_t es = y_f32 ? 4u : 2u;
  if (!encode_2d(&c.map, y_f32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, Y, h.N, M,
                 static_cast<uint64_t>(h.N) * es, 128 / es, 32, CU_TENSOR_MAP_SWIZZLE_128B))
    return nullptr;
  c.y = Y;
  c.M = M;
  c.f32 = y_f32;
  c.S = 0;
  h.y_next = (h.y_next + 1) % 4;
  return &c.map;
}

ActLayout act_layout(const Handle& h, int M, bool lean) {
  ActLayout L;
  L.M_pad = round_up(M > 0 ? M : 1, kBM);
  L.codes_off = 0;
  // kernel (a)'s exchange of partial projections (handles whose rank it takes on the tensor cores)
  auto add_part = [&](ActLayout& l) {
    l.part_off = 0;
    if (h.r_pad == 0 || h.r_pad > kMaxRank) return;
    l.part_off = l.bytes;
    const int C = act_split(h.K, l.M_pad / kBM, h.num_sms);
    l.bytes += up256(static_cast<size_t>(C) * l.M_pad * h.r_pad * 4);
  };
  if (h.fmt == kFmtNvfp4) {  // packed codes [M, K/2], scale atoms (M_pad rows), no epilogue constants
    L.scales_off = up256(static_cast<size_t>(M) * (h.K / 2));
    L.ab_off = L.scales_off + up256(static_cast<size_t>(L.M_pad) * (h.K / kFp4Block));
    L.phat_off = L.ab_off;
    L.bytes = L.phat_off + up256(static_cast<size_t>(M) * h.r_pad * 2 + 16);
    add_part(L);
    L.resid_off = 0;
    if (h.rot && h.r > 0) {
      L.resid_off = L.bytes;
      L.bytes += up256(static_cast<size_t>(M) * h.K * 4);
    }
    L.ytmp_off = 0;
    if (h.r_pad > kMaxRank) {  // the 4-bit part in float32, before the branch is added
      L.ytmp_off = L.bytes;
      L.bytes += up256(static_cast<size_t>(M) * h.N * 4);
    }
    L.w16_off = 0;
    L.gsplit_off = 0;
    return L;
  }
  L.scales_off = up256(static_cast<size_t>(M) * (h.K / 2));
  L.ab_off = L.scales_off + up256(static_cast<size_t>(h.K / h.G) * L.M_pad * 2);
  L.phat_off = L.ab_off;
  L.bytes = L.phat_off + up256(static_cast<size_t>(M) * h.r_pad * 2 + 16);
  add_part(L);
  L.resid_off = 0;
  if (h.rot && h.r > 0) {
    L.resid_off = L.bytes;
    L.bytes += up256(static_cast<size_t>(M) * h.K * 4);
  }
  L.ytmp_off = 0;
  L.w16_off = 0;
  L.gsplit_off = 0;
  if (!lean && L.M_pad / kBM >= kPreExpandMinTiles) {
    L.w16_off = L.bytes;
    L.bytes += up256(static_cast<size_t>(h.N_pad) * (h.K + h.r_pad) * 2);
  } else if (M > 0) {
    const int S = gemm_split(M, h.N, h.K, h.num_sms);
    if (S > 1) {
      L.gsplit_off = L.bytes;
      L.bytes += up256(static_cast<size_t>(S) * M * h.N * 4);
    }
  }
  return L;
}

uint64_t deadline_budget_ns(const Handle& h) { return static_cast<uint64_t>(h.timeout_s * 1e9); }

const ActMaps* get_act_maps(Handle& h, const void* x, const void* ws, int M, bool lean) {
  for (auto& c : h.act_cache)
    if (c.ws == ws && c.M == M && c.lean == lean && (x == nullptr || c.x == x)) return &c;
  ActMaps& c = h.act_cache[h.act_next];
  h.act_next = (h.act_next + 1) % 4;
  c.ws = nullptr;
  const ActLayout L = act_layout(h, M, lean);
  const uint8_t* base = static_cast<const uint8_t*>(ws);
  bool ok = true;
  if (x) {
    ok &= encode_2d(&c.x_map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, x, h.K, M, static_cast<uint64_t>(h.K) * 2, kChunk, kBM,
                    CU_TENSOR_MAP_SWIZZLE_128B);
  }
  if (h.fmt == kFmtNvfp4) {
    ok &= encode_2d(&c.qx4_map, CU_TENSOR_MAP_DATA_TYPE_UINT8, base + L.codes_off, h.K / 2, M, h.K / 2, kFp4KS / 2,
                    kBM, CU_TENSOR_MAP_SWIZZLE_128B);
  } else {
    ok &= encode_2d(&c.qa_map, CU_TENSOR_MAP_DATA_TYPE_UINT8, base + L.codes_off, h.K / 2, M, h.K / 2, 32, kBM,
                    CU_TENSOR_MAP_SWIZZLE_NONE);
    ok &= encode_2d(&c.sx_map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, base + L.scales_off, M, h.K / h.G,
                    static_cast<uint64_t>(L.M_pad) * 2, kBM, 64 / h.G, CU_TENSOR_MAP_SWIZZLE_NONE);
  }
  if (h.r_pad > 0) {
    ok &= encode_2d(&c.ph_map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, base + L.phat_off, h.r_pad, M,
                    static_cast<uint64_t>(h.r_pad) * 2, 8, kBM, CU_TENSOR_MAP_SWIZZLE_NONE);
    ok &= encode_2d(&c.ph64_map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, base + L.phat_off, h.r_pad, M,
                    static_cast<uint64_t>(h.r_pad) * 2, 64, kBM, CU_TENSOR_MAP_SWIZZLE_128B);
  }
  if (L.w16_off)
    ok &= encode_2d(&c.w16_map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, base + L.w16_off, h.K + h.r_pad, h.N_pad,
                    static_cast<uint64_t>(h.K + h.r_pad) * 2, 64, kGemm16BN, CU_TENSOR_MAP_SWIZZLE_128B);
  if (!ok) return nullptr;
  c.ws = ws;
  c.x = x;
  c.M = M;
  c.lean = lean;
  return &c;
}

cudaError_t launch_wait_probe(Handle& h, int timeout_us, cudaStream_t s) {
  wait_probe_kernel<<<1, 32, 0, s>>>(h.err, static_cast<uint64_t>(timeout_us) * 1000ull);
  return cudaGetLastError();
}

}  // namespace qwam

using qwam::Handle;

static qwam_status from_cuda_status(cudaError_t e) { return e == cudaSuccess ? QWAM_OK : QWAM_ERR_CUDA; }

// Frees everything a handle owns (any member may still be unset).
static void release_handle(qwam_asp_handle hs) {
  Handle& h = hs->h;
  if (h.block) cudaFree(h.block);
  if (h.bias) cudaFree(h.bias);
  if (h.done) cudaEventDestroy(h.done);
  if (h.err_stream) cudaStreamDestroy(h.err_stream);
  if (h.err_host) cudaFreeHost(h.err_host);
  delete hs;
}

// After a launch of the handle's kernels on `s`: remember it for qwam_asp_get_error.  Launches
// into a stream capture are not tracked (an event recorded there belongs to the graph).
static cudaError_t note_launch(Handle& h, cudaStream_t s) {
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  cudaError_t e = cudaStreamIsCapturing(s, &cs);
  if (e != cudaSuccess || cs != cudaStreamCaptureStatusNone) return e;
  e = cudaEventRecord(h.done, s);
  if (e == cudaSuccess) h.done_valid = true;
  return e;
}

// expand_w16 / expanded: see launch_actquant.
static qwam_status quantize_impl(const void* X, int M, qwam_asp_handle hs, void* ws, float* dump,
                                 struct CUstream_st* stream, bool expand_w16 = false, bool* expanded = nullptr) {
  if (!hs || M < 0) return QWAM_ERR_INVALID_ARG;
  if (M == 0) return QWAM_OK;
  if (!X || !ws || !qwam::aligned16(X) || !qwam::aligned16(ws)) return QWAM_ERR_INVALID_ARG;
  if (dump && !qwam::aligned16(dump)) return QWAM_ERR_INVALID_ARG;
  Handle& h = hs->h;
  const qwam::ActMaps* am = qwam::get_act_maps(h, X, ws, M);
  if (!am) return QWAM_ERR_CUDA;
  const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e = qwam::launch_actquant(h, *am, ws, M, dump, s, expand_w16, expanded);
  if (e == cudaSuccess) e = note_launch(h, s);
  return from_cuda_status(e);
}

static qwam_status gemm_impl(const void* act_ws, int M, qwam_asp_handle hs, void* Y, int y_dtype,
                             struct CUstream_st* stream, bool lean, bool w16_ready = false) {
  if (!hs || M < 0) return QWAM_ERR_INVALID_ARG;
  if (y_dtype != QWAM_Y_BF16 && y_dtype != QWAM_Y_FP32) return QWAM_ERR_INVALID_ARG;
  if (M == 0) return QWAM_OK;
  if (!act_ws || !Y || !qwam::aligned16(act_ws) || !qwam::aligned16(Y)) return QWAM_ERR_INVALID_ARG;
  Handle& h = hs->h;
  const qwam::ActMaps* am = qwam::get_act_maps(h, nullptr, act_ws, M, lean);
  if (!am) return QWAM_ERR_CUDA;
  const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e = h.fmt == qwam::kFmtNvfp4 ? qwam::launch_gemm_nvfp4(h, *am, act_ws, M, Y, y_dtype == QWAM_Y_FP32, s)
                                           : qwam::launch_gemm(h, *am, act_ws, M, Y, y_dtype == QWAM_Y_FP32, s, lean,
                                                               w16_ready);
  if (e == cudaSuccess) e = note_launch(h, s);
  return from_cuda_status(e);
}

namespace qwam {
// The layer on a workspace of act_layout(h, M, lean): qwam_asp_linear (lean = false) and the
// static-scratch entry (lean = true, no expanded-weight region).
qwam_status linear_impl(const void* X_bf16, int M, qwam_asp_handle h, void* Y, int y_dtype, void* act_ws,
                        struct CUstream_st* stream, bool lean) {
  if (!h || M < 0 || (y_dtype != QWAM_Y_BF16 && y_dtype != QWAM_Y_FP32)) return QWAM_ERR_INVALID_ARG;
  if (M > 0 && (!Y || !qwam::aligned16(Y))) return QWAM_ERR_INVALID_ARG;
  // Through this entry the activation kernel may also write the GEMM's float16 weights (the lean
  // layout has no region for them), which the GEMM then need not expand itself.
  bool expanded = false;
  qwam_status st = quantize_impl(X_bf16, M, h, act_ws, nullptr, stream, !lean, &expanded);
  if (st != QWAM_OK) return st;
  return gemm_impl(act_ws, M, h, Y, y_dtype, stream, lean, expanded);
}
}  // namespace qwam

extern "C" {

const char* qwam_status_string(qwam_status s) {
  switch (s) {
    case QWAM_OK: return "ok";
    case QWAM_ERR_INVALID_ARG: return "invalid argument";
    case QWAM_ERR_UNSUPPORTED: return "unsupported configuration";
    case QWAM_ERR_CUDA: return "CUDA error";
    case QWAM_ERR_OOM: return "out of device memory";
    case QWAM_ERR_TIMEOUT: return "device wait timed out";
    case QWAM_ERR_RANGE: return "value out of 16-bit range";
    case QWAM_ERR_TOO_LARGE: return "activation workspace larger than the static scratch (QWAM_STATIC_WS_BYTES)";
  }
  return "unknown status";
}

static qwam_status pack_impl(int fmt, const void* W_bf16, const float* U, const float* sm, bool rot, int K, int N,
                             int r, int group, struct CUstream_st* stream, qwam_asp_handle* out) {
  if (!out) return QWAM_ERR_INVALID_ARG;
  *out = nullptr;
  if (!W_bf16 || !qwam::aligned16(W_bf16)) return QWAM_ERR_INVALID_ARG;
  if (K <= 0 || K % 64 != 0 || N <= 0 || N % 8 != 0) return QWAM_ERR_INVALID_ARG;
  if (fmt == qwam::kFmtNvfp4 && K % qwam::kFp4KS != 0) return QWAM_ERR_INVALID_ARG;
  if (fmt == qwam::kFmtInt4 && group != 32 && group != 64) return QWAM_ERR_INVALID_ARG;
  if (r < 0 || r > K) return QWAM_ERR_INVALID_ARG;
  if (r > 0 && (!U || !qwam::aligned16(U))) return QWAM_ERR_INVALID_ARG;
  // Ranks above kMaxRank take the general-rank activation path (one warp per 256 channels of a
  // row); the rotated layers keep the tensor-core path only.
  if (r > qwam::kMaxRank && (rot || K % 256 != 0)) return QWAM_ERR_UNSUPPORTED;
  // the run-time rotation works on sub-blocks of 256 channels (one warp, eight per lane)
  if (rot && (K % 256 != 0 || (sm && !qwam::aligned16(sm)))) return QWAM_ERR_INVALID_ARG;
  if (!qwam::ensure_encoder()) return QWAM_ERR_CUDA;

  auto* hs = new (std::nothrow) qwam_asp_handle_s();
  if (!hs) return QWAM_ERR_OOM;
  Handle& h = hs->h;
  h.fmt = fmt;
  h.K = K;
  h.N = N;
  h.r = r;
  h.G = group;
  h.r_pad = r == 0 ? 0 : qwam::round_up(r, 16);
  h.N_pad = qwam::round_up(N, fmt == qwam::kFmtNvfp4 ? qwam::kGemmBN : qwam::kGemm16BN);
  h.ku3 = h.r_pad == 0 ? 0 : qwam::round_up(3 * h.r_pad, 64);
  h.rot = rot;
  if (rot) {
    h.hb = 1;
    while (K % (2 * h.hb) == 0 && 2 * h.hb <= 1024) h.hb *= 2;
  }
  cudaGetDevice(&h.device);
  cudaDeviceGetAttribute(&h.num_sms, cudaDevAttrMultiProcessorCount, h.device);

  const bool nv = fmt == qwam::kFmtNvfp4;
  const size_t b_qw = qwam::up256(static_cast<size_t>(h.N_pad) * (K / 2));
  // INT4: bfloat16 scales, then the GEMM's float16 copies (scaled per column) and column factors;
  // NVFP4: E4M3 scale atoms (N_pad rows)
  const size_t b_sw = nv ? qwam::up256(static_cast<size_t>(h.N_pad) * (K / qwam::kFp4Block))
                         : qwam::up256(static_cast<size_t>(K / group) * h.N_pad * 2);
  const size_t b_s32 = nv ? 0
                          : qwam::up256(static_cast<size_t>(K / group) * h.N_pad * 2) +
                                qwam::up256(static_cast<size_t>(h.N_pad) * h.r_pad * 2) +
                                qwam::up256(static_cast<size_t>(h.N_pad) * 4);
  const size_t b_bh = qwam::up256(static_cast<size_t>(h.N_pad) * h.r_pad * 2);
  // the bf16 split bases feed kernel (a)'s tensor-core path only (r_pad <= kMaxRank)
  const bool tc_bases = h.r_pad > 0 && h.r_pad <= qwam::kMaxRank;
  const size_t b_ut = tc_bases ? qwam::up256(static_cast<size_t>(2 * h.r_pad) * K * 2) : 0;
  const size_t b_u3 = tc_bases ? qwam::up256(static_cast<size_t>(K) * h.ku3 * 2) : 0;
  const size_t b_is = rot ? qwam::up256(static_cast<size_t>(K) * 4) : 0;
  const size_t b_u32 = qwam::up256(static_cast<size_t>(K) * h.r_pad * 4);
  const size_t total = b_qw + b_sw + b_s32 + b_bh + b_ut + b_u3 + b_is + 2 * b_u32 + 256;
  if (cudaMalloc(&h.block, total) != cudaSuccess) {
    cudaGetLastError();
    delete hs;
    return QWAM_ERR_OOM;
  }
  uint8_t* p = static_cast<uint8_t*>(h.block);
  h.qw = p;
  if (nv) {
    h.sfw = p + b_qw;
  } else {
    h.sw = reinterpret_cast<__nv_bfloat16*>(p + b_qw);
    uint8_t* c = p + b_qw + b_sw;
    h.swh = reinterpret_cast<__half*>(c);
    c += qwam::up256(static_cast<size_t>(K / group) * h.N_pad * 2);
    h.Bhs = reinterpret_cast<__half*>(c);
    c += qwam::up256(static_cast<size_t>(h.N_pad) * h.r_pad * 2);
    h.fcol = reinterpret_cast<float*>(c);
  }
  uint8_t* q = p + b_qw + b_sw + b_s32;
  h.Bh = reinterpret_cast<__half*>(q);
  if (tc_bases) {
    h.ucat_t = reinterpret_cast<__nv_bfloat16*>(q + b_bh);
    h.ucat3 = reinterpret_cast<__nv_bfloat16*>(q + b_bh + b_ut);
  }
  if (rot) h.inv_s = reinterpret_cast<float*>(q + b_bh + b_ut + b_u3);
  if (h.r_pad > 0) {
    // without rotation both bases are U: one copy, so the small-M kernel's reconstruction reads
    // what its projection just brought into L1
    h.up32 = reinterpret_cast<float*>(q + b_bh + b_ut + b_u3 + b_is);
    h.ur32 = rot ? reinterpret_cast<float*>(q + b_bh + b_ut + b_u3 + b_is + b_u32) : h.up32;
  }
  h.err = reinterpret_cast<int*>(q + b_bh + b_ut + b_u3 + b_is + 2 * b_u32);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);

  bool ok = true;
  if (nv) {
    ok &= qwam::encode_2d(&h.qw4_map, CU_TENSOR_MAP_DATA_TYPE_UINT8, h.qw, K / 2, N, K / 2, qwam::kFp4KS / 2,
                          qwam::kGemmBN, CU_TENSOR_MAP_SWIZZLE_128B);
  } else {
    ok &= qwam::encode_2d(&h.qw_map, CU_TENSOR_MAP_DATA_TYPE_UINT8, h.qw, K / 2, h.N_pad, K / 2, 32,
                          qwam::kGemm16BN, CU_TENSOR_MAP_SWIZZLE_NONE);
    ok &= qwam::encode_2d(&h.swh_map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, h.swh, h.N_pad, K / group,
                          static_cast<uint64_t>(h.N_pad) * 2, qwam::kGemm16BN, 64 / group,
                          CU_TENSOR_MAP_SWIZZLE_NONE);
    if (h.r_pad > 0)
      ok &= qwam::encode_2d(&h.bhs_map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, h.Bhs, h.r_pad, h.N_pad,
                            static_cast<uint64_t>(h.r_pad) * 2, 64, qwam::kGemm16BN, CU_TENSOR_MAP_SWIZZLE_128B);
  }
  if (h.r_pad > 0) {
    ok &= qwam::encode_2d(&h.Bh_map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, h.Bh, h.r_pad, N,
                          static_cast<uint64_t>(h.r_pad) * 2, 8, qwam::kBM, CU_TENSOR_MAP_SWIZZLE_NONE);
  }
  if (tc_bases) {
    ok &= qwam::encode_2d(&h.ucat_t_map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, h.ucat_t, K, 2 * h.r_pad,
                          static_cast<uint64_t>(K) * 2, qwam::kChunk, 2 * h.r_pad, CU_TENSOR_MAP_SWIZZLE_128B);
    ok &= qwam::encode_2d(&h.ucat3_map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, h.ucat3, h.ku3, K,
                          static_cast<uint64_t>(h.ku3) * 2, 64, 64, CU_TENSOR_MAP_SWIZZLE_128B);
  }
  if (!ok) {
    release_handle(hs);
    return QWAM_ERR_CUDA;
  }
  cudaError_t e = cudaMemsetAsync(h.block, 0, total, s);
  if (e == cudaSuccess) {
    const auto* W = static_cast<const __nv_bfloat16*>(W_bf16);
    if (rot)
      e = qwam::launch_pack_rotated(h, W, sm, r > 0 ? U : nullptr, s);
    else
      e = nv ? qwam::launch_pack_nvfp4(h, W, r > 0 ? U : nullptr, s) : qwam::launch_pack(h, W, r > 0 ? U : nullptr, s);
  }
  int herr = 0;
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);  // `s` may be a non-blocking stream
  if (e == cudaSuccess) e = cudaMemcpy(&herr, h.err, sizeof(int), cudaMemcpyDeviceToHost);
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&h.done, cudaEventDisableTiming);
  if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&h.err_stream, cudaStreamNonBlocking);
  if (e == cudaSuccess) e = cudaMallocHost(&h.err_host, sizeof(int));
  if (e != cudaSuccess || herr != 0) {
    cudaGetLastError();
    release_handle(hs);
    return e != cudaSuccess ? QWAM_ERR_CUDA : QWAM_ERR_RANGE;
  }
  *out = hs;
  return QWAM_OK;
}

qwam_status qwam_asp_pack_weights(const void* W_bf16, const float* U, int K, int N, int r, int group,
                                  struct CUstream_st* stream, qwam_asp_handle* out) {
  return pack_impl(qwam::kFmtInt4, W_bf16, U, nullptr, false, K, N, r, group, stream, out);
}

qwam_status qwam_asp_pack_weights_rotated(const void* W_bf16, const float* s, const float* U, int K, int N, int r,
                                          int group, struct CUstream_st* stream, qwam_asp_handle* out) {
  return pack_impl(qwam::kFmtInt4, W_bf16, U, s, true, K, N, r, group, stream, out);
}

qwam_status qwam_asp_pack_weights_nvfp4_rotated(const void* W_bf16, const float* s, const float* U, int K, int N,
                                                int r, struct CUstream_st* stream, qwam_asp_handle* out) {
  return pack_impl(qwam::kFmtNvfp4, W_bf16, U, s, true, K, N, r, qwam::kFp4Block, stream, out);
}

qwam_status qwam_asp_rotation(qwam_asp_handle hs, int* hadamard_block) {
  if (!hs || !hadamard_block) return QWAM_ERR_INVALID_ARG;
  *hadamard_block = hs->h.rot ? hs->h.hb : 0;
  return QWAM_OK;
}

qwam_status qwam_asp_pack_weights_nvfp4(const void* W_bf16, const float* U, int K, int N, int r,
                                        struct CUstream_st* stream, qwam_asp_handle* out) {
  return pack_impl(qwam::kFmtNvfp4, W_bf16, U, nullptr, false, K, N, r, qwam::kFp4Block, stream, out);
}

qwam_status qwam_asp_format(qwam_asp_handle hs, int* format) {
  if (!hs || !format) return QWAM_ERR_INVALID_ARG;
  *format = hs->h.fmt == qwam::kFmtNvfp4 ? QWAM_FMT_NVFP4 : QWAM_FMT_INT4;
  return QWAM_OK;
}

qwam_status qwam_asp_act_workspace_bytes(qwam_asp_handle hs, int M, size_t* bytes) {
  if (!hs || !bytes || M < 0) return QWAM_ERR_INVALID_ARG;
  *bytes = qwam::act_layout(hs->h, M).bytes;
  return QWAM_OK;
}

qwam_status qwam_asp_act_layout(qwam_asp_handle hs, int M, size_t* codes_off, size_t* scales_off,
                                size_t* ab_off, size_t* phat_off, int* M_pad, int* r_pad) {
  if (!hs || M < 0) return QWAM_ERR_INVALID_ARG;
  const qwam::ActLayout L = qwam::act_layout(hs->h, M);
  if (codes_off) *codes_off = L.codes_off;
  if (scales_off) *scales_off = L.scales_off;
  if (ab_off) *ab_off = L.ab_off;
  if (phat_off) *phat_off = L.phat_off;
  if (M_pad) *M_pad = L.M_pad;
  if (r_pad) *r_pad = hs->h.r_pad;
  return QWAM_OK;
}

qwam_status qwam_asp_quantize_act(const void* X_bf16, int M, qwam_asp_handle h, void* act_ws,
                                  struct CUstream_st* stream) {
  return quantize_impl(X_bf16, M, h, act_ws, nullptr, stream);
}

qwam_status qwam_asp_debug_residual(const void* X_bf16, int M, qwam_asp_handle h, void* act_ws, float* R,
                                    struct CUstream_st* stream) {
  if (!R) return QWAM_ERR_INVALID_ARG;
  return quantize_impl(X_bf16, M, h, act_ws, R, stream);
}

qwam_status qwam_asp_debug_quantize_rows(const float* R, int M, int K, int fmt, int group, void* codes,
                                         void* scales, struct CUstream_st* stream) {
  if (M < 0 || K <= 0 || K % qwam::kChunk != 0) return QWAM_ERR_INVALID_ARG;
  if (fmt != QWAM_FMT_INT4 && fmt != QWAM_FMT_NVFP4) return QWAM_ERR_INVALID_ARG;
  if (fmt == QWAM_FMT_INT4 && group != 32 && group != 64) return QWAM_ERR_INVALID_ARG;
  if (M == 0) return QWAM_OK;
  if (!R || !codes || !scales || !qwam::aligned16(R) || !qwam::aligned16(codes)) return QWAM_ERR_INVALID_ARG;
  if (fmt == QWAM_FMT_INT4 && reinterpret_cast<uintptr_t>(scales) % 2 != 0) return QWAM_ERR_INVALID_ARG;
  return from_cuda_status(qwam::launch_debug_quantize_rows(R, M, K, fmt == QWAM_FMT_NVFP4, group,
                                                           static_cast<uint8_t*>(codes), scales,
                                                           reinterpret_cast<cudaStream_t>(stream)));
}

qwam_status qwam_asp_debug_quantize_lanes(const float* R, int M, int K, int fmt, int group, void* codes, void* scales,
                                          struct CUstream_st* stream) {
  if (M < 0 || K <= 0 || K % 256 != 0) return QWAM_ERR_INVALID_ARG;
  if (fmt != QWAM_FMT_INT4 && fmt != QWAM_FMT_NVFP4) return QWAM_ERR_INVALID_ARG;
  if (fmt == QWAM_FMT_INT4 && group != 32 && group != 64) return QWAM_ERR_INVALID_ARG;
  if (M == 0) return QWAM_OK;
  if (!R || !codes || !scales || !qwam::aligned16(R) || !qwam::aligned16(codes)) return QWAM_ERR_INVALID_ARG;
  if (fmt == QWAM_FMT_INT4 && reinterpret_cast<uintptr_t>(scales) % 2 != 0) return QWAM_ERR_INVALID_ARG;
  const int M_pad = qwam::round_up(M, qwam::kBM);
  return from_cuda_status(qwam::launch_debug_quantize_lanes(
      R, M, K, fmt == QWAM_FMT_NVFP4, fmt == QWAM_FMT_NVFP4 ? qwam::kFp4Block : group, static_cast<uint8_t*>(codes),
      static_cast<uint8_t*>(scales), M_pad, reinterpret_cast<cudaStream_t>(stream)));
}

qwam_status qwam_asp_smoothing_factors(const float* xmax, const void* W_bf16, int K, int N, double alpha, float* s,
                                       struct CUstream_st* stream) {
  if (K <= 0 || N <= 0 || !xmax || !W_bf16 || !s || !(alpha >= 0.0 && alpha <= 1.0)) return QWAM_ERR_INVALID_ARG;
  return from_cuda_status(qwam::launch_smoothing(xmax, static_cast<const __nv_bfloat16*>(W_bf16), K, N, alpha, s,
                                                 reinterpret_cast<cudaStream_t>(stream)));
}

qwam_status qwam_asp_rotated_gramian(const float* G, const float* gamma, int d, float* Gt, float* work,
                                     struct CUstream_st* stream) {
  if (d <= 0 || d > 32768 || !G || !Gt || !work || G == Gt || G == work || Gt == work) return QWAM_ERR_INVALID_ARG;
  return from_cuda_status(qwam::launch_rotated_gramian(G, gamma, d, Gt, work, reinterpret_cast<cudaStream_t>(stream)));
}

qwam_status qwam_asp_gramian_trace(const float* A, int d, double* trace, struct CUstream_st* stream) {
  if (d <= 0 || !A || !trace) return QWAM_ERR_INVALID_ARG;
  return from_cuda_status(qwam::gramian_trace(A, d, trace, reinterpret_cast<cudaStream_t>(stream)));
}

qwam_status qwam_asp_subspace_workspace_bytes(int d, int r, size_t* bytes) {
  if (d <= 0 || r <= 0 || r > d || r > qwam::subspace_width(d, r) || !bytes) return QWAM_ERR_INVALID_ARG;
  *bytes = qwam::subspace_workspace_bytes(d, r);
  return QWAM_OK;
}

qwam_status qwam_asp_action_subspace(const float* Gt, int d, int r, int iters, float* V, float* lambda, void* work,
                                     struct CUstream_st* stream) {
  if (d <= 0 || r <= 0 || r > d || r > qwam::subspace_width(d, r) || iters < 0 || !Gt || !V || !lambda || !work ||
      !qwam::aligned16(work))
    return QWAM_ERR_INVALID_ARG;
  return from_cuda_status(qwam::action_subspace(Gt, d, r, iters, V, lambda, work, reinterpret_cast<cudaStream_t>(stream)));
}

qwam_status qwam_asp_select_experts(const double* mass, const double* cost, int n, double budget, int* chosen,
                                    int* n_chosen) {
  if (n < 0 || (n > 0 && (!mass || !cost || !chosen)) || !n_chosen) return QWAM_ERR_INVALID_ARG;
  for (int i = 0; i < n; ++i)
    if (!(cost[i] > 0.0) || !(mass[i] >= 0.0)) return QWAM_ERR_INVALID_ARG;
  std::vector<int> order(n);
  for (int i = 0; i < n; ++i) order[i] = i;
  // decreasing action mass per added 16-bit value; equal ratios keep the lower index first
  std::stable_sort(order.begin(), order.end(),
                   [&](int a, int b) { return mass[a] / cost[a] > mass[b] / cost[b]; });
  double used = 0.0;
  int k = 0;
  for (int i : order)
    if (used + cost[i] <= budget) {
      chosen[k++] = i;
      used += cost[i];
    }
  *n_chosen = k;
  return QWAM_OK;
}

qwam_status qwam_asp_gemm(const void* act_ws, int M, qwam_asp_handle hs, void* Y, int y_dtype,
                          struct CUstream_st* stream) {
  return gemm_impl(act_ws, M, hs, Y, y_dtype, stream, false);
}

qwam_status qwam_asp_linear(const void* X_bf16, int M, qwam_asp_handle h, void* Y, int y_dtype, void* act_ws,
                            struct CUstream_st* stream) {
  return qwam::linear_impl(X_bf16, M, h, Y, y_dtype, act_ws, stream, false);
}

qwam_status qwam_asp_get_error(qwam_asp_handle hs) {
  if (!hs) return QWAM_ERR_INVALID_ARG;
  Handle& h = hs->h;
  // read and clear the word on the handle's own stream, after the handle's last tracked launch
  cudaError_t e = h.done_valid ? cudaStreamWaitEvent(h.err_stream, h.done, 0) : cudaSuccess;
  if (e == cudaSuccess) e = cudaMemcpyAsync(h.err_host, h.err, sizeof(int), cudaMemcpyDeviceToHost, h.err_stream);
  if (e == cudaSuccess) e = cudaMemsetAsync(h.err, 0, sizeof(int), h.err_stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(h.err_stream);
  if (e != cudaSuccess) return QWAM_ERR_CUDA;
  const int v = *h.err_host;
  if (v & qwam::kErrTimeout) return QWAM_ERR_TIMEOUT;
  if (v & qwam::kErrRange) return QWAM_ERR_RANGE;
  return QWAM_OK;
}

qwam_status qwam_asp_shape(qwam_asp_handle hs, int* K, int* N, int* r, int* group, int* r_pad) {
  if (!hs) return QWAM_ERR_INVALID_ARG;
  if (K) *K = hs->h.K;
  if (N) *N = hs->h.N;
  if (r) *r = hs->h.r;
  if (group) *group = hs->h.G;
  if (r_pad) *r_pad = hs->h.r_pad;
  return QWAM_OK;
}

qwam_status qwam_asp_export(qwam_asp_handle hs, void* qw, void* sw, void* Bh, void* Uhl) {
  if (!hs) return QWAM_ERR_INVALID_ARG;
  Handle& h = hs->h;
  if (h.fmt != qwam::kFmtInt4) return QWAM_ERR_INVALID_ARG;
  if (cudaDeviceSynchronize() != cudaSuccess) return QWAM_ERR_CUDA;
  cudaError_t e = cudaSuccess;
  if (qw) {
    // device rows are OB4 words (word j: k = 8j..8j+7, offset binary, see ob4_word); export
    // two's-complement nibbles, low nibble = even k
    std::vector<uint32_t> t(static_cast<size_t>(h.N) * (h.K / 8));
    e = cudaMemcpy(t.data(), h.qw, t.size() * 4, cudaMemcpyDeviceToHost);
    uint8_t* o = static_cast<uint8_t*>(qw);
    for (size_t wd = 0; e == cudaSuccess && wd < t.size(); ++wd)
      for (int q = 0; q < 4; ++q)
        o[4 * wd + q] = static_cast<uint8_t>((qwam::ob4_code(t[wd], 2 * q) & 0xF) |
                                             ((qwam::ob4_code(t[wd], 2 * q + 1) & 0xF) << 4));
  }
  if (e == cudaSuccess && sw)
    e = cudaMemcpy2D(sw, static_cast<size_t>(h.N) * 2, h.sw, static_cast<size_t>(h.N_pad) * 2,
                     static_cast<size_t>(h.N) * 2, h.K / h.G, cudaMemcpyDeviceToHost);
  if (e == cudaSuccess && Bh && h.r_pad > 0)
    e = cudaMemcpy(Bh, h.Bh, static_cast<size_t>(h.N) * h.r_pad * 2, cudaMemcpyDeviceToHost);
  if (e == cudaSuccess && Uhl && h.r_pad > 0) {
    uint16_t* o = static_cast<uint16_t*>(Uhl);
    if (h.ucat_t) {
      std::vector<uint16_t> t(static_cast<size_t>(2 * h.r_pad) * h.K);
      e = cudaMemcpy(t.data(), h.ucat_t, t.size() * 2, cudaMemcpyDeviceToHost);
      for (int part = 0; part < 2 && e == cudaSuccess; ++part)
        for (int k = 0; k < h.K; ++k)
          for (int j = 0; j < h.r_pad; ++j)
            o[(static_cast<size_t>(part) * h.K + k) * h.r_pad + j] =
                t[static_cast<size_t>(part * h.r_pad + j) * h.K + k];
    } else {
      // the general-rank path keeps no bf16 split: none to export
      std::fill(o, o + static_cast<size_t>(2 * h.K) * h.r_pad, static_cast<uint16_t>(0));
    }
  }
  if (e != cudaSuccess) cudaGetLastError();  // leave no error behind for the next call
  return from_cuda_status(e);
}

qwam_status qwam_asp_export_nvfp4(qwam_asp_handle hs, void* qw, void* sfw, float* sg, void* Bh) {
  if (!hs) return QWAM_ERR_INVALID_ARG;
  Handle& h = hs->h;
  if (h.fmt != qwam::kFmtNvfp4) return QWAM_ERR_INVALID_ARG;
  if (cudaDeviceSynchronize() != cudaSuccess) return QWAM_ERR_CUDA;
  cudaError_t e = cudaSuccess;
  if (qw) e = cudaMemcpy(qw, h.qw, static_cast<size_t>(h.N) * (h.K / 2), cudaMemcpyDeviceToHost);
  if (e == cudaSuccess && sfw) {
    // atoms -> row-major [N, K/16]
    const int nb = h.K / qwam::kFp4Block;
    std::vector<uint8_t> t(static_cast<size_t>(h.N_pad) * nb);
    e = cudaMemcpy(t.data(), h.sfw, t.size(), cudaMemcpyDeviceToHost);
    uint8_t* o = static_cast<uint8_t*>(sfw);
    for (int n = 0; e == cudaSuccess && n < h.N; ++n)
      for (int b = 0; b < nb; ++b) {
        const int nr = n % 128;
        o[static_cast<size_t>(n) * nb + b] =
            t[(static_cast<size_t>(n / 128) * (h.K / 64) + b / 4) * qwam::kSfAtom + (nr % 32) * 16 + (nr / 32) * 4 + b % 4];
      }
  }
  if (e == cudaSuccess && sg) *sg = h.sg;
  if (e == cudaSuccess && Bh && h.r_pad > 0)
    e = cudaMemcpy(Bh, h.Bh, static_cast<size_t>(h.N) * h.r_pad * 2, cudaMemcpyDeviceToHost);
  return from_cuda_status(e);
}

qwam_status qwam_asp_destroy(qwam_asp_handle hs) {
  if (!hs) return QWAM_ERR_INVALID_ARG;
  const cudaError_t e = cudaDeviceSynchronize();
  release_handle(hs);
  return from_cuda_status(e);
}

qwam_status qwam_asp_set_bias(qwam_asp_handle hs, const float* bias, struct CUstream_st* stream) {
  if (!hs) return QWAM_ERR_INVALID_ARG;
  Handle& h = hs->h;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (!bias) {
    if (h.bias) {
      if (cudaStreamSynchronize(s) != cudaSuccess) return QWAM_ERR_CUDA;
      cudaFree(h.bias);
      h.bias = nullptr;
    }
    return QWAM_OK;
  }
  if (!qwam::aligned16(bias)) return QWAM_ERR_INVALID_ARG;
  if (!h.bias) {
    // 16-byte aligned rows of 8 floats: the epilogues read N rounded up to 8
    if (cudaMalloc(&h.bias, sizeof(float) * static_cast<size_t>(h.N_pad)) != cudaSuccess) {
      cudaGetLastError();
      h.bias = nullptr;
      return QWAM_ERR_OOM;
    }
    if (cudaMemsetAsync(h.bias, 0, sizeof(float) * static_cast<size_t>(h.N_pad), s) != cudaSuccess)
      return QWAM_ERR_CUDA;
  }
  cudaError_t e = cudaMemcpyAsync(h.bias, bias, sizeof(float) * static_cast<size_t>(h.N), cudaMemcpyDeviceToDevice, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  return from_cuda_status(e);
}

qwam_status qwam_asp_set_small_m(qwam_asp_handle hs, int max_rows) {
  if (!hs || max_rows < 0) return QWAM_ERR_INVALID_ARG;
  hs->h.small_m = max_rows;
  return QWAM_OK;
}

qwam_status qwam_asp_set_timeout(qwam_asp_handle hs, double seconds) {
  if (!hs || !(seconds > 0.0) || seconds > 3600.0) return QWAM_ERR_INVALID_ARG;
  hs->h.timeout_s = seconds;
  return QWAM_OK;
}

qwam_status qwam_asp_debug_wait_timeout(qwam_asp_handle hs, int timeout_us, struct CUstream_st* stream) {
  if (!hs || timeout_us <= 0 || timeout_us > 10000000) return QWAM_ERR_INVALID_ARG;
  const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e = qwam::launch_wait_probe(hs->h, timeout_us, s);
  if (e == cudaSuccess) e = note_launch(hs->h, s);
  return from_cuda_status(e);
}

}  // extern "C"
