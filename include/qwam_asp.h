/*
 * qwam_asp.h -- C ABI of the GB300 (sm_103a) implementation of the Action-Subspace Protection
 * (ASP) linear layer of Q-WAM (arxiv 2609.33269).
 *
 * The layer (Sec. 4.2, Eq. (xsplit) and Eq. (asp)), in the row-major notation used here
 * (X [M,K] = one token per row, W [K,N], U [K,r] = the paper's V with orthonormal columns):
 *
 *     p      = X U                       (protected coordinates, kept in 16 bits)
 *     X_perp = X - p U^T                 (remainder, orthogonal to span(U))
 *     W_perp = W - U (U^T W)             (deflated weight, Sec. 4.2 "Splitting the layer")
 *     Y      = p_hat B_hat  +  Q4(X_perp) Q4(W_perp)
 *
 * with B_hat = RN_f16(U^T W), p_hat = RN_f16(p), and Q4 the symmetric group quantizer of
 * Eq. (quant) (Sec. 3) with b = 4: scale s = absmax / 7 per group of `group` consecutive input
 * channels (App. B.1), codes = nearest integer to x / s (exact quotient, ties to even), so codes
 * lie in [-7, 7].  Both scales are bfloat16, s = RN_bf16(absmax / 7) rounded once from the exact
 * quotient (Table 3: 4.50 bits per weight at group 32 implies a 16-bit weight scale; the paper
 * leaves the activation scale's format open).  r = 0 gives plain per-group W4A4 (experts that
 * ASP does not select, Sec. 4.3).
 *
 * Conventions for every entry point:
 *   - Pointers marked "device" are CUDA device pointers on the current device; "host" pointers
 *     are ordinary host memory.  All device pointers must be 16-byte aligned.
 *   - The caller owns every buffer it passes in (X, Y, W, U, act_ws).  The handle owns its packed
 *     weights until qwam_asp_destroy.  No entry point retains a caller pointer after it returns.
 *   - `stream` is a cudaStream_t (NULL = the legacy default stream).
 *   - Arguments are validated on the host before anything is launched; an invalid argument
 *     returns QWAM_ERR_INVALID_ARG and launches nothing.  A failed CUDA call returns
 *     QWAM_ERR_CUDA.  Run-time entry points are asynchronous and allocate no device memory.
 *   - Device-side waits are bounded.  A wait that runs out records QWAM_ERR_TIMEOUT in the
 *     handle's error word (read and cleared by qwam_asp_get_error) and the kernel returns.
 *   - Inputs must be finite.  A handle may be used from one host thread at a time.
 */
#ifndef QWAM_ASP_H
#define QWAM_ASP_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

struct CUstream_st; /* cudaStream_t == struct CUstream_st* */

typedef struct qwam_asp_handle_s* qwam_asp_handle;

typedef enum {
  QWAM_OK = 0,
  QWAM_ERR_INVALID_ARG = -1,
  QWAM_ERR_UNSUPPORTED = -2, /* valid request that this build does not implement (e.g. r > 64 when rotated) */
  QWAM_ERR_CUDA = -3,
  QWAM_ERR_OOM = -4,
  QWAM_ERR_TIMEOUT = -5,     /* a bounded device wait gave up */
  QWAM_ERR_RANGE = -6,       /* a scale or branch value does not fit its 16-bit format */
  QWAM_ERR_TOO_LARGE = -7    /* the activation workspace would exceed QWAM_STATIC_WS_BYTES */
} qwam_status;

enum { QWAM_Y_BF16 = 0, QWAM_Y_FP32 = 1 };

/* Offline packing (Sec. 4.2 Eq. (asp); the W_perp derivation; Eq. (quant) on the weight).
 *   W_bf16 : device, bf16 [K, N] row-major (the paper's W~ in its transformed coordinates)
 *   U      : device, float32 [K, r] row-major, orthonormal columns; may be NULL iff r == 0
 *   K      : input dimension, K % 64 == 0;   N : output dimension, N % 8 == 0
 *   r      : protected rank, 0 <= r <= K.  Ranks up to 64 run kernel (a) on the tensor cores;
 *            larger ones take a general-rank activation path on the CUDA cores (cost K r per
 *            token, for correctness rather than speed), which needs K % 256 == 0 (otherwise
 *            QWAM_ERR_UNSUPPORTED).  Rotated handles are limited to r <= 64.
 *   group  : quantization group along K, 32 or 64
 *   out    : receives the new handle
 * Computes, in float64 on the device: B_f = U^T W, W_perp = W - U B_f, per (output channel,
 * group) s_w = RN_bf16(absmax / 7) and the codes of W_perp / s_w, B_hat = RN_f16(B_f), the
 * bf16 hi/lo split of U used by the activation kernel, and the GEMM's float16 copies of s_w and
 * B_hat scaled by a power of two per output column.  Synchronizes `stream` before returning.
 * Returns QWAM_ERR_RANGE if a weight scale or a branch value overflows its 16-bit format. */
qwam_status qwam_asp_pack_weights(const void* W_bf16, const float* U, int K, int N, int r, int group,
                                  struct CUstream_st* stream, qwam_asp_handle* out);

/* Bytes of the caller-owned activation workspace needed for M tokens.  For INT4 layers of 512 or
 * more tokens it includes a float16 copy of the layer's weights, N_pad (K + r_pad) 2 bytes (N_pad =
 * N rounded up to 256), which is filled once per call and read from L2 for every row tile: by
 * kernel (a) inside qwam_asp_linear when r > 0, otherwise by qwam_asp_gemm before its GEMM.  For 0 < r_pad <= 64 it also includes kernel (a)'s scratch for the partial projections of
 * the C CTAs that share a row tile's K (float32, C M_pad r_pad 4 bytes, C <= 8).  Layers of fewer
 * tokens whose 128 x 256 output tiles leave most SMs idle add the split-K GEMM's float32 partial
 * outputs (S M N 4 bytes, S <= 8, at most 8 MiB). */
qwam_status qwam_asp_act_workspace_bytes(qwam_asp_handle h, int M, size_t* bytes);

/* Layout of the activation workspace for M tokens (byte offsets from its start):
 *   codes  : uint8 [M, K/2], the activation codes c in [-7, 7] packed at four bits as OB4 words:
 *            the little-endian 32-bit word j of a row holds k = 8j .. 8j+7 as offset-binary
 *            nibbles c + 8, code 8j + 2p in bits 4p .. 4p+3 and code 8j + 2p + 1 in bits
 *            16 + 4p .. 16 + 4p + 3 (p = 0..3).  (The GEMM turns pair p into two float16 values
 *            with one shift, one and-or under the float16 pattern of 1024 and one subtraction.)
 *   scales : bfloat16 [K/group, M_pad] (M_pad = M rounded up to 128), s_x of token m, group g
 *            at [g * M_pad + m]
 *   ab     : no region (ab_off == phat_off); kept in the call for the layout's stability
 *   p_hat  : float16 [M, r_pad] (r_pad = r rounded up to 16; columns >= r are zero)
 * The workspace is transient (written by qwam_asp_quantize_act, read by qwam_asp_gemm); the
 * weights are the part of the layer that stays packed at 4 bits. */
qwam_status qwam_asp_act_layout(qwam_asp_handle h, int M, size_t* codes_off, size_t* scales_off,
                                size_t* ab_off, size_t* phat_off, int* M_pad, int* r_pad);

/* Kernel (a): Eq. (xsplit) and the run-time half of Eq. (quant), one launch, asynchronous.
 *   X_bf16 : device, bf16 [M, K] row-major;  act_ws : device workspace (see above), written
 * Reads X once from HBM, forms p = X U on tensor cores (bf16 hi/lo split of U, float32
 * accumulation), X_perp = X - p U^T in float32, and writes the packed codes, bfloat16 scales and
 * p_hat. */
qwam_status qwam_asp_quantize_act(const void* X_bf16, int M, qwam_asp_handle h, void* act_ws,
                                  struct CUstream_st* stream);

/* Kernel (b): the 4-bit GEMM with the low-rank branch in its epilogue, asynchronous.
 *   act_ws : device workspace filled by qwam_asp_quantize_act for the same M
 *   Y      : device [M, N] row-major, bf16 (y_dtype QWAM_Y_BF16) or float32 (QWAM_Y_FP32)
 * Both operands stay packed at four bits in HBM.  With bfloat16 scales every dequantized value
 * s c has at most 11 significant bits, so the kernel forms s_x c and s_w c in float16 (exactly,
 * after a power-of-two scaling per token row and per output column that keeps them in float16's
 * range and is undone in the epilogue) and the tensor cores contract [s_x q_x | p_hat] with
 * [s_w q_w | B_hat] over K + r_pad in one float32 accumulator (tcgen05.mma kind::f16): the
 * group scales and the 16-bit branch need no separate pass.  The result differs from the exact
 * sum of Eq. (asp) only by the float32 accumulation. */
qwam_status qwam_asp_gemm(const void* act_ws, int M, qwam_asp_handle h, void* Y, int y_dtype,
                          struct CUstream_st* stream);

/* The whole layer: qwam_asp_quantize_act followed by qwam_asp_gemm on `stream`.  For an INT4 layer
 * of 512 or more tokens with r > 0, kernel (a) also writes the float16 copy of the weights into
 * act_ws (while its first pass waits on HBM) and the GEMM uses it, instead of the separate
 * expansion that qwam_asp_gemm runs when called on its own: the same results, one launch fewer. */
qwam_status qwam_asp_linear(const void* X_bf16, int M, qwam_asp_handle h, void* Y, int y_dtype,
                            void* act_ws, struct CUstream_st* stream);

/* ---- the layer without a caller-provided workspace ---------------------------------------
 * The paper has no counterpart to this call: it is a convenience of this library.
 *
 * qwam_asp_linear needs the caller to hand it `act_ws`, a device buffer.  Some callers cannot
 * provide one: a plain C host without a device allocator of its own, or a serving loop that
 * must not allocate on its hot path (cudaMalloc and cudaFree may synchronize the device and
 * fragment memory).  qwam_asp_linear_static runs the same two kernels as qwam_asp_linear, on
 * `stream`, but with a scratch buffer that the library reserves statically in device memory
 * (QWAM_STATIC_WS_BYTES per device, set aside when the library's device code is loaded).  It
 * allocates nothing: no cudaMalloc, no cudaFree, no allocating library routine.
 *
 *   - Size limit: the workspace must fit in QWAM_STATIC_WS_BYTES (24 MiB); larger requests return
 *     QWAM_ERR_TOO_LARGE before anything is launched.  This call uses the workspace without the
 *     per-call float16 copy of the weights that qwam_asp_act_workspace_bytes counts for INT4
 *     layers of 512 or more tokens (its GEMM converts the weights tile by tile instead), so it
 *     needs less than qwam_asp_act_workspace_bytes reports for such layers.  Per token the workspace holds about K/2 + 2K/G + 2 r_pad bytes (INT4) or
 *     K/2 + K/16 + 2 r_pad bytes (NVFP4), plus 4 C r_pad bytes for kernel (a)'s exchange of
 *     partial projections (C = 2, 4 or 8 CTAs per row tile, fewer for more tokens): at K = 3072,
 *     group 64, r = 32 about 2.2 KB, so up to about 12,800 tokens fit.  A rotated handle with
 *     r > 0 also keeps its float32 remainder, 4K more bytes per token: at K = 3072 about 1,660
 *     tokens fit, and M = 4096 is refused.
 *   - Nothing in the scratch needs to start at zero: kernel (a) writes every byte the GEMM
 *     then reads, on every call, so the scratch is never cleared.
 *   - One scratch per device: calls that may overlap in time on one device (different streams
 *     without ordering between them, or different host threads) race on it and give wrong
 *     results.  Order such calls, e.g. issue them on one stream.
 *   - The first call on each device looks the scratch's device address up (cudaGetSymbolAddress,
 *     with that device current) and keeps it; later calls reuse it.  Make that first call
 *     before any stream capture begins on the stream you pass.  The kept address belongs to
 *     the device context of that first call: after cudaDeviceReset (or any other reset of the
 *     device's primary context) the library's device code is loaded anew and the kept address
 *     is stale, so a process that resets a device must not call this function again on it.
 * Other arguments and errors are those of qwam_asp_linear; the handle's device must be current. */
#define QWAM_STATIC_WS_BYTES (24u * 1024u * 1024u)
qwam_status qwam_asp_linear_static(const void* X_bf16, int M, qwam_asp_handle h, void* Y, int y_dtype,
                                   struct CUstream_st* stream);

/* ---- NVFP4 variant (App. B.1) -----------------------------------------------------------
 * On Blackwell GPUs the paper stores the 4-bit operands as NVFP4: E2M1 values with an E4M3
 * scale for every 16 consecutive input channels, for weights and activations, and one more
 * float32 scale per weight tensor.  The paper fixes that storage format only; this library
 * reads the rest as follows (each exactly as the CPU reference computes it):
 *   - E2M1 values 0, 0.5, 1, 1.5, 2, 3, 4, 6 (and negatives); E4M3 the OCP FP8 "FN" format
 *     (largest finite 448).  Rounding to either is to nearest, ties to even, saturating; a code
 *     of magnitude zero is stored as 0.
 *   - Activations, per token and block b of 16: s = RN_e4m3(RN_f32(amax_b / 6)),
 *     code = RN_e2m1(RN_f32(x_perp / s)) (float32 IEEE division); s == 0 gives zero codes.
 *   - Weights: s_g = RN_f32(amax(W_perp) / (6 * 448)); per output channel and block,
 *     s_b = RN_e4m3(amax_b / (6 s_g)) and code = RN_e2m1(w / (s_b s_g)), both from the float64
 *     quotient.
 *   - Y = s_g sum_b s_a s_b sum_{k in b} qa qb  +  p_hat B_hat.  The block scales are applied by
 *     the tensor cores (tcgen05.mma kind::mxf4nvf4 block_scale, float32 accumulation); the
 *     epilogue multiplies by s_g and adds the branch.
 * The projection, the remainder, p_hat and the branch are those of the INT4 layer above.
 *
 * A handle made by qwam_asp_pack_weights_nvfp4 is used with the same calls as an INT4 handle
 * (qwam_asp_act_workspace_bytes, qwam_asp_act_layout, qwam_asp_quantize_act, qwam_asp_gemm,
 * qwam_asp_linear, qwam_asp_linear_static, qwam_asp_debug_residual), which dispatch on its
 * format.  Its activation workspace for M tokens holds:
 *   codes  : uint8 [M, K/2], two E2M1 codes per byte, low nibble = even k
 *   scales : uint8 E4M3 block scales, M_pad * K/16 bytes, in 512-byte atoms: atom
 *            (m / 128, k / 64) starts at ((m / 128) * (K / 64) + k / 64) * 512, and within it the
 *            four scales of token m (k / 16 in order) start at byte (m % 32) * 16 +
 *            ((m % 128) / 32) * 4.  This is the order in which tcgen05.cp.32x128b.warpx4 places
 *            them in tensor memory where the block-scaled MMA reads them.
 *   ab     : empty (qwam_asp_act_layout reports ab_off == phat_off)
 *   p_hat  : float16 [M, r_pad], as for INT4.                                              */
enum { QWAM_FMT_INT4 = 0, QWAM_FMT_NVFP4 = 1 };

/* Offline packing of the NVFP4 variant.  Arguments as for qwam_asp_pack_weights, without the
 * group (the block is 16); K % 256 == 0.  Synchronizes `stream` before returning. */
qwam_status qwam_asp_pack_weights_nvfp4(const void* W_bf16, const float* U, int K, int N, int r,
                                        struct CUstream_st* stream, qwam_asp_handle* out);

/* ---- Smoothing and block Hadamard rotation in front of the layer (Sec. 3 Eq. (pair); App. B.1)
 * The paper quantizes in rotated coordinates: with per-channel smoothing factors s (App. B.1:
 * s_j = max|X_j|^alpha / max|W_j,:|^(1-alpha), see qwam_asp_smoothing_factors) and the block
 * Hadamard matrix H (block-diagonal, each block the Sylvester Hadamard matrix of size B divided by
 * sqrt(B), B the largest power of two dividing K, at most 1024; H is symmetric and orthogonal),
 *   x~ = H diag(s)^-1 x,   W~ = H diag(s) W,   so that W~^T x~ = W^T x,
 * and ASP runs on x~ and W~ with a basis U given in the rotated coordinates (for instance the one
 * qwam_asp_action_subspace returns for the rotated Gramian).
 *
 * These two calls pack W~ (formed in float64 on the device: W times s_k, the fast Walsh-Hadamard
 * butterflies at spans 1, 2, ..., B/2 inside each block, then times 1/sqrt(B); every operation one
 * float64 rounding) exactly as qwam_asp_pack_weights / qwam_asp_pack_weights_nvfp4 pack a weight,
 * against U.  The handle's activation calls (qwam_asp_quantize_act, qwam_asp_linear,
 * qwam_asp_linear_static, qwam_asp_debug_residual) then take X in the ORIGINAL coordinates and
 * rotate it at run time: the projection p = x~ U is computed as x (diag(s)^-1 H U), the remainder
 * as H diag(s)^-1 (x - diag(s) H U p) = x~ - U p in float32 (the fast Walsh-Hadamard transform,
 * float32), and that is quantized.  With r > 0 the activation workspace also holds the float32
 * remainder before the rotation (M * K * 4 more bytes; qwam_asp_act_workspace_bytes includes
 * them).  qwam_asp_debug_residual writes the rotated remainder x~_perp.
 *   W_bf16, U, K, N, r, group, stream, out: as for qwam_asp_pack_weights (or _nvfp4), and
 *     K % 256 == 0 (QWAM_ERR_INVALID_ARG otherwise).
 *   s : device float32 [K], 16-byte aligned, the smoothing factors; NULL for the rotation alone.
 *       A factor that is not a positive finite number gives QWAM_ERR_RANGE.
 * Synchronizes `stream` before returning; the temporary float64 W~ (K * N * 8 bytes) is freed. */
qwam_status qwam_asp_pack_weights_rotated(const void* W_bf16, const float* s, const float* U, int K, int N, int r,
                                          int group, struct CUstream_st* stream, qwam_asp_handle* out);
qwam_status qwam_asp_pack_weights_nvfp4_rotated(const void* W_bf16, const float* s, const float* U, int K, int N,
                                                int r, struct CUstream_st* stream, qwam_asp_handle* out);

/* The Hadamard block B of a rotated handle, 0 for a handle without rotation. */
qwam_status qwam_asp_rotation(qwam_asp_handle h, int* hadamard_block);

/* The handle's format: QWAM_FMT_INT4 or QWAM_FMT_NVFP4. */
qwam_status qwam_asp_format(qwam_asp_handle h, int* format);

/* Copy the packed NVFP4 weights to HOST buffers (any may be NULL), synchronously:
 *   qw  : uint8 [N, K/2] E2M1 codes of W_perp, low nibble = even k
 *   sfw : uint8 [N, K/16] E4M3 block scales, row-major
 *   sg  : the float32 per-tensor scale
 *   Bh  : uint16 (float16 bits) [N, r_pad]
 * Returns QWAM_ERR_INVALID_ARG for an INT4 handle (and qwam_asp_export does for an NVFP4 one). */
qwam_status qwam_asp_export_nvfp4(qwam_asp_handle h, void* qw, void* sfw, float* sg, void* Bh);

/* Read-and-clear: returns the handle's device-side error word (QWAM_OK, QWAM_ERR_TIMEOUT or
 * QWAM_ERR_RANGE) and resets it to QWAM_OK.  The word keeps the first error of any launch of
 * the handle until this call reads it.  The call waits for the handle's last launch made outside
 * a stream capture (an event on that launch's stream), not for the whole device: other streams
 * and other users of the GPU go on.  Launches captured into a CUDA graph are not tracked:
 * synchronize the stream that replays the graph before calling.  A timeout in kernel (a) does not
 * stop the GEMM that follows it on the stream from running on the half-written workspace: treat
 * the outputs of every launch since the last QWAM_OK as invalid when this returns an error. */
qwam_status qwam_asp_get_error(qwam_asp_handle h);

/* Shape of a handle (any output pointer may be NULL); `group` is 16 for an NVFP4 handle. */
qwam_status qwam_asp_shape(qwam_asp_handle h, int* K, int* N, int* r, int* group, int* r_pad);

/* Copy the packed weights to HOST buffers (any may be NULL), synchronously:
 *   qw  : uint8 [N, K/2] codes of W_perp, low nibble = even k (two's complement)
 *   sw  : uint16 (bfloat16 bits) [K/group, N]
 *   Bh  : uint16 (float16 bits) [N, r_pad]   (B_hat transposed, zero beyond r)
 *   Uhl : uint16 (bf16 bits) [2, K, r_pad]   (hi and lo parts of the projection basis: U, or
 *         diag(s)^-1 H U for a rotated handle; zero beyond r; all zero for r > 64, whose
 *         general-rank path keeps the basis in float32 only) */
qwam_status qwam_asp_export(qwam_asp_handle h, void* qw, void* sw, void* Bh, void* Uhl);

/* Free the handle and its device buffers (synchronizes the device). */
qwam_status qwam_asp_destroy(qwam_asp_handle h);

/* Bias of the layer (App. B.1: the GEMM kernel adds the bias in its epilogue).  `bias` is a
 * device float32 [N], 16-byte aligned; it is copied into the handle (synchronously on `stream`),
 * and every later qwam_asp_gemm / qwam_asp_linear / qwam_asp_linear_static of the handle stores
 * Y[m, n] = RN(acc[m, n] + bias[n]) with acc the float32 result described above (one float32
 * addition, then the conversion to the output type).  NULL removes the bias.  Errors:
 * QWAM_ERR_INVALID_ARG (no handle, unaligned bias), QWAM_ERR_OOM, QWAM_ERR_CUDA. */
qwam_status qwam_asp_set_bias(qwam_asp_handle h, const float* bias, struct CUstream_st* stream);

const char* qwam_status_string(qwam_status s);

/* ---- test support ------------------------------------------------------------------------ */

/* Kernel (a) with one more output: R, device float32 [M, K], receives X_perp exactly as the
 * kernel forms it before quantization (so the quantizer can be checked bit for bit). */
qwam_status qwam_asp_debug_residual(const void* X_bf16, int M, qwam_asp_handle h, void* act_ws, float* R,
                                    struct CUstream_st* stream);

/* Test support: kernel (a)'s quantizer alone (Eq. (quant) with the rounding of readings R2, R3
 * and R5; for fmt == QWAM_FMT_NVFP4 the block rule of App. B.1 read as N1-N3) applied to
 * caller-given float32 rows, so that its rounding can be checked on chosen values such as exact
 * ties and values a few units in the last place from a rounding boundary.  No handle is needed.
 *   R      : device float32 [M, K], row-major, 16-byte aligned; K % 64 == 0
 *   fmt    : QWAM_FMT_INT4 or QWAM_FMT_NVFP4
 *   group  : 32 or 64 for INT4 (ignored for NVFP4, whose block is 16)
 *   codes  : device, 16-byte aligned.  INT4: uint8 [M, K/2], OB4 words as in the activation
 *            workspace.  NVFP4: uint8 [M, K/2], two E2M1 codes per byte, low nibble = even k.
 *   scales : device.  INT4: bfloat16 [M, K/group] row-major (2-byte aligned).  NVFP4: uint8 E4M3
 *            bit patterns [M, K/16] row-major.
 * Asynchronous on `stream`; QWAM_ERR_INVALID_ARG for bad sizes, formats or alignment. */
qwam_status qwam_asp_debug_quantize_rows(const float* R, int M, int K, int fmt, int group, void* codes,
                                         void* scales, struct CUstream_st* stream);

/* Test support: the warp-wide quantizers of the small-M and rotation kernels (8 consecutive values
 * per lane, a group over neighbouring lanes) on caller-given float32 rows, with the same rounding
 * rules as qwam_asp_debug_quantize_rows; K % 256 == 0.  Outputs are written in the activation
 * workspace's layouts with M_pad = ceil(M / 128) * 128 rows:
 *   INT4:  codes uint8 [M, K/2] (OB4 words, described at qwam_asp_act_layout), scales bfloat16
 *          [K/group, M_pad];
 *   NVFP4: codes uint8 [M, K/2] (two per byte, low nibble = even k), scales uint8 E4M3 in the
 *          512-byte atoms described above (M_pad * K/16 bytes).
 * Device pointers; codes 16-byte aligned.  Errors: QWAM_ERR_INVALID_ARG, QWAM_ERR_CUDA. */
qwam_status qwam_asp_debug_quantize_lanes(const float* R, int M, int K, int fmt, int group, void* codes,
                                          void* scales, struct CUstream_st* stream);

/* ---- The offline choice of what to protect (Sec. 4.2-4.3; App. A; App. B.1) -----------------
 * Calibration-time steps that pick U (the paper's V) and which experts carry a branch, from a given
 * Action Observability Gramian G (the AOG of Sec. 4.1, estimated elsewhere).  None of them needs a
 * handle.  All matrices are float32, row-major, on the device unless stated otherwise.        */

/* Smoothing factors of App. B.1: s_j = xmax_j^alpha / max_n |W[j, n]|^(1 - alpha) for every input
 * channel j (row j of W).  xmax [K] (device float32): each channel's calibration maximum |x_j|;
 * W_bf16 [K, N] device; alpha in [0, 1]; s [K] device float32 output.  A channel whose activation
 * or weight maximum is zero is left unsmoothed (s_j = 1).  Computed in float64, rounded once.
 * Asynchronous on `stream`. */
qwam_status qwam_asp_smoothing_factors(const float* xmax, const void* W_bf16, int K, int N, double alpha, float* s,
                                       struct CUstream_st* stream);

/* The AOG in the rotated coordinates (Sec. 4.2): Gt = H diag(gamma) G diag(gamma) H, with H the block
 * Hadamard rotation of Eq. (pair) (normalised Sylvester blocks of size B, the largest power of two
 * dividing d, at most 1024).  G, Gt, work: [d, d] (work is scratch); gamma [d] or NULL for no
 * smoothing.  G, Gt and work must be distinct.  d <= 32768.  Asynchronous on `stream`. */
qwam_status qwam_asp_rotated_gramian(const float* G, const float* gamma, int d, float* Gt, float* work,
                                     struct CUstream_st* stream);

/* tr(A) of a [d, d] device matrix, accumulated in float64 and returned in *trace (host): the
 * per-layer term of an expert's action mass mu_E = sum of tr Gt (Sec. 4.3, Eq. (mass)).
 * Synchronizes `stream`. */
qwam_status qwam_asp_gramian_trace(const float* A, int d, double* trace, struct CUstream_st* stream);

/* Scratch bytes of qwam_asp_action_subspace for a [d, d] matrix and rank r (1 <= r <= min(d, 96)). */
qwam_status qwam_asp_subspace_workspace_bytes(int d, int r, size_t* bytes);

/* The action subspace (Sec. 4.2, Eq. (gtilde); App. A): the eigenvectors of the r largest
 * eigenvalues of the symmetric positive semidefinite Gt [d, d].  V [d, r] receives them as columns
 * (decreasing eigenvalue, orthonormal; each column's sign is arbitrary) and lambda [r] (device)
 * the eigenvalues.  Subspace iteration with r + max(8, r/2) vectors (at most 96) for `iters`
 * steps, then a Rayleigh-Ritz step: the subspace's error falls like (lambda_{p+1}/lambda_r)^iters,
 * so a spectrum with a gap after the r-th eigenvalue converges in few steps.  work: device scratch
 * of qwam_asp_subspace_workspace_bytes, 16-byte aligned.  Synchronizes `stream`. */
qwam_status qwam_asp_action_subspace(const float* Gt, int d, int r, int iters, float* V, float* lambda, void* work,
                                     struct CUstream_st* stream);

/* Which experts to protect (Sec. 4.3): in decreasing order of action mass per added 16-bit value,
 * mass[i] / cost[i] (equal ratios: lower index first), each expert whose added values still fit the
 * budget.  mass[n] >= 0, cost[n] > 0 (the 16-bit values its branches add, r (d + d') per layer),
 * host arrays; chosen[n] (host) receives the chosen indices in that order and *n_chosen their count.
 * Host only. */
qwam_status qwam_asp_select_experts(const double* mass, const double* cost, int n, double budget, int* chosen,
                                    int* n_chosen);

/* Set the bound of every device wait of this handle's kernels, in seconds (default 2.0). */
qwam_status qwam_asp_set_timeout(qwam_asp_handle h, double seconds);

/* Activation path for few tokens.  On a handle with K % 256 == 0, calls with M <= max_rows tokens
 * (default 256), and calls of any M on an r = 0 handle without rotation, run the activation side
 * on the CUDA cores, one CTA per token (float32 projection and remainder, the rotation of a
 * rotated handle, the same quantizers); other calls take the tensor-core kernel (and, for a
 * rotated handle, the rotation kernel).  Both meet the same parity bars; max_rows = 0 always
 * takes the tensor-core kernel.
 * Errors: QWAM_ERR_INVALID_ARG (no handle, max_rows < 0). */
qwam_status qwam_asp_set_small_m(qwam_asp_handle h, int max_rows);

/* Launch one CTA that waits on a shared-memory barrier nothing arrives on, with a bound of
 * `timeout_us` microseconds; the wait runs out, the kernel records QWAM_ERR_TIMEOUT in the
 * handle's error word and returns.  Exercises the bounded-wait path without a fault. */
qwam_status qwam_asp_debug_wait_timeout(qwam_asp_handle h, int timeout_us, struct CUstream_st* stream);

#ifdef __cplusplus
}
#endif
#endif /* QWAM_ASP_H */
