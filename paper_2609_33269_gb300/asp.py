"""Python binding of libqwam_asp.so (C ABI in include/qwam_asp.h).

Argument marshalling only: every step of the layer runs in the library's CUDA kernels.  PyTorch
supplies device memory and the current stream.  There is no fallback: if the shared library is
missing or fails to load, every call raises.

The functions keep the C names (qwam_asp_pack_weights, qwam_asp_quantize_act, qwam_asp_linear,
...).  ``AspLinear`` bundles a handle with its activation workspace for convenience.
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libqwam_asp.so")

QWAM_OK = 0
QWAM_ERR_INVALID_ARG = -1
QWAM_ERR_UNSUPPORTED = -2
QWAM_ERR_CUDA = -3
QWAM_ERR_OOM = -4
QWAM_ERR_TIMEOUT = -5
QWAM_ERR_RANGE = -6
QWAM_ERR_TOO_LARGE = -7
STATIC_WS_BYTES = 24 * 1024 * 1024  # QWAM_STATIC_WS_BYTES of the header
QWAM_Y_BF16 = 0
QWAM_Y_FP32 = 1
QWAM_FMT_INT4 = 0
QWAM_FMT_NVFP4 = 1

EXPORTED = [
    "qwam_asp_pack_weights", "qwam_asp_act_workspace_bytes", "qwam_asp_act_layout",
    "qwam_asp_quantize_act", "qwam_asp_gemm", "qwam_asp_linear", "qwam_asp_get_error",
    "qwam_asp_shape", "qwam_asp_export", "qwam_asp_destroy", "qwam_status_string",
    "qwam_asp_debug_residual", "qwam_asp_set_timeout", "qwam_asp_debug_wait_timeout",
    "qwam_asp_linear_static", "qwam_asp_pack_weights_nvfp4", "qwam_asp_format", "qwam_asp_export_nvfp4",
    "qwam_asp_debug_quantize_rows", "qwam_asp_smoothing_factors", "qwam_asp_rotated_gramian",
    "qwam_asp_gramian_trace", "qwam_asp_subspace_workspace_bytes", "qwam_asp_action_subspace",
    "qwam_asp_select_experts", "qwam_asp_pack_weights_rotated", "qwam_asp_pack_weights_nvfp4_rotated",
    "qwam_asp_rotation", "qwam_asp_set_bias", "qwam_asp_set_small_m", "qwam_asp_debug_quantize_lanes",
]

_lib = None
_lock = threading.Lock()


class QwamError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__(f"{what}: {status_string(status)} ({status})")


def load(path: str | None = None) -> ctypes.CDLL:
    """Load the shared library (does not build it; see ``paper_2609_33269_gb300.build``)."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        p = path or LIB_PATH
        if not os.path.exists(p):
            raise RuntimeError(f"libqwam_asp.so not built ({p}); run __graft_entry__.build()")
        lib = ctypes.CDLL(p)
        V, I, S, H = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t, ctypes.c_void_p
        lib.qwam_asp_pack_weights.argtypes = [V, V, I, I, I, I, V, ctypes.POINTER(H)]
        lib.qwam_asp_act_workspace_bytes.argtypes = [H, I, ctypes.POINTER(S)]
        lib.qwam_asp_act_layout.argtypes = [H, I, ctypes.POINTER(S), ctypes.POINTER(S), ctypes.POINTER(S),
                                            ctypes.POINTER(S), ctypes.POINTER(I), ctypes.POINTER(I)]
        lib.qwam_asp_quantize_act.argtypes = [V, I, H, V, V]
        lib.qwam_asp_gemm.argtypes = [V, I, H, V, I, V]
        lib.qwam_asp_linear.argtypes = [V, I, H, V, I, V, V]
        lib.qwam_asp_linear_static.argtypes = [V, I, H, V, I, V]
        lib.qwam_asp_get_error.argtypes = [H]
        lib.qwam_asp_shape.argtypes = [H] + [ctypes.POINTER(I)] * 5
        lib.qwam_asp_export.argtypes = [H, V, V, V, V]
        lib.qwam_asp_destroy.argtypes = [H]
        lib.qwam_status_string.argtypes = [I]
        lib.qwam_status_string.restype = ctypes.c_char_p
        lib.qwam_asp_debug_residual.argtypes = [V, I, H, V, V, V]
        lib.qwam_asp_debug_quantize_rows.argtypes = [V, I, I, I, I, V, V, V]
        lib.qwam_asp_smoothing_factors.argtypes = [V, V, I, I, ctypes.c_double, V, V]
        lib.qwam_asp_rotated_gramian.argtypes = [V, V, I, V, V, V]
        lib.qwam_asp_gramian_trace.argtypes = [V, I, V, V]
        lib.qwam_asp_subspace_workspace_bytes.argtypes = [I, I, V]
        lib.qwam_asp_action_subspace.argtypes = [V, I, I, I, V, V, V, V]
        lib.qwam_asp_select_experts.argtypes = [V, V, I, ctypes.c_double, V, V]
        lib.qwam_asp_set_timeout.argtypes = [H, ctypes.c_double]
        lib.qwam_asp_debug_wait_timeout.argtypes = [H, I, V]
        lib.qwam_asp_pack_weights_nvfp4.argtypes = [V, V, I, I, I, V, ctypes.POINTER(H)]
        lib.qwam_asp_format.argtypes = [H, ctypes.POINTER(I)]
        lib.qwam_asp_pack_weights_rotated.argtypes = [V, V, V, I, I, I, I, V, ctypes.POINTER(H)]
        lib.qwam_asp_pack_weights_nvfp4_rotated.argtypes = [V, V, V, I, I, I, V, ctypes.POINTER(H)]
        lib.qwam_asp_rotation.argtypes = [H, ctypes.POINTER(I)]
        lib.qwam_asp_set_bias.argtypes = [H, V, V]
        lib.qwam_asp_set_small_m.argtypes = [H, I]
        lib.qwam_asp_debug_quantize_lanes.argtypes = [V, I, I, I, I, V, V, V]
        lib.qwam_asp_export_nvfp4.argtypes = [H, V, V, ctypes.POINTER(ctypes.c_float), V]
        for name in EXPORTED:
            if name != "qwam_status_string":
                getattr(lib, name).restype = I
        _lib = lib
        return lib


def status_string(status: int) -> str:
    return load().qwam_status_string(int(status)).decode()


def _check(status: int, what: str):
    if status != QWAM_OK:
        raise QwamError(status, what)


def _ptr(t) -> int | None:
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(stream=None) -> int | None:
    s = stream if stream is not None else torch.cuda.current_stream()
    return s.cuda_stream if hasattr(s, "cuda_stream") else s


# ------------------------------------------------------------------ C entry points, same names

def qwam_asp_pack_weights(W_bf16, U, K: int, N: int, r: int, group: int, stream=None) -> int:
    h = ctypes.c_void_p()
    _check(load().qwam_asp_pack_weights(_ptr(W_bf16), _ptr(U), K, N, r, group, _stream(stream),
                                        ctypes.byref(h)), "qwam_asp_pack_weights")
    return h.value


def qwam_asp_pack_weights_nvfp4(W_bf16, U, K: int, N: int, r: int, stream=None) -> int:
    h = ctypes.c_void_p()
    _check(load().qwam_asp_pack_weights_nvfp4(_ptr(W_bf16), _ptr(U), K, N, r, _stream(stream), ctypes.byref(h)),
           "qwam_asp_pack_weights_nvfp4")
    return h.value


def qwam_asp_pack_weights_rotated(W_bf16, s, U, K: int, N: int, r: int, group: int, stream=None) -> int:
    h = ctypes.c_void_p()
    _check(load().qwam_asp_pack_weights_rotated(_ptr(W_bf16), _ptr(s), _ptr(U), K, N, r, group, _stream(stream),
                                                ctypes.byref(h)), "qwam_asp_pack_weights_rotated")
    return h.value


def qwam_asp_pack_weights_nvfp4_rotated(W_bf16, s, U, K: int, N: int, r: int, stream=None) -> int:
    h = ctypes.c_void_p()
    _check(load().qwam_asp_pack_weights_nvfp4_rotated(_ptr(W_bf16), _ptr(s), _ptr(U), K, N, r, _stream(stream),
                                                      ctypes.byref(h)), "qwam_asp_pack_weights_nvfp4_rotated")
    return h.value


def qwam_asp_set_bias(h: int, bias, stream=None):
    """Bias [N] float32 (device) added in the GEMM epilogue; None removes it."""
    _check(load().qwam_asp_set_bias(h, _ptr(bias), _stream(stream)), "qwam_asp_set_bias")


def qwam_asp_set_small_m(h: int, max_rows: int):
    """Token counts up to max_rows take the small-M (CUDA-core) activation kernel; 0 never."""
    _check(load().qwam_asp_set_small_m(h, int(max_rows)), "qwam_asp_set_small_m")


def qwam_asp_rotation(h: int) -> int:
    b = ctypes.c_int()
    _check(load().qwam_asp_rotation(h, ctypes.byref(b)), "qwam_asp_rotation")
    return b.value


def qwam_asp_format(h: int) -> int:
    f = ctypes.c_int()
    _check(load().qwam_asp_format(h, ctypes.byref(f)), "qwam_asp_format")
    return f.value


def qwam_asp_act_workspace_bytes(h: int, M: int) -> int:
    b = ctypes.c_size_t()
    _check(load().qwam_asp_act_workspace_bytes(h, M, ctypes.byref(b)), "qwam_asp_act_workspace_bytes")
    return b.value


def qwam_asp_act_layout(h: int, M: int) -> dict:
    c, s, cs, p = ctypes.c_size_t(), ctypes.c_size_t(), ctypes.c_size_t(), ctypes.c_size_t()
    mp, rp = ctypes.c_int(), ctypes.c_int()
    _check(load().qwam_asp_act_layout(h, M, ctypes.byref(c), ctypes.byref(s), ctypes.byref(cs), ctypes.byref(p),
                                      ctypes.byref(mp), ctypes.byref(rp)), "qwam_asp_act_layout")
    return dict(codes_off=c.value, scales_off=s.value, ab_off=cs.value, phat_off=p.value, M_pad=mp.value,
                r_pad=rp.value)


def qwam_asp_quantize_act(X_bf16, M: int, h: int, act_ws, stream=None):
    _check(load().qwam_asp_quantize_act(_ptr(X_bf16), M, h, _ptr(act_ws), _stream(stream)), "qwam_asp_quantize_act")


def qwam_asp_gemm(act_ws, M: int, h: int, Y, y_dtype: int, stream=None):
    _check(load().qwam_asp_gemm(_ptr(act_ws), M, h, _ptr(Y), y_dtype, _stream(stream)), "qwam_asp_gemm")


def qwam_asp_linear(X_bf16, M: int, h: int, Y, y_dtype: int, act_ws, stream=None):
    _check(load().qwam_asp_linear(_ptr(X_bf16), M, h, _ptr(Y), y_dtype, _ptr(act_ws), _stream(stream)),
           "qwam_asp_linear")


def qwam_asp_linear_static(X_bf16, M: int, h: int, Y, y_dtype: int, stream=None):
    """The layer with the library's static scratch workspace (no act_ws; see the header)."""
    _check(load().qwam_asp_linear_static(_ptr(X_bf16), M, h, _ptr(Y), y_dtype, _stream(stream)),
           "qwam_asp_linear_static")


def qwam_asp_get_error(h: int) -> int:
    return int(load().qwam_asp_get_error(h))


def qwam_asp_shape(h: int) -> dict:
    v = [ctypes.c_int() for _ in range(5)]
    _check(load().qwam_asp_shape(h, *[ctypes.byref(x) for x in v]), "qwam_asp_shape")
    return dict(zip(("K", "N", "r", "group", "r_pad"), (x.value for x in v)))


def qwam_asp_export(h: int):
    """Packed weights on the host: qw uint8 [N, K/2], sw bfloat16-bits [K/G, N],
    Bh float16-bits [N, r_pad], Uhl bf16-bits [2, K, r_pad] (numpy arrays)."""
    import numpy as np
    sh = qwam_asp_shape(h)
    K, N, G, rp = sh["K"], sh["N"], sh["group"], sh["r_pad"]
    qw = np.empty((N, K // 2), np.uint8)
    sw = np.empty((K // G, N), np.uint16)
    Bh = np.empty((N, rp), np.uint16)
    Uhl = np.empty((2, K, rp), np.uint16)
    _check(load().qwam_asp_export(h, qw.ctypes.data, sw.ctypes.data, Bh.ctypes.data if rp else None,
                                  Uhl.ctypes.data if rp else None), "qwam_asp_export")
    return dict(qw=qw, sw=sw, Bh=Bh, Uhl=Uhl)


def qwam_asp_export_nvfp4(h: int):
    """Packed NVFP4 weights on the host: qw uint8 [N, K/2] (low nibble = even k), sfw uint8
    E4M3 bits [N, K/16], sg float32, Bh float16-bits [N, r_pad] (numpy)."""
    import numpy as np
    sh = qwam_asp_shape(h)
    K, N, rp = sh["K"], sh["N"], sh["r_pad"]
    qw = np.empty((N, K // 2), np.uint8)
    sfw = np.empty((N, K // 16), np.uint8)
    sg = ctypes.c_float()
    Bh = np.empty((N, rp), np.uint16)
    _check(load().qwam_asp_export_nvfp4(h, qw.ctypes.data, sfw.ctypes.data, ctypes.byref(sg),
                                        Bh.ctypes.data if rp else None), "qwam_asp_export_nvfp4")
    return dict(qw=qw, sfw=sfw, sg=np.float32(sg.value), Bh=Bh)


def qwam_asp_destroy(h: int):
    _check(load().qwam_asp_destroy(h), "qwam_asp_destroy")


def qwam_asp_debug_residual(X_bf16, M: int, h: int, act_ws, R, stream=None):
    _check(load().qwam_asp_debug_residual(_ptr(X_bf16), M, h, _ptr(act_ws), _ptr(R), _stream(stream)),
           "qwam_asp_debug_residual")


def qwam_asp_debug_quantize_rows(R, M: int, K: int, fmt: int, group: int, codes, scales, stream=None):
    _check(load().qwam_asp_debug_quantize_rows(_ptr(R), M, K, fmt, group, _ptr(codes), _ptr(scales),
                                               _stream(stream)), "qwam_asp_debug_quantize_rows")


def qwam_asp_debug_quantize_lanes(R, M: int, K: int, fmt: int, group: int, codes, scales, stream=None):
    _check(load().qwam_asp_debug_quantize_lanes(_ptr(R), M, K, fmt, group, _ptr(codes), _ptr(scales),
                                                _stream(stream)), "qwam_asp_debug_quantize_lanes")


def qwam_asp_smoothing_factors(xmax, W_bf16, K: int, N: int, alpha: float, s, stream=None):
    _check(load().qwam_asp_smoothing_factors(_ptr(xmax), _ptr(W_bf16), K, N, float(alpha), _ptr(s), _stream(stream)),
           "qwam_asp_smoothing_factors")


def qwam_asp_rotated_gramian(G, gamma, d: int, Gt, work, stream=None):
    _check(load().qwam_asp_rotated_gramian(_ptr(G), None if gamma is None else _ptr(gamma), d, _ptr(Gt), _ptr(work),
                                           _stream(stream)), "qwam_asp_rotated_gramian")


def qwam_asp_gramian_trace(A, d: int, stream=None) -> float:
    out = ctypes.c_double(0.0)
    _check(load().qwam_asp_gramian_trace(_ptr(A), d, ctypes.byref(out), _stream(stream)), "qwam_asp_gramian_trace")
    return out.value


def qwam_asp_subspace_workspace_bytes(d: int, r: int) -> int:
    out = ctypes.c_size_t(0)
    _check(load().qwam_asp_subspace_workspace_bytes(d, r, ctypes.byref(out)), "qwam_asp_subspace_workspace_bytes")
    return out.value


def qwam_asp_action_subspace(Gt, d: int, r: int, iters: int, V, lam, work, stream=None):
    _check(load().qwam_asp_action_subspace(_ptr(Gt), d, r, iters, _ptr(V), _ptr(lam), _ptr(work), _stream(stream)),
           "qwam_asp_action_subspace")


def qwam_asp_select_experts(mass, cost, budget: float):
    """Host-only: the chosen expert indices, in the order chosen (Sec. 4.3)."""
    import numpy as np
    m = np.ascontiguousarray(mass, np.float64)
    c = np.ascontiguousarray(cost, np.float64)
    n = m.shape[0]
    chosen = np.zeros(max(n, 1), np.int32)
    k = ctypes.c_int(0)
    _check(load().qwam_asp_select_experts(m.ctypes.data, c.ctypes.data, n, float(budget), chosen.ctypes.data,
                                          ctypes.byref(k)), "qwam_asp_select_experts")
    return [int(v) for v in chosen[:k.value]]


def qwam_asp_set_timeout(h: int, seconds: float):
    _check(load().qwam_asp_set_timeout(h, float(seconds)), "qwam_asp_set_timeout")


def qwam_asp_debug_wait_timeout(h: int, timeout_us: int, stream=None):
    _check(load().qwam_asp_debug_wait_timeout(h, int(timeout_us), _stream(stream)), "qwam_asp_debug_wait_timeout")


# ------------------------------------------------------------------ convenience wrapper

class AspLinear:
    """One packed ASP layer plus a reusable activation workspace on the current device."""

    def __init__(self, W_bf16: torch.Tensor, U: torch.Tensor | None, group: int = 64, stream=None,
                 fmt: int = QWAM_FMT_INT4, rotate: bool = False, s: torch.Tensor | None = None):
        """fmt QWAM_FMT_INT4 (group 32 or 64) or QWAM_FMT_NVFP4 (App. B.1's Blackwell format;
        `group` is then ignored: the block is 16).  rotate=True packs W~ = H diag(s) W (Sec. 3
        Eq. (pair); s float32 [K] smoothing factors or None) and rotates X at run time; U is then
        the basis in the rotated coordinates."""
        assert W_bf16.is_cuda and W_bf16.dtype == torch.bfloat16 and W_bf16.is_contiguous()
        K, N = W_bf16.shape
        r = 0 if U is None else U.shape[1]
        if U is not None:
            assert U.is_cuda and U.dtype == torch.float32 and U.is_contiguous() and U.shape[0] == K
        self.fmt = fmt
        self.K, self.N, self.r = K, N, r
        self.group = 16 if fmt == QWAM_FMT_NVFP4 else group
        if s is not None:
            assert rotate and s.is_cuda and s.dtype == torch.float32 and s.is_contiguous() and s.numel() == K
        self.rotate = rotate
        if rotate and fmt == QWAM_FMT_NVFP4:
            self.h = qwam_asp_pack_weights_nvfp4_rotated(W_bf16, s, U if r > 0 else None, K, N, r, stream)
        elif rotate:
            self.h = qwam_asp_pack_weights_rotated(W_bf16, s, U if r > 0 else None, K, N, r, group, stream)
        elif fmt == QWAM_FMT_NVFP4:
            self.h = qwam_asp_pack_weights_nvfp4(W_bf16, U if r > 0 else None, K, N, r, stream)
        else:
            self.h = qwam_asp_pack_weights(W_bf16, U if r > 0 else None, K, N, r, group, stream)
        self.r_pad = qwam_asp_shape(self.h)["r_pad"]
        self._ws = None
        self._ws_M = -1

    def workspace(self, M: int) -> torch.Tensor:
        if self._ws is None or self._ws_M < M:
            nbytes = qwam_asp_act_workspace_bytes(self.h, M)
            self._ws = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
            self._ws_M = M
        return self._ws

    def act_views(self, M: int, ws: torch.Tensor | None = None):
        """Views of the workspace for M tokens: packed codes uint8 [M, K/2] (OB4 words: word j of a
        row holds k = 8j..8j+7, see qwam_asp_act_layout), scales bf16 [K/G, M_pad], p_hat f16
        [M, r_pad]."""
        ws = self.workspace(M) if ws is None else ws
        L = qwam_asp_act_layout(self.h, M)
        if self.fmt == QWAM_FMT_NVFP4:
            return self.act_views_nvfp4(M, ws)
        codes = ws[L["codes_off"]:L["codes_off"] + M * (self.K // 2)].view(M, self.K // 2)
        ns = self.K // self.group
        scales = ws[L["scales_off"]:L["scales_off"] + ns * L["M_pad"] * 2].view(torch.bfloat16).view(ns, L["M_pad"])
        ph = ws[L["phat_off"]:L["phat_off"] + M * self.r_pad * 2].view(torch.float16).view(M, self.r_pad)
        return codes, scales, ph

    def act_views_nvfp4(self, M: int, ws: torch.Tensor | None = None):
        """NVFP4 workspace views: packed codes uint8 [M, K/2] (low nibble = even k), the scale
        atoms uint8 [M_pad * K/16] (see the header for their order), p_hat f16 [M, r_pad]."""
        ws = self.workspace(M) if ws is None else ws
        L = qwam_asp_act_layout(self.h, M)
        codes = ws[L["codes_off"]:L["codes_off"] + M * (self.K // 2)].view(M, self.K // 2)
        atoms = ws[L["scales_off"]:L["scales_off"] + L["M_pad"] * (self.K // 16)]
        ph = ws[L["phat_off"]:L["phat_off"] + M * self.r_pad * 2].view(torch.float16).view(M, self.r_pad)
        return codes, atoms, ph

    def quantize(self, X: torch.Tensor, stream=None) -> torch.Tensor:
        M = X.shape[0]
        ws = self.workspace(M)
        qwam_asp_quantize_act(X, M, self.h, ws, stream)
        return ws

    def __call__(self, X: torch.Tensor, out: torch.Tensor | None = None, fp32: bool = False, stream=None):
        assert X.is_cuda and X.dtype == torch.bfloat16 and X.is_contiguous() and X.shape[1] == self.K
        M = X.shape[0]
        if out is None:
            out = torch.empty((M, self.N), dtype=torch.float32 if fp32 else torch.bfloat16, device=X.device)
        ydt = QWAM_Y_FP32 if out.dtype == torch.float32 else QWAM_Y_BF16
        qwam_asp_linear(X, M, self.h, out, ydt, self.workspace(M), stream)
        return out

    def close(self):
        if getattr(self, "h", None):
            qwam_asp_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
