"""CPU oracle for the ASP linear layer (Q-WAM, Sec. 4.2 Eq. (asp); Sec. 3 Eq. (quant); App. B.1).

TEST INFRASTRUCTURE ONLY.  The tests, the smoke check and the CPU-baseline leg of the benchmark
load this module; the library under ``paper_2609_33269_gb300`` never imports it and shares no
code with it.  The arithmetic lives in ``qwam_oracle.c`` (float64 / int64, OpenMP over rows);
this file only compiles it with gcc and marshals numpy arrays through ctypes.

The NVFP4 variant (App. B.1's Blackwell format) has its own entry points with the suffix
``_nvfp4``: E2M1 codes (one 4-bit code per uint8), E4M3 block scales (uint8 bits, one per 16
consecutive K entries) and one float32 scale per weight tensor.

Smoothing and the block Hadamard rotation in front of the layer (Sec. 3 Eq. (pair)):
``rotate_weights`` / ``rotate_acts`` / ``fwht_cols`` form W~ = H diag(s) W and x~ = H diag(s)^-1 x
in float64 (the block fast Walsh-Hadamard transform of ``qo_block_fwht``), the ``*_f64`` entry
points run the pack and the activation path on those float64 values, and ``forward_rotated`` /
``forward_rotated_nvfp4`` chain them.  The offline choice of what to protect is in ``subspace``.

Every function returns semantic arrays in the paper's row-major notation:
X [M,K] tokens, W [K,N], U [K,r] (the paper's V), codes as int8 in [-7, 7], activation scales
[M, K/G] (bfloat16 values held in float32), weight scales bfloat16 bits [K/G, N], branch factors
float16.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "qwam_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "libqwam_oracle.so")
_lib = None
_lock = threading.Lock()


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (-O2 -fopenmp -ffp-contract=off); returns the .so path."""
    os.makedirs(_BUILD, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fopenmp", "-ffp-contract=off", "-fno-fast-math",
           "-fPIC", "-shared", _SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            P = ctypes.c_void_p
            I = ctypes.c_int
            lib.qo_pack.argtypes = [P, P, I, I, I, I, P, P, P, P, P]
            lib.qo_quantize_act.argtypes = [P, P, I, I, I, I, P, P, P, P, P]
            lib.qo_quantize_residual_f32.argtypes = [P, I, I, I, P, P]
            lib.qo_linear.argtypes = [P, P, P, P, P, P, I, I, I, I, I, P]
            lib.qo_linear_split_exact.argtypes = [P, P, P, P, I, I, I, I, P]
            lib.qo_f16_bits_rn.argtypes = [ctypes.c_double]
            lib.qo_f16_bits_rn.restype = ctypes.c_uint16
            lib.qo_f16_value.argtypes = [ctypes.c_uint16]
            lib.qo_f16_value.restype = ctypes.c_double
            lib.qo_nearest_code.argtypes = [ctypes.c_double, ctypes.c_double]
            lib.qo_nearest_code.restype = ctypes.c_int
            lib.qo_bf16_bits_div7_rn.argtypes = [ctypes.c_double]
            lib.qo_bf16_bits_div7_rn.restype = ctypes.c_uint16
            lib.qo_pack_nvfp4.argtypes = [P, P, I, I, I, P, P, P, P]
            lib.qo_quantize_act_nvfp4.argtypes = [P, P, I, I, I, P, P, P]
            lib.qo_pack_nvfp4_f64.argtypes = [P, P, I, I, I, P, P, P, P]
            lib.qo_quantize_act_nvfp4_f64.argtypes = [P, P, I, I, I, P, P, P]
            lib.qo_quantize_residual_nvfp4_f32.argtypes = [P, I, I, P, P]
            lib.qo_linear_nvfp4.argtypes = [P, P, P, P, P, ctypes.c_float, P, I, I, I, I, P]
            lib.qo_e2m1_value.argtypes = [I]
            lib.qo_e2m1_value.restype = ctypes.c_double
            lib.qo_e2m1_code_rn.argtypes = [ctypes.c_double]
            lib.qo_e2m1_code_rn.restype = I
            lib.qo_e4m3_value.argtypes = [ctypes.c_uint8]
            lib.qo_e4m3_value.restype = ctypes.c_double
            lib.qo_e4m3_bits_rn.argtypes = [ctypes.c_double]
            lib.qo_e4m3_bits_rn.restype = ctypes.c_uint8
            lib.qo_pack_f64.argtypes = [P, P, I, I, I, I, P, P, P, P, P]
            lib.qo_quantize_act_f64.argtypes = [P, P, I, I, I, I, P, P, P, P, P]
            lib.qo_block_fwht.argtypes = [P, I, I, ctypes.c_long, ctypes.c_long, P, I]
            _lib = lib
    return _lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


class OracleError(RuntimeError):
    pass


def _check(rc, what):
    if rc != 0:
        raise OracleError(f"{what}: oracle status {rc} ({'range' if rc == -2 else 'invalid argument'})")


def pack(W_bf16_bits, U, G, want_float64=False):
    """Offline packing (Sec. 4.2 Eq. (asp) and the W_perp derivation; Eq. (quant) on weights).

    W_bf16_bits: uint16 [K,N]; U: float32 [K,r] (r may be 0).
    Returns dict(qw int8 [N,K], sw uint16 bf16-bits [K/G,N], Bh uint16 fp16-bits [r,N],
    and Bf / Wperp float64 when want_float64)."""
    W = _c(W_bf16_bits, np.uint16)
    K, N = W.shape
    U = _c(U, np.float32).reshape(K, -1)
    r = U.shape[1]
    qw = np.empty((N, K), np.int8)
    sw = np.empty((K // G, N), np.uint16)
    Bh = np.empty((r, N), np.uint16)
    Bf = np.empty((r, N), np.float64) if want_float64 else None
    Wp = np.empty((K, N), np.float64) if want_float64 else None
    _check(_load().qo_pack(_ptr(W), _ptr(U), K, N, r, G, _ptr(qw), _ptr(sw), _ptr(Bh), _ptr(Bf), _ptr(Wp)),
           "pack")
    out = dict(qw=qw, sw=sw, Bh=Bh)
    if want_float64:
        out.update(Bf=Bf, Wperp=Wp)
    return out


def quantize_act(X_bf16_bits, U, G, want_float64=False):
    """Run-time activation path (Eq. (xsplit), then Eq. (quant) per token and group).

    Returns dict(qx int8 [M,K], sx float32 [M,K/G] (bfloat16 values), ph uint16 fp16-bits [M,r],
    and p / Xperp float64 when want_float64)."""
    X = _c(X_bf16_bits, np.uint16)
    M, K = X.shape
    U = _c(U, np.float32).reshape(K, -1)
    r = U.shape[1]
    qx = np.empty((M, K), np.int8)
    sx = np.empty((M, K // G), np.float32)
    ph = np.empty((M, r), np.uint16)
    p = np.empty((M, r), np.float64) if want_float64 else None
    Xp = np.empty((M, K), np.float64) if want_float64 else None
    _check(_load().qo_quantize_act(_ptr(X), _ptr(U), M, K, r, G, _ptr(qx), _ptr(sx), _ptr(ph), _ptr(p), _ptr(Xp)),
           "quantize_act")
    out = dict(qx=qx, sx=sx, ph=ph)
    if want_float64:
        out.update(p=p, Xperp=Xp)
    return out


def pack_f64(W, U, G, want_float64=False):
    """pack() of a float64 weight W [K,N] (the smoothed and rotated W~ of Sec. 3 Eq. (pair))."""
    W = _c(W, np.float64)
    K, N = W.shape
    U = _c(U, np.float32).reshape(K, -1)
    r = U.shape[1]
    qw = np.empty((N, K), np.int8)
    sw = np.empty((K // G, N), np.uint16)
    Bh = np.empty((r, N), np.uint16)
    Bf = np.empty((r, N), np.float64) if want_float64 else None
    Wp = np.empty((K, N), np.float64) if want_float64 else None
    _check(_load().qo_pack_f64(_ptr(W), _ptr(U), K, N, r, G, _ptr(qw), _ptr(sw), _ptr(Bh), _ptr(Bf), _ptr(Wp)),
           "pack_f64")
    out = dict(qw=qw, sw=sw, Bh=Bh)
    if want_float64:
        out.update(Bf=Bf, Wperp=Wp)
    return out


def quantize_act_f64(X, U, G, want_float64=False):
    """quantize_act() of float64 activations X [M,K] (the smoothed and rotated x~)."""
    X = _c(X, np.float64)
    M, K = X.shape
    U = _c(U, np.float32).reshape(K, -1)
    r = U.shape[1]
    qx = np.empty((M, K), np.int8)
    sx = np.empty((M, K // G), np.float32)
    ph = np.empty((M, r), np.uint16)
    p = np.empty((M, r), np.float64) if want_float64 else None
    Xp = np.empty((M, K), np.float64) if want_float64 else None
    _check(_load().qo_quantize_act_f64(_ptr(X), _ptr(U), M, K, r, G, _ptr(qx), _ptr(sx), _ptr(ph), _ptr(p), _ptr(Xp)),
           "quantize_act_f64")
    out = dict(qx=qx, sx=sx, ph=ph)
    if want_float64:
        out.update(p=p, Xperp=Xp)
    return out


def fwht_cols(A, s=None):
    """H diag(s) A for a float64 A [K,n] (the transform of rotate_weights on any float64 input)."""
    A = np.array(A, np.float64, order="C", copy=True)
    K, n = A.shape
    sc = None if s is None else _c(s, np.float64)
    _check(_load().qo_block_fwht(_ptr(A), n, K, 1, n, _ptr(sc), 0), "block_fwht")
    return A


def rotate_weights(W_bf16_bits, s=None):
    """Sec. 3 Eq. (pair), weight side: W~ = H diag(s) W in float64 ([K,N]; H along K by the block
    fast Walsh-Hadamard transform of App. B.1, in a fixed butterfly order)."""
    W = bf16_bits_to_f64(W_bf16_bits)
    K, N = W.shape
    sc = None if s is None else _c(s, np.float64)
    _check(_load().qo_block_fwht(_ptr(W), N, K, 1, N, _ptr(sc), 0), "block_fwht")
    return W


def rotate_acts(X_bf16_bits, s=None):
    """Sec. 3 Eq. (pair), activation side: x~ = H diag(s)^-1 x for every token row, float64 [M,K]."""
    X = bf16_bits_to_f64(X_bf16_bits)
    M, K = X.shape
    sc = None if s is None else _c(s, np.float64)
    _check(_load().qo_block_fwht(_ptr(X), M, K, K, 1, _ptr(sc), 1), "block_fwht")
    return X


def forward_rotated(X_bf16_bits, W_bf16_bits, s, U, G):
    """The layer with smoothing and rotation (Eq. (pair)) in front of ASP: x~ and W~ first, then
    the same pack, activation path and output on them.  U lives in the rotated coordinates."""
    wts = pack_f64(rotate_weights(W_bf16_bits, s), U, G)
    act = quantize_act_f64(rotate_acts(X_bf16_bits, s), U, G)
    return linear(act, wts, G), act, wts


def bf16_bits_to_f64(bits):
    b = _c(bits, np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def quantize_residual(R_f32, G):
    """The quantizer alone on a float32 remainder R [M,K] -> (codes int8 [M,K], scales f32 [M,K/G])."""
    R = _c(R_f32, np.float32)
    M, K = R.shape
    q = np.empty((M, K), np.int8)
    s = np.empty((M, K // G), np.float32)
    _check(_load().qo_quantize_residual_f32(_ptr(R), M, K, G, _ptr(q), _ptr(s)), "quantize_residual")
    return q, s


def linear(act, wts, G):
    """Layer output of Eq. (asp) from codes and scales -> float64 Y [M,N]."""
    qx = _c(act["qx"], np.int8)
    M, K = qx.shape
    qw = _c(wts["qw"], np.int8)
    N = qw.shape[0]
    r = wts["Bh"].shape[0]
    Y = np.empty((M, N), np.float64)
    _check(_load().qo_linear(_ptr(qx), _ptr(_c(act["sx"], np.float32)), _ptr(_c(act["ph"], np.uint16)),
                             _ptr(qw), _ptr(_c(wts["sw"], np.uint16)), _ptr(_c(wts["Bh"], np.uint16)),
                             M, K, N, r, G, _ptr(Y)), "linear")
    return Y


def linear_split_exact(p, Xperp, Bf, Wperp):
    """Eq. (asp) with Q replaced by the identity: p B_f + X_perp W_perp (float64)."""
    p = _c(p, np.float64)
    Xp = _c(Xperp, np.float64)
    Bf = _c(Bf, np.float64)
    Wp = _c(Wperp, np.float64)
    M, K = Xp.shape
    N = Wp.shape[1]
    r = p.shape[1]
    Y = np.empty((M, N), np.float64)
    _check(_load().qo_linear_split_exact(_ptr(p), _ptr(Xp), _ptr(Bf), _ptr(Wp), M, K, N, r, _ptr(Y)),
           "linear_split_exact")
    return Y


def forward(X_bf16_bits, W_bf16_bits, U, G):
    """Whole layer: pack, quantize the activations, output.  Returns (Y, act, wts)."""
    wts = pack(W_bf16_bits, U, G)
    act = quantize_act(X_bf16_bits, U, G)
    return linear(act, wts, G), act, wts


def f16_bits(x: float) -> int:
    return int(_load().qo_f16_bits_rn(float(x)))


def f16_value(h: int) -> float:
    return float(_load().qo_f16_value(int(h)))


def nearest_code(x: float, s: float) -> int:
    return int(_load().qo_nearest_code(float(x), float(s)))


def bf16_bits_div7(a: float) -> int:
    """bfloat16 bits of RN_bf16(a / 7) for the exact quotient (readings R3, R4), a >= 0."""
    return int(_load().qo_bf16_bits_div7_rn(float(a)))


# ---- NVFP4 variant (App. B.1) ----------------------------------------------------------------

FP4_BLOCK = 16


def pack_nvfp4_f64(W, U):
    """pack_nvfp4() of a float64 weight W [K,N] (the smoothed and rotated W~ of Eq. (pair))."""
    W = _c(W, np.float64)
    K, N = W.shape
    U = _c(U, np.float32).reshape(K, -1)
    r = U.shape[1]
    qw = np.empty((N, K), np.uint8)
    sfw = np.empty((N, K // FP4_BLOCK), np.uint8)
    sg = ctypes.c_float(0.0)
    Bh = np.empty((r, N), np.uint16)
    _check(_load().qo_pack_nvfp4_f64(_ptr(W), _ptr(U), K, N, r, _ptr(qw), _ptr(sfw), ctypes.byref(sg), _ptr(Bh)),
           "pack_nvfp4_f64")
    return dict(qw=qw, sfw=sfw, sg=np.float32(sg.value), Bh=Bh)


def quantize_act_nvfp4_f64(X, U):
    """quantize_act_nvfp4() of float64 activations X [M,K] (the smoothed and rotated x~)."""
    X = _c(X, np.float64)
    M, K = X.shape
    U = _c(U, np.float32).reshape(K, -1)
    r = U.shape[1]
    qx = np.empty((M, K), np.uint8)
    sfx = np.empty((M, K // FP4_BLOCK), np.uint8)
    ph = np.empty((M, r), np.uint16)
    _check(_load().qo_quantize_act_nvfp4_f64(_ptr(X), _ptr(U), M, K, r, _ptr(qx), _ptr(sfx), _ptr(ph)),
           "quantize_act_nvfp4_f64")
    return dict(qx=qx, sfx=sfx, ph=ph)


def forward_rotated_nvfp4(X_bf16_bits, W_bf16_bits, s, U):
    """The NVFP4 layer on x~ and W~ (Eq. (pair)).  Returns (Y, act, wts)."""
    wts = pack_nvfp4_f64(rotate_weights(W_bf16_bits, s), U)
    act = quantize_act_nvfp4_f64(rotate_acts(X_bf16_bits, s), U)
    return linear_nvfp4(act, wts), act, wts


def pack_nvfp4(W_bf16_bits, U):
    """Offline packing of the NVFP4 variant (readings N1, N2, N4 of qwam_oracle.c).

    Returns dict(qw uint8 E2M1 codes [N,K], sfw uint8 E4M3 bits [N,K/16], sg float32,
    Bh uint16 fp16-bits [r,N])."""
    W = _c(W_bf16_bits, np.uint16)
    K, N = W.shape
    U = _c(U, np.float32).reshape(K, -1)
    r = U.shape[1]
    qw = np.empty((N, K), np.uint8)
    sfw = np.empty((N, K // FP4_BLOCK), np.uint8)
    sg = ctypes.c_float(0.0)
    Bh = np.empty((r, N), np.uint16)
    _check(_load().qo_pack_nvfp4(_ptr(W), _ptr(U), K, N, r, _ptr(qw), _ptr(sfw), ctypes.byref(sg), _ptr(Bh)),
           "pack_nvfp4")
    return dict(qw=qw, sfw=sfw, sg=np.float32(sg.value), Bh=Bh)


def quantize_act_nvfp4(X_bf16_bits, U):
    """Activation path of the NVFP4 variant (Eq. (xsplit), reading N3).

    Returns dict(qx uint8 E2M1 codes [M,K], sfx uint8 E4M3 bits [M,K/16], ph uint16 [M,r])."""
    X = _c(X_bf16_bits, np.uint16)
    M, K = X.shape
    U = _c(U, np.float32).reshape(K, -1)
    r = U.shape[1]
    qx = np.empty((M, K), np.uint8)
    sfx = np.empty((M, K // FP4_BLOCK), np.uint8)
    ph = np.empty((M, r), np.uint16)
    _check(_load().qo_quantize_act_nvfp4(_ptr(X), _ptr(U), M, K, r, _ptr(qx), _ptr(sfx), _ptr(ph)),
           "quantize_act_nvfp4")
    return dict(qx=qx, sfx=sfx, ph=ph)


def quantize_residual_nvfp4(R_f32):
    """Reading N3 alone on a float32 remainder R [M,K] -> (codes uint8 [M,K], E4M3 bits [M,K/16])."""
    R = _c(R_f32, np.float32)
    M, K = R.shape
    q = np.empty((M, K), np.uint8)
    sf = np.empty((M, K // FP4_BLOCK), np.uint8)
    _check(_load().qo_quantize_residual_nvfp4_f32(_ptr(R), M, K, _ptr(q), _ptr(sf)), "quantize_residual_nvfp4")
    return q, sf


def linear_nvfp4(act, wts):
    """Layer output of the NVFP4 variant (reading N5) -> float64 Y [M,N]."""
    qx = _c(act["qx"], np.uint8)
    M, K = qx.shape
    qw = _c(wts["qw"], np.uint8)
    N = qw.shape[0]
    r = wts["Bh"].shape[0]
    Y = np.empty((M, N), np.float64)
    _check(_load().qo_linear_nvfp4(_ptr(qx), _ptr(_c(act["sfx"], np.uint8)), _ptr(_c(act["ph"], np.uint16)),
                                   _ptr(qw), _ptr(_c(wts["sfw"], np.uint8)), float(wts["sg"]),
                                   _ptr(_c(wts["Bh"], np.uint16)), M, K, N, r, _ptr(Y)), "linear_nvfp4")
    return Y


def forward_nvfp4(X_bf16_bits, W_bf16_bits, U):
    """Whole NVFP4 layer: pack, quantize the activations, output.  Returns (Y, act, wts)."""
    wts = pack_nvfp4(W_bf16_bits, U)
    act = quantize_act_nvfp4(X_bf16_bits, U)
    return linear_nvfp4(act, wts), act, wts


def e2m1_value(c: int) -> float:
    return float(_load().qo_e2m1_value(int(c)))


def e2m1_code(x: float) -> int:
    return int(_load().qo_e2m1_code_rn(float(x)))


def e4m3_value(b: int) -> float:
    return float(_load().qo_e4m3_value(int(b)))


def e4m3_bits(x: float) -> int:
    return int(_load().qo_e4m3_bits_rn(float(x)))
