"""Shared helpers of the GPU parity tests: seeded inputs on both sides, workspace read-back,
nibble unpacking and the comparison rules."""
from __future__ import annotations

import math

import numpy as np
import torch

import oracle
from paper_2609_33269_gb300 import asp
from paper_2609_33269_gb300 import workloads as wl


def to_dev_bf16(bits: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).cuda().view(torch.bfloat16)


def decode_ob4(packed: np.ndarray) -> np.ndarray:
    """INT4 codes packed as OB4 words, uint8 [R, K/2] -> int8 [R, K].

    Word j of a row (little-endian 32 bits) holds k = 8j..8j+7 as offset-binary nibbles c + 8:
    code 8j + 2p in bits 4p..4p+3 and code 8j + 2p + 1 in bits 16 + 4p..16 + 4p + 3."""
    p = np.ascontiguousarray(packed, np.uint8)
    w = p.view("<u4")
    out = np.empty((p.shape[0], w.shape[1], 8), np.int8)
    for q in range(4):
        out[:, :, 2 * q] = ((w >> (4 * q)) & 0xF).astype(np.int16) - 8
        out[:, :, 2 * q + 1] = ((w >> (16 + 4 * q)) & 0xF).astype(np.int16) - 8
    return out.reshape(p.shape[0], -1)


def unpack_nibbles(packed: np.ndarray) -> np.ndarray:
    """uint8 [R, K/2] -> int8 [R, K] (low nibble = even k, two's complement)."""
    p = np.ascontiguousarray(packed)
    lo = (p & 0xF).astype(np.int16)
    hi = (p >> 4).astype(np.int16)
    out = np.empty((p.shape[0], p.shape[1] * 2), np.int16)
    out[:, 0::2] = lo
    out[:, 1::2] = hi
    return ((out ^ 8) - 8).astype(np.int8)


class Case:
    """One layer on both sides: host inputs, the packed GPU layer, oracle outputs on demand."""

    def __init__(self, M, K, N, r, G=64, seed=0, layer_id=0, dist="outlier", n_outlier=None, Xb=None,
                 rotate=False, s=None):
        """rotate=True: the layer with smoothing factors s (float64 [K] or None) and the block
        Hadamard rotation in front (Eq. (pair)); U is then a basis of the rotated coordinates."""
        self.M, self.K, self.N, self.r, self.G = M, K, N, r, G
        self.Xb = (wl.activations(M, K, seed=seed, layer_id=layer_id, dist=dist, n_outlier=n_outlier)
                   if Xb is None else np.ascontiguousarray(Xb, np.uint16))
        self.Wb = wl.weight(K, N, seed=seed, layer_id=layer_id)
        self.U = wl.basis(K, r, seed=seed, layer_id=layer_id)
        self.X = to_dev_bf16(self.Xb)
        self.W = to_dev_bf16(self.Wb)
        self.Ud = torch.from_numpy(self.U).cuda() if r > 0 else None
        self.rotate, self.s = rotate, s
        sd = torch.from_numpy(np.asarray(s, np.float32)).cuda() if s is not None else None
        self.layer = asp.AspLinear(self.W, self.Ud, G, rotate=rotate, s=sd)
        self._ow = None

    # oracle side
    def s64(self):
        """The smoothing factors as the GPU holds them (float32), widened for the oracle."""
        return None if self.s is None else np.asarray(self.s, np.float32).astype(np.float64)

    def oracle_weights(self):
        if self._ow is None:
            if self.rotate:
                self._ow = oracle.pack_f64(oracle.rotate_weights(self.Wb, self.s64()), self.U, self.G)
            else:
                self._ow = oracle.pack(self.Wb, self.U, self.G)
        return self._ow

    def oracle_act(self, rows=None, want_float64=True):
        Xb = self.Xb if rows is None else self.Xb[rows]
        if self.rotate:
            return oracle.quantize_act_f64(oracle.rotate_acts(Xb, self.s64()), self.U, self.G,
                                           want_float64=want_float64)
        return oracle.quantize_act(Xb, self.U, self.G, want_float64=want_float64)

    # GPU side
    def gpu_weights(self):
        e = asp.qwam_asp_export(self.layer.h)
        return dict(qw=unpack_nibbles(e["qw"]), sw=e["sw"], Bh=e["Bh"][:, :self.r].T.copy(), Uhl=e["Uhl"])

    def gpu_act(self, rows=None):
        codes, scales, ph = self.layer.act_views(self.M)
        torch.cuda.synchronize()
        qx = decode_ob4(codes.cpu().numpy())
        sx = scales.float().cpu().numpy()[:, :self.M].T.copy()
        phv = ph.cpu().numpy().view(np.uint16)[:, :self.r].copy()
        if rows is not None:
            qx, sx, phv = qx[rows], sx[rows], phv[rows]
        return dict(qx=qx, sx=sx, ph=phv)

    def run(self, fp32=True):
        Y = self.layer(self.X, fp32=fp32)
        torch.cuda.synchronize()
        return Y

    def residual(self):
        R = torch.empty((self.M, self.K), dtype=torch.float32, device="cuda")
        ws = self.layer.workspace(self.M)
        asp.qwam_asp_debug_residual(self.X, self.M, self.layer.h, ws, R)
        torch.cuda.synchronize()
        return R.cpu().numpy()

    def close(self):
        self.layer.close()


def rowwise_rel_err(Y, ref):
    """max |Y - ref| / max |ref| per row."""
    d = np.abs(np.asarray(Y, np.float64) - ref).max(axis=1)
    n = np.abs(ref).max(axis=1)
    return d / np.maximum(n, 1e-30)


def gemm_tol(K, r_pad=0):
    """Bound on max |Y - Yk| / max |Yk| per row, Yk the oracle's output on the kernel's own codes,
    scales and branch inputs.  The kernel forms every product exactly (float16 x float16) and adds
    the K + r_pad of them into one float32 accumulator, 16 per MMA step; a rounding of 2^-24 of the
    running sum per step grows like sqrt((K + r_pad) / 16) 2^-24 times the sum's scale, and
    4e-7 sqrt(K + r_pad) is about four times the largest error measured (K = 12288)."""
    return max(1e-5, 4e-7 * math.sqrt(K + r_pad))


def near_tie_mismatches(q_gpu, q_ref, x_ref, s_ref, G, eps_rel):
    """Indices where the codes differ, and whether each lies within eps (relative to the scale)
    of a rounding boundary of the reference remainder x_ref / s_ref."""
    bad = np.argwhere(q_gpu != q_ref)
    ok = []
    for m, k in bad:
        s = float(s_ref[m, k // G])
        t = abs(float(x_ref[m, k]) / s) if s > 0 else 0.0
        ok.append(abs((t - np.floor(t)) - 0.5) <= eps_rel)
    return bad, np.array(ok, bool)


def _bf16_bits(v):
    return int(np.float32(v).view(np.uint32)) >> 16


def check_int4_act(ga, oa, G):
    """INT4 activation codes and scales at r > 0 against the oracle's (readings R2, R3, R5), with
    oa the oracle's float64 path (Xperp and p).  The kernel's float32 remainder is within
    2e-5 max|x| of the oracle's (asserted by the residual tests), and max|x| <= max|Xperp| + |p|.

    * A scale may differ only by one bfloat16 step, and only where the oracle's amax / 7 lies
      within that remainder error (over 7) of the midpoint between the two values.
    * A code in a group whose scale agrees may differ only within 1e-3 (relative to the scale) of
      a rounding boundary of the oracle's quotient; codes of a group whose scale differs follow
      that scale (the quantizer on the kernel's own remainder is checked bit for bit elsewhere).
    * At most max(2, 1e-2 groups) scales and max(2, 1e-4 codes) codes differ.
    Returns a bool per row: any code or scale of the row differs."""
    Xp = np.asarray(oa["Xperp"], np.float64)
    M, K = Xp.shape
    pn = np.linalg.norm(oa["p"], axis=1) if oa["p"].size else np.zeros(M)
    delta = 2e-5 * (np.abs(Xp).max(axis=1) + pn)
    amax = np.abs(Xp).reshape(M, K // G, G).max(axis=2)
    sg, so = np.asarray(ga["sx"], np.float32), np.asarray(oa["sx"], np.float32)
    sdiff = sg != so
    sbad = np.argwhere(sdiff)
    for m, g in sbad:
        bg, bo = _bf16_bits(sg[m, g]), _bf16_bits(so[m, g])
        assert abs(int(bg) - int(bo)) == 1, (m, g, sg[m, g], so[m, g])
        mid = (float(sg[m, g]) + float(so[m, g])) / 2
        assert abs(amax[m, g] / 7 - mid) <= delta[m] / 7, (m, g, amax[m, g] / 7, mid, delta[m])
    assert len(sbad) <= max(2, 1e-2 * sg.size), len(sbad)
    same = np.repeat(~sdiff, G, axis=1)
    qbad, qnear = near_tie_mismatches(np.where(same, ga["qx"], 0), np.where(same, oa["qx"], 0), Xp,
                                      oa["sx"], G, 1e-3)
    assert qnear.all(), qbad[~qnear][:5]
    assert len(qbad) <= max(2, 1e-4 * ga["qx"].size), len(qbad)
    return np.any(ga["qx"] != oa["qx"], axis=1) | np.any(sdiff, axis=1)


def check_layer_output(Y, Yo, Yk, flip, tol_k=1e-5):
    """Rows whose activation codes and scales all equal the oracle's meet max |dY| <= 1e-3 |y|inf
    against the oracle.  A row holding a near-tie flip (checked separately) differs from the
    oracle by that flip's weight column times s_x s_w, which can exceed 1e-3 in an outlier group;
    such a row must equal the oracle evaluated on the kernel's own codes (tol_k, see gemm_tol)."""
    flip = np.asarray(flip, bool)
    e = rowwise_rel_err(Y, Yo)
    if (~flip).any():
        assert e[~flip].max() <= 1e-3, e[~flip].max()
    if flip.any():
        assert rowwise_rel_err(Y[flip], Yk[flip]).max() <= tol_k
    assert flip.mean() <= 0.05, flip.mean()


E2M1_MIDPOINTS = np.array([0.25, 0.75, 1.25, 1.75, 2.5, 3.5, 5.0])
_E4M3_POSITIVE = None


def e4m3_positive_values():
    """Values of the E4M3 codes 0..126 (the non-negative finite ones), from the oracle."""
    global _E4M3_POSITIVE
    if _E4M3_POSITIVE is None:
        _E4M3_POSITIVE = np.array([oracle.e4m3_value(b) for b in range(127)])
    return _E4M3_POSITIVE


def nvfp4_mismatches(qx_gpu, sfx_gpu, qx_ref, sfx_ref, Xperp, eps=1e-3):
    """NVFP4 activation codes and block scales against the oracle's (reading N3: per block of 16,
    s = RN_e4m3(amax / 6) and code = RN_e2m1(x / s)), with Xperp the oracle's float64 remainder.

    A block scale may differ only where amax / 6 lies within eps (relative) of a midpoint between
    two E4M3 values; a code in a block whose scale agrees may differ only where |x| / s lies within
    eps of an E2M1 midpoint.  Codes in a block whose scale differs follow that scale and are not
    counted again.  Returns (number of mismatches, whether each is such a near tie)."""
    M, K = qx_ref.shape
    nb = K // 16
    tab = e4m3_positive_values()
    mids = (tab[1:] + tab[:-1]) / 2
    t = np.abs(np.asarray(Xperp, np.float64)).reshape(M, nb, 16).max(axis=2) / 6.0
    near = []
    sbad = np.argwhere(sfx_gpu != sfx_ref)
    for m, b in sbad:
        near.append(np.abs(mids - t[m, b]).min() <= eps * t[m, b])
    cbad = np.argwhere((qx_gpu != qx_ref) & np.repeat(sfx_gpu == sfx_ref, 16, axis=1))
    for m, k in cbad:
        s = tab[int(sfx_ref[m, k // 16])]
        near.append(s > 0 and np.abs(E2M1_MIDPOINTS - abs(float(Xperp[m, k])) / s).min() <= eps)
    return len(sbad) + len(cbad), np.array(near, bool)


def check_nvfp4_activations(ga, oa, Xperp, R, Xin):
    """The NVFP4 activation bar at r > 0: every differing code or block scale is a near tie, at
    most max(2, 1e-4 * codes) differ, and the kernel's float32 remainder R is within 2e-5 of the
    float64 one per row (relative to the row's largest input value Xin)."""
    err = np.abs(R - Xperp).max(axis=1) / np.maximum(np.abs(Xin).max(axis=1), 1e-30)
    assert err.max() <= 2e-5, err.max()
    n_bad, near = nvfp4_mismatches(ga["qx"], ga["sfx"], oa["qx"], oa["sfx"], Xperp)
    assert near.all(), (n_bad, near)
    assert n_bad <= max(2, 1e-4 * ga["qx"].size), n_bad
    return n_bad


def unpack_e2m1(packed):
    """uint8 [R, K/2] -> E2M1 codes uint8 [R, K], low nibble = even k."""
    p = np.ascontiguousarray(packed)
    out = np.empty((p.shape[0], p.shape[1] * 2), np.uint8)
    out[:, 0::2] = p & 0xF
    out[:, 1::2] = p >> 4
    return out


def atoms_to_rows(atoms, rows, K):
    """Scale atoms (512 bytes per 128 rows x 64 K; row r's four scales at (r % 32) * 16 +
    (r % 128 // 32) * 4) -> row-major uint8 [rows, K/16]."""
    a = np.asarray(atoms, np.uint8)
    r = np.arange(rows)[:, None]
    b = np.arange(K // 16)[None, :]
    idx = ((r // 128) * (K // 64) + b // 4) * 512 + (r % 32) * 16 + ((r % 128) // 32) * 4 + b % 4
    return a[idx]


class NvCase:
    def __init__(self, M, K, N, r, seed=0, layer_id=0, dist="outlier"):
        self.M, self.K, self.N, self.r = M, K, N, r
        self.Xb = wl.activations(M, K, seed=seed, layer_id=layer_id, dist=dist)
        self.Wb = wl.weight(K, N, seed=seed, layer_id=layer_id)
        self.U = wl.basis(K, r, seed=seed, layer_id=layer_id)
        self.X = to_dev_bf16(self.Xb)
        W = to_dev_bf16(self.Wb)
        Ud = torch.from_numpy(self.U).cuda() if r > 0 else None
        self.layer = asp.AspLinear(W, Ud, fmt=asp.QWAM_FMT_NVFP4)
        self._ow = None

    def oracle_weights(self):
        if self._ow is None:
            self._ow = oracle.pack_nvfp4(self.Wb, self.U)
        return self._ow

    def gpu_weights(self):
        e = asp.qwam_asp_export_nvfp4(self.layer.h)
        return dict(qw=unpack_e2m1(e["qw"]), sfw=e["sfw"], sg=e["sg"], Bh=e["Bh"][:, :self.r].T.copy())

    def gpu_act(self):
        codes, atoms, ph = self.layer.act_views_nvfp4(self.M)
        torch.cuda.synchronize()
        return dict(qx=unpack_e2m1(codes.cpu().numpy()),
                    sfx=atoms_to_rows(atoms.cpu().numpy(), self.M, self.K),
                    ph=ph.cpu().numpy().view(np.uint16)[:, :self.r].copy())

    def residual(self):
        R = torch.empty((self.M, self.K), dtype=torch.float32, device="cuda")
        asp.qwam_asp_debug_residual(self.X, self.M, self.layer.h, self.layer.workspace(self.M), R)
        torch.cuda.synchronize()
        return R.cpu().numpy()

    def run(self, fp32=True):
        Y = self.layer(self.X, fp32=fp32)
        torch.cuda.synchronize()
        return Y

    def close(self):
        self.layer.close()
