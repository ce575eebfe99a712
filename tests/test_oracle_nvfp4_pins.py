"""Pins of the oracle's NVFP4 variant (App. B.1: E2M1 values, an E4M3 scale per 16 elements,
one float32 scale per weight tensor), against definitions written out here independently of the
oracle's C code: the OCP bit layouts decoded from their fields, brute-force nearest-value search
over every code, the quantizer's error bound, the layer as a plain matrix product of the
dequantized operands, and the special cases r = 0 and r = K of Eq. (asp)."""
from __future__ import annotations

import math
from fractions import Fraction

import numpy as np
import pytest

import oracle
from paper_2609_33269_gb300 import workloads as wl


# ---- number formats, decoded from their bit fields ------------------------------------------

def e2m1_from_fields(c: int) -> float:
    """OCP FP4 E2M1: sign bit 3, exponent bits 2..1 (bias 1), mantissa bit 0."""
    s, e, m = (c >> 3) & 1, (c >> 1) & 3, c & 1
    v = m * 0.5 if e == 0 else (1.0 + m / 2.0) * 2.0 ** (e - 1)
    return -v if s else v


def e4m3_from_fields(b: int) -> float:
    """OCP FP8 E4M3 ("FN"): sign bit 7, exponent bits 6..3 (bias 7), mantissa bits 2..0;
    S.1111.111 is NaN, there are no infinities."""
    s, e, m = (b >> 7) & 1, (b >> 3) & 15, b & 7
    if e == 15 and m == 7:
        return math.nan
    v = m * 2.0 ** -9 if e == 0 else (1.0 + m / 8.0) * 2.0 ** (e - 7)
    return -v if s else v


E2M1_POS = [(c, e2m1_from_fields(c)) for c in range(8)]
E4M3_POS = [(b, e4m3_from_fields(b)) for b in range(0x7f)]  # every finite non-negative value


def nearest_even(x: float, table):
    """Brute force: the entry of `table` nearest to |x|, ties to the even code; sign of x kept
    for non-zero results."""
    a = abs(x)
    best = min(table, key=lambda cv: (abs(a - cv[1]), cv[0] & 1))
    return best


def test_e2m1_decode_matches_fields():
    for c in range(16):
        assert oracle.e2m1_value(c) == e2m1_from_fields(c)
    assert [e2m1_from_fields(c) for c in range(8)] == [0, 0.5, 1, 1.5, 2, 3, 4, 6]


def test_e4m3_decode_matches_fields():
    for b in range(256):
        v, ref = oracle.e4m3_value(b), e4m3_from_fields(b)
        assert (math.isnan(v) and math.isnan(ref)) or v == ref, b
    assert e4m3_from_fields(0x7e) == 448.0 and e4m3_from_fields(0x01) == 2.0 ** -9
    assert e4m3_from_fields(0x08) == 2.0 ** -6 and e4m3_from_fields(0x38) == 1.0


def _probe_points(values, rng, n_random):
    """Every grid value, every midpoint (the ties), points just either side of each midpoint and
    random points in between."""
    vals = sorted(set(values))
    pts = list(vals)
    for lo, hi in zip(vals, vals[1:]):
        mid = (lo + hi) / 2
        pts += [mid, np.nextafter(mid, 0.0), np.nextafter(mid, np.inf)]
    pts += list(rng.uniform(0, vals[-1] * 1.1, n_random))
    return pts


def test_e2m1_rounding_is_nearest_ties_even_saturating():
    rng = np.random.default_rng(1)
    for a in _probe_points([v for _, v in E2M1_POS], rng, 4000) + [6.0, 6.5, 7.0, 100.0]:
        for x in (a, -a):
            c = oracle.e2m1_code(x)
            code, val = nearest_even(x, E2M1_POS) if abs(x) < 6.0 else (7, 6.0)
            want = 0 if code == 0 else (code | 8 if x < 0 else code)
            assert c == want, (x, c, want)
    # the ties, spelled out: 0.25->0, 0.75->1, 1.25->1, 1.75->2, 2.5->2, 3.5->4, 5->4
    assert [e2m1_from_fields(oracle.e2m1_code(t)) for t in (0.25, 0.75, 1.25, 1.75, 2.5, 3.5, 5.0)] == \
        [0, 1, 1, 2, 2, 4, 4]


def test_e4m3_rounding_is_nearest_ties_even_saturating():
    rng = np.random.default_rng(2)
    pos = [v for _, v in E4M3_POS]
    pts = _probe_points(pos, rng, 4000) + list(np.exp(rng.uniform(np.log(1e-5), np.log(500.0), 4000)))
    for a in pts + [448.0, 460.0, 470.0, 1e6]:
        b = oracle.e4m3_bits(a)
        want = nearest_even(a, E4M3_POS)[0] if a < 448.0 else 0x7e
        assert b == want, (a, b, want)
        assert oracle.e4m3_bits(-a) == want | 0x80  # the sign is kept, zero included


# ---- the quantizer (reading N3) -------------------------------------------------------------

def _half_gap(u: float) -> float:
    """Half the E2M1 grid spacing around |u|."""
    a = abs(u)
    return 0.25 if a < 2 else (0.5 if a < 4 else 1.0)


def test_activation_quantizer_error_bound_and_scales():
    rng = np.random.default_rng(3)
    R = (rng.standard_normal((16, 256)) * np.exp(rng.uniform(-3, 3, (16, 1)))).astype(np.float32)
    R[0, :16] = 0.0                   # an all-zero block
    R[1, 16:32] = 1e-4                # a block whose scale underflows to an E4M3 subnormal
    q, sf = oracle.quantize_residual_nvfp4(R)
    assert q.max() <= 15 and (q != 8).all()   # zero is always code 0
    for m in range(R.shape[0]):
        for b in range(R.shape[1] // 16):
            blk = R[m, 16 * b:16 * b + 16].astype(np.float64)
            amax = float(np.abs(blk).max())
            t = float(np.float32(amax / 6.0))
            s_bits = nearest_even(t, E4M3_POS)[0] if t < 448 else 0x7e
            assert sf[m, b] == s_bits
            s = e4m3_from_fields(s_bits)
            for k in range(16):
                x = blk[k]
                v = e2m1_from_fields(int(q[m, 16 * b + k]))
                if s == 0:
                    assert v == 0
                    continue
                u = float(np.float32(x / s))
                if abs(u) <= 6.0:
                    assert abs(x - s * v) <= s * _half_gap(u) * (1 + 1e-6), (m, b, k)
                else:  # the scale rounded down and x / s lies beyond the grid: saturated
                    assert v == math.copysign(6.0, x)


def test_weight_pack_r0_brute_force():
    """r = 0: W_perp = W, and every code and scale follows reading N4, recomputed by brute force."""
    K, N = 64, 6
    W = wl.weight(K, N, seed=11, layer_id=0)
    out = oracle.pack_nvfp4(W, np.zeros((K, 0), np.float32))
    Wv = wl.bf16_bits_to_f32(W).astype(np.float64)
    sg = np.float32(np.abs(Wv).max() / (6.0 * 448.0))
    assert out["sg"] == sg
    for n in range(N):
        for b in range(K // 16):
            blk = Wv[16 * b:16 * b + 16, n]
            s_bits = nearest_even(np.abs(blk).max() / (6.0 * float(sg)), E4M3_POS)[0]
            assert out["sfw"][n, b] == s_bits
            scale = e4m3_from_fields(s_bits) * float(sg)
            for k in range(16):
                u = blk[k] / scale
                code, _ = nearest_even(u, E2M1_POS) if abs(u) < 6 else (7, 6.0)
                want = 0 if code == 0 else (code | 8 if u < 0 else code)
                assert out["qw"][n, 16 * b + k] == want


def nearest_even_exact(x: float, s: float, table):
    """Brute force on the exact quotient x / s (rational arithmetic): the entry of `table`
    nearest to |x| / s, ties to the even code."""
    u = abs(Fraction(x)) / Fraction(s)
    return min(table, key=lambda cv: (abs(u - Fraction(cv[1])), cv[0] & 1))


@pytest.mark.parametrize("r", [1, 5])
def test_activation_path_brute_force_on_the_pinned_remainder(r):
    """0 < r < K: the NVFP4 activation path follows reading N3 on the remainder of Eq. (xsplit),
    recomputed here by brute force from the INT4 oracle's float64 remainder (which the exact
    rational test of the INT4 layer pins).  Scales: RN_e4m3 of RN_f32(amax / 6); codes: nearest
    E2M1 value to the exact quotient, ties to even, saturating at 6."""
    M, K = 6, 128
    X = wl.activations(M, K, seed=81, layer_id=r, dist="outlier", n_outlier=3)
    U = wl.basis(K, r, seed=81, layer_id=r)
    Xp = oracle.quantize_act(X, U, 64, want_float64=True)["Xperp"]
    out = oracle.quantize_act_nvfp4(X, U)
    for m in range(M):
        for b in range(K // 16):
            blk = Xp[m, 16 * b:16 * b + 16]
            t = float(np.float32(np.abs(blk).max() / 6.0))
            s_bits = nearest_even(t, E4M3_POS)[0] if t < 448 else 0x7e
            assert out["sfx"][m, b] == s_bits, (m, b)
            s = e4m3_from_fields(s_bits)
            for k in range(16):
                x = float(blk[k])
                code = 0 if s == 0 else (7 if abs(Fraction(x)) / Fraction(s) >= 6 else
                                         nearest_even_exact(x, s, E2M1_POS)[0])
                want = 0 if code == 0 else (code | 8 if x < 0 else code)
                assert out["qx"][m, 16 * b + k] == want, (m, b, k)


@pytest.mark.parametrize("r", [1, 5])
def test_weight_pack_brute_force_on_the_pinned_deflated_weight(r):
    """0 < r < K: every code and scale of the NVFP4 pack follows reading N4 on W_perp, recomputed by
    brute force from the INT4 oracle's float64 W_perp (pinned by the exact rational test)."""
    K, N = 128, 6
    W = wl.weight(K, N, seed=82, layer_id=r)
    U = wl.basis(K, r, seed=82, layer_id=r)
    Wp = oracle.pack(W, U, 64, want_float64=True)["Wperp"]
    out = oracle.pack_nvfp4(W, U)
    sg = np.float32(np.abs(Wp).max() / (6.0 * 448.0))
    assert out["sg"] == sg
    for n in range(N):
        for b in range(K // 16):
            blk = Wp[16 * b:16 * b + 16, n]
            s_bits = nearest_even(np.abs(blk).max() / (6.0 * float(sg)), E4M3_POS)[0]
            assert out["sfw"][n, b] == s_bits, (n, b)
            scale = e4m3_from_fields(s_bits) * float(sg)
            for k in range(16):
                u = blk[k] / scale
                code, _ = nearest_even(u, E2M1_POS) if abs(u) < 6 else (7, 6.0)
                want = 0 if code == 0 else (code | 8 if u < 0 else code)
                assert out["qw"][n, 16 * b + k] == want, (n, b, k)


def test_activation_quantizer_rounds_the_exact_quotient():
    """A float64 remainder just above or below an E2M1 midpoint product m * s rounds by its exact
    quotient (a float32 rounding of x / s would land on the midpoint and go to the even code)."""
    s_bits = 0x38  # s = 1
    for mid, lo_code, hi_code in ((0.25, 0, 1), (0.75, 1, 2), (1.25, 2, 3), (2.5, 4, 5), (5.0, 6, 7)):
        R = np.zeros((1, 16), np.float64)
        R[0, 0] = 6.0  # amax 6 -> s = 1 exactly
        R[0, 1] = mid * (1 + 2.0 ** -40)
        R[0, 2] = mid * (1 - 2.0 ** -40)
        R[0, 3] = mid
        q = oracle.quantize_act_nvfp4_f64(R, np.zeros((16, 0), np.float32))
        assert q["sfx"][0, 0] == s_bits
        tie = lo_code if lo_code % 2 == 0 else hi_code
        assert list(q["qx"][0, 1:4]) == [hi_code, lo_code, tie], mid


# ---- the layer (reading N5) -----------------------------------------------------------------

def _deq(codes, sf):
    vals = np.array([e2m1_from_fields(c) for c in range(16)])
    scales = np.array([e4m3_from_fields(b) for b in range(256)])
    return vals[codes] * np.repeat(scales[sf], 16, axis=1)


def _f16(bits):
    return bits.astype(np.uint16).view(np.float16).astype(np.float64)


@pytest.mark.parametrize("r", [0, 5])
def test_layer_equals_matrix_product_of_dequantized_operands(r):
    M, K, N = 7, 96, 10
    X = wl.activations(M, K, seed=21, layer_id=1)
    W = wl.weight(K, N, seed=21, layer_id=1)
    U = wl.basis(K, r, seed=21, layer_id=1) if r else np.zeros((K, 0), np.float32)
    Y, act, wts = oracle.forward_nvfp4(X, W, U)
    ref = float(wts["sg"]) * (_deq(act["qx"], act["sfx"]) @ _deq(wts["qw"], wts["sfw"]).T)
    if r:
        ref = ref + _f16(act["ph"]) @ _f16(wts["Bh"])
    np.testing.assert_allclose(Y, ref, rtol=1e-12, atol=1e-12 * np.abs(ref).max())


def test_full_rank_protection_gives_the_16_bit_product():
    """r = K: x_perp = 0 and W_perp = 0 up to rounding, so Y is the branch alone, i.e. the
    16-bit product X W within the fp16 rounding of p and B."""
    M, K, N = 6, 64, 12
    X = wl.activations(M, K, seed=31, layer_id=2)
    W = wl.weight(K, N, seed=31, layer_id=2)
    U = wl.basis(K, K, seed=31, layer_id=2)
    Y, _, _ = oracle.forward_nvfp4(X, W, U)
    exact = wl.bf16_bits_to_f32(X).astype(np.float64) @ wl.bf16_bits_to_f32(W).astype(np.float64)
    err = np.abs(Y - exact).max(axis=1) / np.abs(exact).max(axis=1)
    assert err.max() <= 1e-3


def test_nvfp4_layer_is_a_4_bit_approximation_of_xw():
    """Loose: on Gaussian inputs the NVFP4 output is within a few percent of X W (row-wise,
    relative to the row's largest entry), and protecting r directions does not make it worse."""
    M, K, N = 32, 256, 64
    X = wl.activations(M, K, seed=41, layer_id=3)
    W = wl.weight(K, N, seed=41, layer_id=3)
    exact = wl.bf16_bits_to_f32(X).astype(np.float64) @ wl.bf16_bits_to_f32(W).astype(np.float64)
    Y0, _, _ = oracle.forward_nvfp4(X, W, np.zeros((K, 0), np.float32))
    Y1, _, _ = oracle.forward_nvfp4(X, W, wl.basis(K, 16, seed=41, layer_id=3))
    e0 = (np.abs(Y0 - exact).max(axis=1) / np.abs(exact).max(axis=1)).mean()
    e1 = (np.abs(Y1 - exact).max(axis=1) / np.abs(exact).max(axis=1)).mean()
    assert e0 < 0.2 and e1 < 0.2


# ---- smoothing and rotation in front of the NVFP4 layer (Eq. (pair)) --------------------------

def test_float64_entry_points_reduce_to_the_bf16_ones():
    M, K, N, r = 9, 256, 24, 4
    X = wl.activations(M, K, seed=51, layer_id=4, dist="outlier", n_outlier=3)
    W = wl.weight(K, N, seed=51, layer_id=4)
    U = wl.basis(K, r, seed=51, layer_id=4)
    a, a64 = oracle.quantize_act_nvfp4(X, U), oracle.quantize_act_nvfp4_f64(oracle.bf16_bits_to_f64(X), U)
    w, w64 = oracle.pack_nvfp4(W, U), oracle.pack_nvfp4_f64(oracle.bf16_bits_to_f64(W), U)
    for k in a:
        np.testing.assert_array_equal(a[k], a64[k])
    for k in w:
        np.testing.assert_array_equal(w[k], w64[k])


@pytest.mark.parametrize("r", [0, 5])
def test_rotated_layer_equals_matrix_product_of_dequantized_operands(r):
    """On x~ and W~ the layer is still sg * deq(qx) deq(qw)^T + p_hat B_hat, and the codes of W~
    follow reading N4 (brute force, r = 0)."""
    M, K, N = 5, 256, 8
    X = wl.activations(M, K, seed=61, layer_id=r, dist="outlier", n_outlier=3)
    W = wl.weight(K, N, seed=61, layer_id=r)
    U = wl.basis(K, r, seed=61, layer_id=r) if r else np.zeros((K, 0), np.float32)
    s = np.exp(np.random.default_rng(r).uniform(-1, 1, K))
    Y, act, wts = oracle.forward_rotated_nvfp4(X, W, s, U)
    ref = float(wts["sg"]) * (_deq(act["qx"], act["sfx"]) @ _deq(wts["qw"], wts["sfw"]).T)
    if r:
        ref = ref + _f16(act["ph"]) @ _f16(wts["Bh"])
    np.testing.assert_allclose(Y, ref, rtol=1e-12, atol=1e-12 * np.abs(ref).max())
    if r == 0:
        Wt = oracle.rotate_weights(W, s)
        sg = np.float32(np.abs(Wt).max() / (6.0 * 448.0))
        assert wts["sg"] == sg
        for n in range(N):
            for b in range(K // 16):
                blk = Wt[16 * b:16 * b + 16, n]
                s_bits = nearest_even(np.abs(blk).max() / (6.0 * float(sg)), E4M3_POS)[0]
                assert wts["sfw"][n, b] == s_bits


def test_rotated_full_rank_protection_gives_the_16_bit_product():
    M, K, N = 6, 256, 12
    X = wl.activations(M, K, seed=71, layer_id=2)
    W = wl.weight(K, N, seed=71, layer_id=2)
    U = wl.basis(K, K, seed=71, layer_id=2)
    s = np.exp(np.random.default_rng(5).uniform(-1, 1, K))
    Y, _, _ = oracle.forward_rotated_nvfp4(X, W, s, U)
    exact = wl.bf16_bits_to_f32(X).astype(np.float64) @ wl.bf16_bits_to_f32(W).astype(np.float64)
    err = np.abs(Y - exact).max(axis=1) / np.abs(exact).max(axis=1)
    assert err.max() <= 1e-3
