"""Pins of the CPU oracle against what the paper and the mathematics fix (no GPU).

Each pin is independent of the oracle's own code:
  * exact rational arithmetic (fractions.Fraction) of the whole layer on tiny shapes,
  * brute-force argmin over the code grid for the quantizer (Eq. (quant)),
  * hand-derived closed-form group cases (tests/golden/quant_cases.txt),
  * library conversions (numpy float16) for the float16 format and exact rational rounding for
    the bfloat16 scales,
  * invariants of Sec. 4.2: x = U(U^T x) + x_perp, U^T W_perp = 0, x_perp U = 0, Eq. (asp) with
    Q = identity equals X W, r = 0 is plain per-group W4A4, r = K leaves a zero remainder,
  * storage of Table 3 (4.50 bits per weight at group 32) and the isotropy share r/K of App. C.
"""
import math
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle
from paper_2609_33269_gb300 import workloads as wl

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "quant_cases.txt")


# ---------------------------------------------------------------- exact helpers (tests only)

def f32_bits(x: float) -> int:
    return int(np.array([x], np.float32).view(np.uint32)[0])


def f32_from_bits(b: int) -> float:
    return float(np.array([b], np.uint32).view(np.float32)[0])


def rn_binary(fr: Fraction, mant: int, emin: int) -> Fraction:
    """Round |fr| to the nearest number with `mant` significant bits (ties to even), gradual
    underflow below 2**emin; sign restored.  Exact, for pins only."""
    if fr == 0:
        return Fraction(0)
    sgn = -1 if fr < 0 else 1
    a = abs(fr)
    e = a.numerator.bit_length() - a.denominator.bit_length()
    if Fraction(2) ** e > a:
        e -= 1
    if Fraction(2) ** (e + 1) <= a:
        e += 1
    e = max(e, emin)
    quantum = Fraction(2) ** (e - (mant - 1))
    q = a / quantum
    n = q.numerator // q.denominator
    rem = q - n
    if rem > Fraction(1, 2) or (rem == Fraction(1, 2) and n % 2 == 1):
        n += 1
    return sgn * n * quantum


def rn_f16(fr):
    return rn_binary(fr, 11, -14)


def rn_bf16(fr):
    return rn_binary(fr, 8, -126)


def brute_code(x: Fraction, s: Fraction) -> int:
    """argmin over the 15 codes -7..7 of |x - c s|, ties to the even code; s == 0 -> 0."""
    if s == 0:
        return 0
    best = None
    for c in range(-7, 8):
        d = abs(x - c * s)
        if best is None or d < best[0] or (d == best[0] and c % 2 == 0):
            best = (d, c)
    return best[1]


def bf16_frac(bits):
    return Fraction(float(wl.bf16_bits_to_f32(np.array([bits], np.uint16))[0]))


def f16_frac(bits):
    return Fraction(float(np.array([bits], np.uint16).view(np.float16)[0]))


# ---------------------------------------------------------------- number formats

def test_f16_rounding_matches_numpy():
    g = np.random.default_rng(7)
    xs = np.concatenate([
        g.standard_normal(20000) * 10.0 ** g.integers(-9, 5, 20000),
        np.array([0.0, -0.0, 65504.0, 65519.99, 65520.0, -65520.0, 6.1e-5, 5.96e-8, 2.98e-8,
                  2.9802322387695312e-08, 1.0 + 2.0 ** -11, 1.0 + 3 * 2.0 ** -11, 2.0 ** -25]),
    ])
    # exact ties of the 11-bit grid
    xs = np.concatenate([xs, (1024 + np.arange(0, 1024) + 0.5) * 2.0 ** -10])
    with np.errstate(over="ignore"):
        want = xs.astype(np.float16).view(np.uint16)
    got = np.array([oracle.f16_bits(x) for x in xs], np.uint16)
    np.testing.assert_array_equal(got, want)
    for h in (0, 1, 0x3c00, 0x3092, 0x7bff, 0x8001, 0x0400):
        assert oracle.f16_value(h) == float(np.array([h], np.uint16).view(np.float16)[0])


def test_bf16_scale_rounding_is_exact_rounding_of_the_quotient():
    """Readings R3 and R4: s = RN_bf16(a / 7), one rounding of the exact quotient, against exact
    rational rounding -- including float32 subnormal absmaxes, where rounding the quotient to
    float32 first can land on a bfloat16 midpoint that the exact quotient is not on."""
    g = np.random.default_rng(17)
    vals = list(np.abs(g.standard_normal(4000) * 10.0 ** g.integers(-30, 30, 4000)).astype(np.float32))
    vals += list((g.integers(1, 2 ** 23, 2000) * 2.0 ** -149).astype(np.float32))  # float32 subnormals
    # 7 times every bfloat16 midpoint of a few binades, and its float32 neighbours
    for e in (-133, -130, -10, 0, 5, 100):
        for n in range(0, 256, 7):
            t = np.float32(7 * (2 * n + 1) * 2.0 ** (e - 1))
            vals += [t, np.nextafter(t, np.float32(0)), np.nextafter(t, np.float32(np.inf))]
    vals += [np.float32(1146881 * 2.0 ** -149), np.float32(7.0), np.float32(1.0), np.float32(0.0)]
    for a in vals:
        a = float(a)
        want = rn_bf16(Fraction(a) / 7)
        got = bf16_frac(oracle.bf16_bits_div7(a))
        assert got == want, a
    # the float32-first double rounding differs on this subnormal absmax (the golden file has it)
    a = 1146881 * 2.0 ** -149
    assert float(np.float32(a / 7)) == 5 * 2.0 ** -134   # RN_f32 lands on a bfloat16 midpoint
    assert oracle.bf16_bits_div7(a) == 0x0003            # the exact quotient is above it


# ---------------------------------------------------------------- quantizer (Eq. (quant))

def _golden_cases():
    cases = []
    for line in open(GOLDEN):
        line = line.strip()
        if not line or line.startswith("#"):
            continue
        kind, vals, sbits, codes = [t.strip() for t in line.split("|")]
        num = [float.fromhex(v) if "p" in v else float(v) for v in vals.split(",")]
        cases.append((kind, num, int(sbits, 16),
                      [int(c) for c in codes.split(",")]))
    return cases


@pytest.mark.parametrize("case", _golden_cases())
def test_golden_group_cases(case):
    kind, vals, sbits, codes = case
    G = len(vals)
    if kind == "act":
        R = np.array([vals], np.float32)
        assert R[0].tolist() == vals  # every value is exact in float32
        q, s = oracle.quantize_residual(R, G)
        b = f32_bits(float(s[0, 0]))
        assert b & 0xFFFF == 0 and b >> 16 == sbits  # a bfloat16 value
        assert q[0].tolist() == codes
    else:
        # weight path: one output channel, K = G, r = 0, W holds the values exactly in bf16
        W = wl.f32_to_bf16_bits(np.array(vals, np.float32).reshape(G, 1))
        assert np.array_equal(wl.bf16_bits_to_f32(W)[:, 0], np.array(vals, np.float32))
        out = oracle.pack(W, np.zeros((G, 0), np.float32), G)
        assert int(out["sw"][0, 0]) == sbits
        assert out["qw"][0].tolist() == codes


def test_nearest_code_bruteforce_with_ties():
    g = np.random.default_rng(3)
    checked = 0
    for _ in range(3000):
        # scales with few significant bits make exact ties x = (c + 1/2) s representable
        s = float(np.float32(g.integers(1, 2 ** 10) * 2.0 ** int(g.integers(-20, 5))))
        u = g.random()
        if u < 0.4:
            c = int(g.integers(-8, 8))  # includes the ties -7.5 and 7.5, which saturate to -+7
            x = float(np.float32((c + 0.5) * s))
        elif u < 0.8:
            x = float(np.float32(g.uniform(-7.4, 7.4) * s))
        else:
            x = float(np.float32(g.uniform(-9.0, 9.0) * s))  # beyond the code range: saturates
        got = oracle.nearest_code(x, s)
        assert got == brute_code(Fraction(x), Fraction(s)), (x, s)
        checked += 1
    assert checked == 3000


def test_quantize_residual_bruteforce_and_error_bound():
    g = np.random.default_rng(11)
    for G in (32, 64):
        R = (g.standard_normal((3, 128)) * np.exp(g.uniform(-3, 3, (3, 1)))).astype(np.float32)
        R[1, :G] = 0.0  # an all-zero group
        q, s = oracle.quantize_residual(R, G)
        for m in range(R.shape[0]):
            for gi in range(128 // G):
                grp = [Fraction(float(v)) for v in R[m, gi * G:(gi + 1) * G]]
                amax = max(abs(v) for v in grp)
                s_exact = rn_bf16(amax / 7)
                assert Fraction(float(s[m, gi])) == s_exact
                for k, v in enumerate(grp):
                    c = brute_code(v, s_exact)
                    assert int(q[m, gi * G + k]) == c
                    # with a normal scale every |x| / s <= 7 (1 + 2^-8) < 7.5: no code saturates,
                    # and the dequantization error is at most s / 2
                    assert abs(v) < Fraction(15, 2) * s_exact or s_exact == 0 == v
                    assert abs(c * s_exact - v) <= s_exact / 2


# ---------------------------------------------------------------- whole layer, exact arithmetic

def _exact_layer(Xb, Wb, U, G):
    """Eq. (xsplit) + Eq. (asp) + Eq. (quant) in exact rationals, with the stated readings."""
    M, K = Xb.shape
    N = Wb.shape[1]
    X = [[bf16_frac(Xb[m, k]) for k in range(K)] for m in range(M)]
    W = [[bf16_frac(Wb[k, n]) for n in range(N)] for k in range(K)]
    return _exact_layer_values(X, W, U, G)


def _exact_layer_values(X, W, U, G):
    """_exact_layer on inputs given as lists of exact rationals X [M][K], W [K][N]."""
    M, K, N = len(X), len(W), len(W[0])
    r = U.shape[1]
    Uf = [[Fraction(float(U[k, j])) for j in range(r)] for k in range(K)]
    # pack
    Bf = [[sum(Uf[k][j] * W[k][n] for k in range(K)) for n in range(N)] for j in range(r)]
    Wp = [[W[k][n] - sum(Uf[k][j] * Bf[j][n] for j in range(r)) for n in range(N)] for k in range(K)]
    ng = K // G
    sw = [[rn_bf16(max(abs(Wp[k][n]) for k in range(g * G, (g + 1) * G)) / 7) for n in range(N)]
          for g in range(ng)]
    qw = [[brute_code(Wp[k][n], sw[k // G][n]) for k in range(K)] for n in range(N)]
    Bh = [[rn_f16(Bf[j][n]) for n in range(N)] for j in range(r)]
    # activations
    p = [[sum(X[m][k] * Uf[k][j] for k in range(K)) for j in range(r)] for m in range(M)]
    Xp = [[X[m][k] - sum(p[m][j] * Uf[k][j] for j in range(r)) for k in range(K)] for m in range(M)]
    sx = [[rn_bf16(max(abs(Xp[m][k]) for k in range(g * G, (g + 1) * G)) / 7) for g in range(ng)]
          for m in range(M)]
    qx = [[brute_code(Xp[m][k], sx[m][k // G]) for k in range(K)] for m in range(M)]
    ph = [[rn_f16(p[m][j]) for j in range(r)] for m in range(M)]
    Y = [[sum(sx[m][g] * sw[g][n] * sum(qx[m][k] * qw[n][k] for k in range(g * G, (g + 1) * G))
              for g in range(ng)) + sum(ph[m][j] * Bh[j][n] for j in range(r))
          for n in range(N)] for m in range(M)]
    return dict(qw=qw, sw=sw, Bh=Bh, qx=qx, sx=sx, ph=ph, Y=Y)


@pytest.mark.parametrize("r", [0, 1, 2])
@pytest.mark.parametrize("G", [32, 64])
def test_layer_matches_exact_rational_arithmetic(r, G):
    M, K, N = 4, 128, 8
    Xb = wl.activations(M, K, seed=5, layer_id=r, dist="outlier", n_outlier=3)
    Wb = wl.weight(K, N, seed=5, layer_id=r)
    U = wl.basis(K, r, seed=5, layer_id=r)
    ex = _exact_layer(Xb, Wb, U, G)
    w = oracle.pack(Wb, U, G)
    a = oracle.quantize_act(Xb, U, G)
    Y = oracle.linear(a, w, G)
    assert w["qw"].tolist() == ex["qw"]
    assert [[bf16_frac(b) for b in row] for row in w["sw"]] == ex["sw"]
    assert [[f16_frac(b) for b in row] for row in w["Bh"]] == ex["Bh"]
    assert a["qx"].tolist() == ex["qx"]
    assert [[Fraction(float(v)) for v in row] for row in a["sx"]] == ex["sx"]
    assert [[f16_frac(b) for b in row] for row in a["ph"]] == ex["ph"]
    Yex = np.array([[float(v) for v in row] for row in ex["Y"]])
    np.testing.assert_allclose(Y, Yex, rtol=1e-12, atol=1e-12 * np.abs(Yex).max())


# ---------------------------------------------------------------- invariants of Sec. 4.2

def _small_case(M=16, K=256, N=96, r=8, G=64, seed=1):
    Xb = wl.activations(M, K, seed=seed, layer_id=7, dist="outlier", n_outlier=4)
    Wb = wl.weight(K, N, seed=seed, layer_id=7)
    U = wl.basis(K, r, seed=seed, layer_id=7)
    return Xb, Wb, U


def test_split_identity_and_projection_invariants():
    Xb, Wb, U = _small_case()
    G = 64
    X = wl.bf16_bits_to_f32(Xb).astype(np.float64)
    W = wl.bf16_bits_to_f32(Wb).astype(np.float64)
    Ud = U.astype(np.float64)
    w = oracle.pack(Wb, U, G, want_float64=True)
    a = oracle.quantize_act(Xb, U, G, want_float64=True)
    scale = np.abs(X).max()
    # x = U (U^T x) + x_perp  (Eq. (xsplit))
    np.testing.assert_allclose(a["p"] @ Ud.T + a["Xperp"], X, rtol=0, atol=1e-12 * scale)
    # p = x U, B_f = U^T W (library matmul as an independent check)
    np.testing.assert_allclose(a["p"], X @ Ud, rtol=0, atol=1e-12 * scale)
    np.testing.assert_allclose(w["Bf"], Ud.T @ W, rtol=0, atol=1e-12 * np.abs(W).max())
    # (I - Pi) removes span(U): x_perp U = p (I - U^T U) and U^T W_perp = (I - U^T U) B_f hold
    # exactly for any U; with float32 U, I - U^T U is ~1e-7, so both are ~1e-7 and not 0.
    D = np.eye(U.shape[1]) - Ud.T @ Ud
    np.testing.assert_allclose(a["Xperp"] @ Ud, a["p"] @ D, rtol=0, atol=1e-12 * scale)
    np.testing.assert_allclose(Ud.T @ w["Wperp"], D @ w["Bf"], rtol=0, atol=1e-12 * np.abs(W).max())
    assert np.abs(a["Xperp"] @ Ud).max() <= 1e-5 * scale
    # Eq. (asp) with Q = identity: (U^T W)^T (U^T x) + W_perp^T x_perp = W^T x for orthonormal U;
    # for any U the two sides differ by exactly p (I - U^T U) B_f (expand the product).
    Y = oracle.linear_split_exact(a["p"], a["Xperp"], w["Bf"], w["Wperp"])
    ref = X @ W
    np.testing.assert_allclose(Y, ref - a["p"] @ D @ w["Bf"], rtol=0, atol=1e-12 * np.abs(ref).max())
    np.testing.assert_allclose(Y, ref, rtol=0, atol=1e-5 * np.abs(ref).max())


def test_r0_is_plain_per_group_w4a4():
    M, K, N, G = 64, 512, 128, 64
    Xb = wl.activations(M, K, seed=2, layer_id=3)
    Wb = wl.weight(K, N, seed=2, layer_id=3)
    U0 = np.zeros((K, 0), np.float32)
    Y, a, w = oracle.forward(Xb, Wb, U0, G)
    # independent numpy statement of per-group W4A4 (Eq. (quant) on both operands)
    X = wl.bf16_bits_to_f32(Xb).reshape(M, K // G, G)
    amax = np.abs(X).max(axis=2)
    sx = np.array([[float(rn_bf16(Fraction(float(a)) / 7)) for a in row] for row in amax], np.float32)
    with np.errstate(invalid="ignore", divide="ignore"):
        qx = np.where(sx[..., None] > 0, np.rint(X / sx[..., None].astype(np.float64)), 0).astype(np.int64)
    np.testing.assert_array_equal(a["sx"], sx)
    np.testing.assert_array_equal(a["qx"], qx.reshape(M, K))
    Wt = wl.bf16_bits_to_f32(Wb).astype(np.float64).T.reshape(N, K // G, G)
    swf = np.array([[float(rn_bf16(Fraction(float(a)) / 7)) for a in row] for row in np.abs(Wt).max(axis=2)])
    sw_bits = (swf.astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)
    np.testing.assert_array_equal(w["sw"], sw_bits.T)
    with np.errstate(invalid="ignore", divide="ignore"):
        qw = np.where(swf[..., None] > 0, np.rint(Wt / swf[..., None]), 0).astype(np.int64)
    np.testing.assert_array_equal(w["qw"], qw.reshape(N, K))
    P = np.einsum("mgk,ngk->mng", qx, qw)  # exact int64 group partial sums
    ref = np.einsum("mng,mg,ng->mn", P.astype(np.float64), sx.astype(np.float64), swf)
    np.testing.assert_allclose(Y, ref, rtol=1e-13, atol=1e-13 * np.abs(ref).max())
    assert a["ph"].shape == (M, 0) and w["Bh"].shape == (0, N)


def test_r_equals_K_zero_remainder_and_bf16_gemm():
    M, K, N, G = 32, 128, 64, 64
    Xb = wl.activations(M, K, seed=4, layer_id=9)
    Wb = wl.weight(K, N, seed=4, layer_id=9)
    U = wl.basis(K, K, seed=4, layer_id=9)
    w = oracle.pack(Wb, U, G, want_float64=True)
    a = oracle.quantize_act(Xb, U, G, want_float64=True)
    X = wl.bf16_bits_to_f32(Xb).astype(np.float64)
    W = wl.bf16_bits_to_f32(Wb).astype(np.float64)
    assert np.abs(a["Xperp"]).max() <= 1e-5 * np.abs(X).max()  # only float32 U roundoff remains
    assert np.abs(w["Wperp"]).max() <= 1e-5 * np.abs(W).max()
    Y = oracle.linear(a, w, G)
    ref = X @ W
    err = np.abs(Y - ref).max(axis=1) / np.abs(ref).max(axis=1)
    assert err.max() <= 1e-3, err.max()


def test_codes_range_and_storage_table3():
    Xb, Wb, U = _small_case(K=512, N=128, r=0)
    for G in (32, 64):
        w = oracle.pack(Wb, U, G)
        assert w["qw"].min() >= -7 and w["qw"].max() <= 7
        K, N = Wb.shape
        bits = 4 * w["qw"].size + 16 * w["sw"].size  # 4-bit codes + 16-bit scales
        bpw = bits / (K * N)
        assert bpw == 4 + 16 / G
    assert 4 + 16 / 32 == 4.50  # Table 3: per-group W4A4 at group 32


def test_isotropy_share_of_the_4bit_residual():
    """App. C: the rounding error of the 4-bit remainder puts about r/K of its squared norm in
    span(U).  Loose statistical check on synthetic data (factor of 2)."""
    M, K, r, G = 256, 1024, 32, 64
    Xb = wl.activations(M, K, seed=6, layer_id=11)
    U = wl.basis(K, r, seed=6, layer_id=11)
    a = oracle.quantize_act(Xb, U, G, want_float64=True)
    deq = a["qx"].astype(np.float64) * np.repeat(a["sx"].astype(np.float64), G, axis=1)
    delta = deq - a["Xperp"]
    share = (np.linalg.norm(delta @ U.astype(np.float64)) ** 2) / (np.linalg.norm(delta) ** 2)
    assert 0.5 * r / K <= share <= 2.0 * r / K, share


# ---------------------------------------------------------------- smoothing and rotation (Eq. (pair))

def _hadamard_dense(d):
    """Block-diagonal H from the bit formula H[i, j] = (-1)^popcount(i & j) / sqrt(B) per block of
    B (the largest power of two dividing d, at most 1024), written out element by element."""
    b = 1
    while d % (2 * b) == 0 and 2 * b <= 1024:
        b *= 2
    H = np.zeros((d, d))
    for i in range(d):
        for j in range(d):
            if i // b == j // b:
                H[i, j] = (-1) ** bin((i % b) & (j % b)).count("1") / math.sqrt(b)
    return H


@pytest.mark.parametrize("K", [64, 96, 640])
def test_rotation_is_the_dense_block_hadamard_and_keeps_the_product(K):
    M, N = 5, 12
    Xb = wl.activations(M, K, seed=8, layer_id=K, dist="outlier", n_outlier=3)
    Wb = wl.weight(K, N, seed=8, layer_id=K)
    s = np.exp(np.random.default_rng(K).uniform(-2, 2, K))
    X = wl.bf16_bits_to_f32(Xb).astype(np.float64)
    W = wl.bf16_bits_to_f32(Wb).astype(np.float64)
    H = _hadamard_dense(K)
    Wt = oracle.rotate_weights(Wb, s)
    Xt = oracle.rotate_acts(Xb, s)
    np.testing.assert_allclose(Wt, H @ (s[:, None] * W), rtol=0, atol=1e-13 * np.abs(Wt).max())
    np.testing.assert_allclose(Xt, (X / s[None, :]) @ H.T, rtol=0, atol=1e-13 * np.abs(Xt).max())
    # Eq. (pair): W~^T x~ = W^T diag(s) H^T H diag(s)^-1 x = W^T x
    ref = X @ W
    np.testing.assert_allclose(Xt @ Wt, ref, rtol=0, atol=1e-12 * np.abs(ref).max())
    # without smoothing factors the rotation alone; H is an involution: rotating twice is identity
    np.testing.assert_allclose(oracle.rotate_weights(Wb), H @ W, rtol=0, atol=1e-13 * np.abs(W).max())
    Xb2 = wl.f32_to_bf16_bits(np.eye(K, dtype=np.float32)[:3])
    np.testing.assert_allclose(oracle.rotate_acts(Xb2), H[:3], rtol=0, atol=1e-15)


def test_float64_entry_points_reduce_to_the_bf16_ones():
    """pack_f64 / quantize_act_f64 on the float64 values of bf16 inputs are the bf16 entry points,
    bit for bit (the bf16 ones are pinned above by exact rational arithmetic)."""
    M, K, N, r, G = 8, 256, 32, 4, 64
    Xb = wl.activations(M, K, seed=9, layer_id=2, dist="outlier", n_outlier=3)
    Wb = wl.weight(K, N, seed=9, layer_id=2)
    U = wl.basis(K, r, seed=9, layer_id=2)
    X = wl.bf16_bits_to_f32(Xb).astype(np.float64)
    W = wl.bf16_bits_to_f32(Wb).astype(np.float64)
    a, a64 = oracle.quantize_act(Xb, U, G, True), oracle.quantize_act_f64(X, U, G, True)
    w, w64 = oracle.pack(Wb, U, G, True), oracle.pack_f64(W, U, G, True)
    for k in a:
        np.testing.assert_array_equal(a[k], a64[k])
    for k in w:
        np.testing.assert_array_equal(w[k], w64[k])


@pytest.mark.parametrize("r", [0, 2])
def test_rotated_layer_matches_exact_rational_arithmetic(r):
    """The layer on x~ and W~ (float64 values that are not bf16) against exact rationals."""
    M, K, N, G = 3, 64, 4, 32
    Xb = wl.activations(M, K, seed=10, layer_id=r, dist="outlier", n_outlier=2)
    Wb = wl.weight(K, N, seed=10, layer_id=r)
    U = wl.basis(K, r, seed=10, layer_id=r)
    s = np.exp(np.random.default_rng(r).uniform(-1, 1, K))
    Y, a, w = oracle.forward_rotated(Xb, Wb, s, U, G)
    Xt, Wt = oracle.rotate_acts(Xb, s), oracle.rotate_weights(Wb, s)
    ex = _exact_layer_values([[Fraction(float(v)) for v in row] for row in Xt],
                             [[Fraction(float(v)) for v in row] for row in Wt], U, G)
    assert w["qw"].tolist() == ex["qw"]
    assert [[bf16_frac(b) for b in row] for row in w["sw"]] == ex["sw"]
    assert [[f16_frac(b) for b in row] for row in w["Bh"]] == ex["Bh"]
    assert a["qx"].tolist() == ex["qx"]
    assert [[Fraction(float(v)) for v in row] for row in a["sx"]] == ex["sx"]
    assert [[f16_frac(b) for b in row] for row in a["ph"]] == ex["ph"]
    Yex = np.array([[float(v) for v in row] for row in ex["Y"]])
    np.testing.assert_allclose(Y, Yex, rtol=1e-12, atol=1e-12 * np.abs(Yex).max())


def test_rotation_with_full_rank_protection_is_the_plain_product():
    """r = K in the rotated coordinates: the 4-bit remainder vanishes and the output is X W up to
    the float16 branch rounding, whatever the smoothing factors."""
    M, K, N, G = 16, 128, 32, 64
    Xb = wl.activations(M, K, seed=12, layer_id=1, dist="outlier", n_outlier=4)
    Wb = wl.weight(K, N, seed=12, layer_id=1)
    U = wl.basis(K, K, seed=12, layer_id=1)
    s = np.exp(np.random.default_rng(3).uniform(-1, 1, K))
    Y, _, _ = oracle.forward_rotated(Xb, Wb, s, U, G)
    ref = wl.bf16_bits_to_f32(Xb).astype(np.float64) @ wl.bf16_bits_to_f32(Wb).astype(np.float64)
    err = np.abs(Y - ref).max(axis=1) / np.abs(ref).max(axis=1)
    assert err.max() <= 1e-3, err.max()


def test_rotation_spreads_an_outlier_channel():
    """Sec. 3: the rotation spreads one large channel over its Hadamard block: every rotated entry
    is at most ||x||_1 / sqrt(B) (each is a +-1/sqrt(B) combination of the block), and the norm is
    kept (H is orthogonal)."""
    K = 256
    X = np.zeros((1, K), np.float32)
    X[0, 5] = 64.0
    X[0, 6:] = np.random.default_rng(1).uniform(-0.5, 0.5, K - 6).astype(np.float32)
    Xb = wl.f32_to_bf16_bits(X)
    Xd = wl.bf16_bits_to_f32(Xb).astype(np.float64)
    Xt = oracle.rotate_acts(Xb)
    assert np.abs(Xt).max() <= np.abs(Xd).sum() / math.sqrt(K) * (1 + 1e-15)
    assert np.abs(Xt).max() < 64.0 / 4
    np.testing.assert_allclose(np.linalg.norm(Xt), np.linalg.norm(Xd), rtol=1e-14)


def _hadamard_dense_vec(d):
    """The same block-diagonal H as _hadamard_dense, from the bit formula with numpy bit counts."""
    b = 1
    while d % (2 * b) == 0 and 2 * b <= 1024:
        b *= 2
    i = np.arange(b)
    x = np.bitwise_and(i[:, None], i[None, :]).astype(np.uint32)
    pc = np.zeros_like(x)
    while x.any():
        pc += x & 1
        x >>= 1
    blk = np.where(pc % 2 == 0, 1.0, -1.0) / math.sqrt(b)
    return np.kron(np.eye(d // b), blk), b


@pytest.mark.parametrize("K,B", [(1536, 512), (3072, 1024), (768, 256)])
def test_rotation_blocks_of_the_bench_shapes(K, B):
    """The block sizes of the benchmark's shapes (B = 256, 512, 1024) against the bit formula."""
    H, b = _hadamard_dense_vec(K)
    assert b == B
    Xb = wl.activations(3, K, seed=K, layer_id=2, dist="outlier")
    s = np.exp(np.random.default_rng(K).uniform(-1, 1, K))
    X = wl.bf16_bits_to_f32(Xb).astype(np.float64)
    Xt = oracle.rotate_acts(Xb, s)
    np.testing.assert_allclose(Xt, (X / s[None, :]) @ H.T, rtol=0, atol=1e-12 * np.abs(Xt).max())
