"""Directed rounding cases for both quantizer implementations, against the CPU oracle, bit for bit:
kernel (a)'s thread-per-row quantizers through qwam_asp_debug_quantize_rows, and the warp-wide ones
of the small-M and rotation kernels through qwam_asp_debug_quantize_lanes (the same device
functions those kernels run).

Random activations reach a rounding boundary too rarely to exercise the kernels' fast paths
where they hand over to exact decisions, so the values here are placed on and next to the
boundaries themselves:

* INT4 (Eq. (quant), readings R2/R3/R5): code = nearest integer to x / s, ties to even, with
  s = RN_bf16(amax / 7) of the exact quotient.  Values sit at (c + 1/2) s exactly (a bfloat16 s
  makes these products exact, so they are true ties) and one to three float32 steps either side,
  for scales from absmaxes of few and of many significant bits; groups of zeros, groups small
  enough to take the power-of-two rescaling path, and a float32 subnormal absmax whose quotient
  rounded to float32 would sit on a bfloat16 midpoint are included.
* NVFP4 (App. B.1, readings N1-N3): code = RN_e2m1(RN_f32(x / s)), s = RN_e4m3(RN_f32(amax / 6)).
  Values sit on every E2M1 midpoint m (m s is exact for an E4M3 s), one to four float32 steps
  from it (where the float32 quotient can round onto the midpoint and become a tie), at relative
  distances 2^-21 .. 2^-17 (either side of the fast path's bracket), beyond 6 s after a scale
  that rounded down (saturation), and in blocks of zeros and with subnormal E4M3 scales.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_33269_gb300 import asp

from gpu_helpers import decode_ob4

pytestmark = pytest.mark.gpu

E2M1_MIDPOINTS = (0.25, 0.75, 1.25, 1.75, 2.5, 3.5, 5.0)


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2609_33269_gb300 import build
    build.build()
    asp.load()


def f32(x):
    return np.float32(x)


def steps(x, n):
    """x moved n float32 steps (n < 0: toward -inf)."""
    x = f32(x)
    d = np.float32(np.inf) if n > 0 else np.float32(-np.inf)
    for _ in range(abs(n)):
        x = np.nextafter(x, d)
    return x


def fill(vals, size, amax, rng):
    """Pad a list of values to `size` with random values of magnitude <= amax / 2 and shuffle,
    keeping amax itself in the group."""
    vals = [f32(v) for v in vals][: size - 1]
    while len(vals) < size - 1:
        vals.append(f32(rng.uniform(-0.5, 0.5) * amax))
    vals.append(f32(amax))
    out = np.array(vals, np.float32)
    rng.shuffle(out)
    return out


def bf16_scale(A):
    """The oracle's scale RN_bf16(A / 7) as a float32 value."""
    return np.array([oracle.bf16_bits_div7(float(f32(A))) << 16], np.uint32).view(np.float32)[0]


def int4_groups(G, rng):
    groups = []
    # exact ties: scales with few significant bits, amax = 7 s exactly
    for s_t in (0.375, 1.0, 0.0625, 3.0, 5.0 * 2.0 ** -20, 0.8125):
        s = f32(s_t)
        A = f32(7 * s)
        assert bf16_scale(A) == s
        vals = [(c + 0.5) * s for c in range(-7, 7)] + [-(c + 0.5) * s for c in range(0, 7)]
        vals += [c * s for c in range(-7, 8)]
        groups.append(fill(vals, G, A, rng))
        groups.append(fill([-v for v in vals], G, -A, rng))
    # near ties: absmaxes of many significant bits; the ties (c + 1/2) s and their neighbours
    for A in (1.0, 2.9, 0.123456, 17.77, 3.3e-5, 1234.5678):
        s = bf16_scale(A)
        vals = []
        for c in range(-7, 7):
            t = f32((c + 0.5) * np.float64(s))
            vals += [steps(t, k) for k in (-3, -2, -1, 0, 1, 2, 3)]
        for i in range(0, len(vals), G - 1):
            groups.append(fill(vals[i:i + G - 1], G, A, rng))
    groups.append(np.zeros(G, np.float32))
    # tiny groups: the scale is below 2^-100 and the codes are formed on rescaled values; the
    # last absmax is a float32 subnormal whose exact quotient lies just above a bfloat16 midpoint
    for A in (3e-33, 7.5e-36, 1146881 * 2.0 ** -149):
        s = bf16_scale(A)
        vals = []
        for c in range(-7, 7):
            t = f32((c + 0.5) * np.float64(s))
            vals += [steps(t, k) for k in (-1, 0, 1)]
        groups.append(fill(vals[: G - 1], G, A, rng))
    return groups


def e4m3_values():
    v = [oracle.e4m3_value(b) for b in range(1, 0x7F)]
    return [x for x in v if np.isfinite(x)]


def nvfp4_blocks(rng):
    blocks = []
    scales = [1.25, 1.75, 0.375, 13.0, 0.8125, 1.0, 2.0 ** -7 * 1.625, 3 * 2.0 ** -9, 448.0 / 8]
    for s_t in scales:
        s = f32(s_t)
        A = f32(6 * np.float64(s))
        assert f32(np.float64(A) / 6) == s, s_t
        mids = [f32(m * np.float64(s)) for m in E2M1_MIDPOINTS]
        blocks.append(fill(mids + [-v for v in mids], 16, A, rng))
        for k in (1, 2, 3, 4):
            near = [steps(v, k) for v in mids] + [steps(v, -k) for v in mids]
            blocks.append(fill(near[:15], 16, A, rng))
        for e in (-21, -20, -19, -18, -17):
            f_up, f_dn = 1.0 + 2.0 ** e, 1.0 - 2.0 ** e
            br = [f32(m * np.float64(s) * f_up) for m in E2M1_MIDPOINTS] + \
                 [f32(-m * np.float64(s) * f_dn) for m in E2M1_MIDPOINTS]
            blocks.append(fill(br, 16, A, rng))
    # saturation: amax / 6 rounds down to the E4M3 grid, so amax / s exceeds 6
    for A in (6 * 1.0624, 6 * 1.124, 6 * 13.4):
        blocks.append(fill([A * 0.99, -A, A * 0.9], 16, A, rng))
    blocks.append(np.zeros(16, np.float32))
    # every E4M3 scale once, with values on the midpoints
    for s_t in rng.choice(e4m3_values(), 40, replace=False):
        s = f32(s_t)
        A = f32(6 * np.float64(s))
        if f32(np.float64(A) / 6) != s:
            continue
        mids = [f32(m * np.float64(s)) for m in E2M1_MIDPOINTS]
        blocks.append(fill(mids + [steps(v, 1) for v in mids], 16, A, rng))
    return blocks


def as_rows(chunks, width, K):
    """Concatenate chunks of `width` values into rows of K (zero-padded at the end)."""
    per_row = K // width
    n = -(-len(chunks) // per_row) * per_row
    chunks = list(chunks) + [np.zeros(width, np.float32)] * (n - len(chunks))
    return np.concatenate(chunks).reshape(-1, K)


def run_lanes(R, fmt, G):
    """The warp-wide quantizers (small-M and rotation kernels): outputs in the workspace layouts,
    returned row-major like run()."""
    M, K = R.shape
    M_pad = -(-M // 128) * 128
    Rd = torch.from_numpy(R).cuda()
    if fmt == asp.QWAM_FMT_NVFP4:
        codes = torch.zeros((M, K // 2), dtype=torch.uint8, device="cuda")
        atoms = torch.zeros(M_pad * K // 16, dtype=torch.uint8, device="cuda")
        asp.qwam_asp_debug_quantize_lanes(Rd, M, K, fmt, 16, codes, atoms)
        torch.cuda.synchronize()
        a = atoms.cpu().numpy()
        r = np.arange(M)[:, None]
        b = np.arange(K // 16)[None, :]
        sf = a[((r // 128) * (K // 64) + b // 4) * 512 + (r % 32) * 16 + ((r % 128) // 32) * 4 + b % 4]
        return codes.cpu().numpy(), sf
    codes = torch.zeros((M, K // 2), dtype=torch.uint8, device="cuda")
    scales = torch.zeros((K // G, M_pad), dtype=torch.bfloat16, device="cuda")
    asp.qwam_asp_debug_quantize_lanes(Rd, M, K, fmt, G, codes, scales)
    torch.cuda.synchronize()
    return decode_ob4(codes.cpu().numpy()), scales.float().cpu().numpy()[:, :M].T.copy()


IMPLS = {"thread_rows": None, "warp_lanes": run_lanes}


def run(R, fmt, G, impl="thread_rows"):
    if IMPLS[impl] is not None:
        return IMPLS[impl](R, fmt, G)
    M, K = R.shape
    Rd = torch.from_numpy(R).cuda()
    if fmt == asp.QWAM_FMT_NVFP4:
        codes = torch.zeros((M, K // 2), dtype=torch.uint8, device="cuda")
        scales = torch.zeros((M, K // 16), dtype=torch.uint8, device="cuda")
    else:
        codes = torch.zeros((M, K // 2), dtype=torch.uint8, device="cuda")
        scales = torch.zeros((M, K // G), dtype=torch.bfloat16, device="cuda")
    asp.qwam_asp_debug_quantize_rows(Rd, M, K, fmt, G, codes, scales)
    torch.cuda.synchronize()
    c = codes.cpu().numpy()
    if fmt == asp.QWAM_FMT_NVFP4:
        return c, scales.cpu().numpy()
    return decode_ob4(c), scales.float().cpu().numpy()


@pytest.mark.parametrize("impl", list(IMPLS))
@pytest.mark.parametrize("G", [64, 32])
def test_int4_rounding_on_and_next_to_ties(G, impl):
    rng = np.random.default_rng(100 + G)
    R = as_rows(int4_groups(G, rng), G, 256)
    q, s = run(R, asp.QWAM_FMT_INT4, G, impl)
    q = q.astype(np.int16)
    oq, os_ = oracle.quantize_residual(R, G)
    np.testing.assert_array_equal(s.view(np.uint32), os_.view(np.uint32))
    np.testing.assert_array_equal(q, oq.astype(np.int16))
    # the cases reach both sides of the ties and the ties themselves
    assert np.abs(q).max() == 7 and (q == 0).any()


@pytest.mark.parametrize("impl", list(IMPLS))
def test_nvfp4_rounding_on_and_next_to_midpoints(impl):
    rng = np.random.default_rng(7)
    R = as_rows(nvfp4_blocks(rng), 16, 256)
    packed, sf = run(R, asp.QWAM_FMT_NVFP4, 16, impl)
    q = np.empty((R.shape[0], R.shape[1]), np.uint8)
    q[:, 0::2] = packed & 0xF
    q[:, 1::2] = packed >> 4
    oq, osf = oracle.quantize_residual_nvfp4(R)
    np.testing.assert_array_equal(sf, osf)
    np.testing.assert_array_equal(q, oq)
    assert (q & 7).max() == 7 and (q == 0).any()


def test_debug_quantize_rows_rejects_bad_arguments():
    R = torch.zeros((2, 96), dtype=torch.float32, device="cuda")
    c = torch.zeros((2, 96), dtype=torch.uint8, device="cuda")
    s = torch.zeros((2, 3), dtype=torch.float32, device="cuda")
    for args in ((R, 2, 96, asp.QWAM_FMT_INT4, 32),      # K % 64 != 0
                 (R, 2, 64, 7, 32),                      # unknown format
                 (R, 2, 64, asp.QWAM_FMT_INT4, 48)):     # group not 32 or 64
        with pytest.raises(asp.QwamError) as ei:
            asp.qwam_asp_debug_quantize_rows(*args, c, s)
        assert ei.value.status == asp.QWAM_ERR_INVALID_ARG
