"""GPU parity of protected ranks above 64 (the general-rank activation path: Eq. (xsplit) on the
CUDA cores, one CTA per token row) and of r = K, through the C ABI, against the float64 oracle.

Bars (those of the rank <= 64 tests):
  * INT4: codes and scales bit-exact given the kernel's own float32 remainder; that remainder
    within 2e-5 of the oracle's float64 one per row; p_hat within one float16 ulp plus 2e-5 of the
    row's largest projection; end to end every differing code a near tie (at most 1e-4 of them),
    the output within 1e-5 per row of the oracle on the kernel's own codes and within 1e-3 of the
    oracle for rows without a flip; bf16 output = RN_bf16 of the float32 output;
  * NVFP4: the same with the NVFP4 near-tie rule (E2M1 and E4M3 midpoints);
  * r = K (Eq. (asp) with U a basis of the whole space): the remainder vanishes, the 4-bit part is
    zero (INT4; NVFP4 quantizes the float32 basis' round-off of zero), and the layer is the
    16-bit GEMM p_hat B_hat^T, i.e. X W up to float16 rounding.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_33269_gb300 import asp
from paper_2609_33269_gb300 import workloads as wl

from gpu_helpers import Case, NvCase, check_int4_act, check_layer_output, check_nvfp4_activations, gemm_tol, rowwise_rel_err

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2609_33269_gb300 import build
    build.build()
    asp.load()


SHAPES = [  # M, K, N, r, G
    (96, 512, 256, 96, 64),
    (130, 1024, 136, 200, 32),   # ragged M and N, r_pad = 208
    (33, 768, 64, 128, 64),
    (300, 512, 512, 480, 32),    # several CTAs per column of M tiles, r close to K
]
IDS = ["M%d_K%d_N%d_r%d_g%d" % s for s in SHAPES]


def _check_phat(ga_ph, oa):
    gp = ga_ph.view(np.float16).astype(np.float64)
    op = oa["ph"].view(np.float16).astype(np.float64)
    ulp = np.spacing(np.maximum(np.abs(gp), np.abs(op)).astype(np.float16)).astype(np.float64)
    tol = ulp + 2e-5 * np.abs(oa["p"]).max(axis=1, keepdims=True)
    assert (np.abs(gp - op) <= tol).all(), np.abs(gp - op).max()


@pytest.mark.parametrize("shape", SHAPES, ids=IDS)
def test_int4_quantizer_bit_exact_on_kernel_remainder(shape):
    M, K, N, r, G = shape
    c = Case(M, K, N, r, G, seed=21, layer_id=r)
    try:
        R = c.residual()
        ga = c.gpu_act()
        q, s = oracle.quantize_residual(R, G)
        np.testing.assert_array_equal(ga["sx"].view(np.uint32), s.view(np.uint32))
        np.testing.assert_array_equal(ga["qx"], q)
        oa = c.oracle_act()
        X = wl.bf16_bits_to_f32(c.Xb).astype(np.float64)
        err = np.abs(R - oa["Xperp"]).max(axis=1) / np.abs(X).max(axis=1)
        assert err.max() <= 2e-5, err.max()
        _check_phat(ga["ph"], oa)
    finally:
        c.close()


@pytest.mark.parametrize("shape", SHAPES, ids=IDS)
def test_int4_end_to_end(shape):
    M, K, N, r, G = shape
    c = Case(M, K, N, r, G, seed=22, layer_id=r)
    try:
        Y = c.run(fp32=True).cpu().numpy()
        ga, gw = c.gpu_act(), c.gpu_weights()
        oa, ow = c.oracle_act(), c.oracle_weights()
        np.testing.assert_array_equal(gw["qw"], ow["qw"])
        np.testing.assert_array_equal(gw["Bh"], ow["Bh"])
        flip = check_int4_act(ga, oa, G)
        tol = gemm_tol(K, -(-r // 16) * 16)
        Yk = oracle.linear(ga, dict(qw=gw["qw"], sw=gw["sw"], Bh=gw["Bh"]), G)
        assert rowwise_rel_err(Y, Yk).max() <= tol
        check_layer_output(Y, oracle.linear(oa, ow, G), Yk, flip, tol)
        Yb = c.run(fp32=False)
        assert torch.equal(Yb.view(torch.int16), torch.from_numpy(Y).cuda().to(torch.bfloat16).view(torch.int16))
        assert asp.qwam_asp_get_error(c.layer.h) == asp.QWAM_OK
    finally:
        c.close()


@pytest.mark.parametrize("G", [32, 64])
@pytest.mark.parametrize("K", [256, 512])
def test_int4_r_equals_K_gives_the_16_bit_gemm(K, G):
    M, N = 96, 192
    c = Case(M, K, N, K, G, seed=23, layer_id=K + G)
    try:
        Y = c.run(fp32=True).cpu().numpy()
        R = c.residual()
        X = wl.bf16_bits_to_f32(c.Xb).astype(np.float64)
        W = wl.bf16_bits_to_f32(c.Wb).astype(np.float64)
        assert np.abs(R).max() <= 1e-4 * np.abs(X).max()
        gw = c.gpu_weights()
        # W_perp is float64 roundoff of the float32 basis: the 4-bit part is negligible (its
        # bfloat16 scales are tiny, not zero: bfloat16 has float32's exponent range)
        sw = wl.bf16_bits_to_f32(gw["sw"]).astype(np.float64)
        assert 7 * sw.max() <= 2e-5 * np.abs(W).max()
        Yo = oracle.linear(c.oracle_act(), c.oracle_weights(), G)
        assert rowwise_rel_err(Y, Yo).max() <= 1e-3
        assert rowwise_rel_err(Y, X @ W).max() <= 5e-3
    finally:
        c.close()


NV_SHAPES = [(96, 512, 256, 96), (130, 1024, 136, 200), (40, 512, 128, 512)]


@pytest.mark.parametrize("shape", NV_SHAPES, ids=lambda s: "M%d_K%d_N%d_r%d" % s)
def test_nvfp4_large_rank(shape):
    M, K, N, r = shape
    c = NvCase(M, K, N, r, seed=24, layer_id=r)
    try:
        Y = c.run(fp32=True).cpu().numpy()
        ga, gw, ow = c.gpu_act(), c.gpu_weights(), c.oracle_weights()
        np.testing.assert_array_equal(gw["qw"], ow["qw"])
        np.testing.assert_array_equal(gw["Bh"], ow["Bh"])
        R = c.residual()
        q, sf = oracle.quantize_residual_nvfp4(R)
        np.testing.assert_array_equal(ga["qx"], q)
        np.testing.assert_array_equal(ga["sfx"], sf)
        Yk = oracle.linear_nvfp4(ga, dict(qw=gw["qw"], sfw=gw["sfw"], sg=gw["sg"], Bh=ow["Bh"]))
        assert rowwise_rel_err(Y, Yk).max() <= 1e-5
        oa = oracle.quantize_act_nvfp4(c.Xb, c.U)
        Yo = oracle.linear_nvfp4(oa, ow)
        X = wl.bf16_bits_to_f32(c.Xb)
        if r < K:
            Xp = oracle.quantize_act(c.Xb, c.U, 32, want_float64=True)["Xperp"]
            check_nvfp4_activations(ga, oa, Xp, R, X)
            same = np.all(ga["qx"] == oa["qx"], axis=1) & np.all(ga["sfx"] == oa["sfx"], axis=1)
            assert rowwise_rel_err(Y[same], Yo[same]).max() <= 1e-3
        else:
            # W_perp is the float32 basis' round-off of zero: its codes are noise at scale ~1e-7 |W|
            assert np.abs(R).max() <= 1e-4 * np.abs(X).max()
            assert rowwise_rel_err(Y, Yo).max() <= 1e-3
            W = wl.bf16_bits_to_f32(c.Wb).astype(np.float64)
            assert rowwise_rel_err(Y, X.astype(np.float64) @ W).max() <= 5e-3
        Yb = c.run(fp32=False).float().cpu().numpy()
        np.testing.assert_array_equal(Yb, torch.from_numpy(Y).to(torch.bfloat16).float().numpy())
    finally:
        c.close()


def test_large_rank_with_bias_and_static_entry():
    """The general-rank path with a bias in both formats, and through the static scratch."""
    M, K, N, r = 64, 512, 256, 160
    for fmt in (asp.QWAM_FMT_INT4, asp.QWAM_FMT_NVFP4):
        c = NvCase(M, K, N, r, seed=25, layer_id=fmt) if fmt == asp.QWAM_FMT_NVFP4 else Case(M, K, N, r, 64, seed=25)
        try:
            Y0 = c.run(fp32=True)
            bias = torch.linspace(-3.0, 3.0, N, device="cuda", dtype=torch.float32)
            asp.qwam_asp_set_bias(c.layer.h, bias)
            Y1 = c.run(fp32=True)
            d = (Y1 - Y0 - bias[None, :]).abs().max().item()
            assert d <= 1e-5 * max(Y0.abs().max().item(), 3.0), d
            Ys = torch.empty_like(Y1)
            asp.qwam_asp_linear_static(c.X, M, c.layer.h, Ys, asp.QWAM_Y_FP32)
            torch.cuda.synchronize()
            assert torch.equal(Ys, Y1)
            assert asp.qwam_asp_get_error(c.layer.h) == asp.QWAM_OK
        finally:
            c.close()
