"""GPU parity: the CUDA path (through the C ABI) against the CPU oracle, element by element.

Bars (stated once here, used below):
  * integer and byte work -- weight codes, weight scales, branch weights, the bf16 hi/lo split of
    U, and every activation code and scale when r = 0 -- bit-exact;
  * with r > 0, the quantizer applied to the kernel's own float32 remainder is bit-exact; end to
    end against the float64 oracle, codes may differ only at near-ties of the float64 remainder
    (Sec. 4.2 remainder formed in float32 on the GPU), at a rate below 1e-4;
  * the layer output (float32 variant) within max |dY| <= 1e-3 * max |y| per row of the oracle;
    given the kernel's own codes and scales, within 1e-5 (float32 accumulation order only);
  * the bf16 output equals RN_bf16 of the float32 output bit for bit.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_33269_gb300 import asp
from paper_2609_33269_gb300 import workloads as wl

from gpu_helpers import (Case, check_int4_act, check_layer_output, gemm_tol, rowwise_rel_err, to_dev_bf16,
                         unpack_nibbles)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2609_33269_gb300 import build
    build.build()
    asp.load()


SHAPES = [  # M, K, N, r, G
    (256, 512, 512, 16, 64),    # the tiny workload
    (33, 576, 200, 32, 32),     # ragged: M, N not tile multiples; K/128 not whole
    (1, 256, 136, 0, 64),       # single token, r = 0
    (200, 1024, 384, 48, 64),
    (130, 640, 264, 64, 32),
    (600, 512, 200, 16, 64),    # >= 512 tokens: float16 weight copy, TMA-store epilogue; M, N ragged
    (520, 384, 72, 0, 32),      # the same with r = 0, group 32, a single partial column tile
    (128, 64, 64, 64, 64),      # r = K
]


@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: "M%d_K%d_N%d_r%d_g%d" % s)
def test_pack_bit_exact(shape):
    M, K, N, r, G = shape
    c = Case(M, K, N, r, G, seed=3, layer_id=K + r)
    try:
        gw, ow = c.gpu_weights(), c.oracle_weights()
        np.testing.assert_array_equal(gw["qw"], ow["qw"])
        np.testing.assert_array_equal(gw["sw"], ow["sw"])
        if r > 0:
            np.testing.assert_array_equal(gw["Bh"], ow["Bh"])
            hi = wl.f32_to_bf16_bits(c.U)
            lo = wl.f32_to_bf16_bits(c.U - wl.bf16_bits_to_f32(hi))
            np.testing.assert_array_equal(gw["Uhl"][0][:, :r], hi)
            np.testing.assert_array_equal(gw["Uhl"][1][:, :r], lo)
            assert not gw["Uhl"][:, :, r:].any()
        assert gw["qw"].min() >= -7
    finally:
        c.close()


@pytest.mark.parametrize("M", [1, 33, 256, 300])
@pytest.mark.parametrize("G", [32, 64])
def test_activation_codes_bit_exact_r0(M, G):
    c = Case(M, 512, 128, 0, G, seed=4, layer_id=M)
    try:
        c.layer.quantize(c.X)
        ga, oa = c.gpu_act(), c.oracle_act(want_float64=False)
        np.testing.assert_array_equal(ga["sx"], oa["sx"])
        np.testing.assert_array_equal(ga["qx"], oa["qx"])
    finally:
        c.close()


@pytest.mark.parametrize("shape", [s for s in SHAPES if 0 < s[3] < s[1]], ids=lambda s: "M%d_K%d_N%d_r%d_g%d" % s)
def test_quantizer_bit_exact_on_kernel_remainder(shape):
    M, K, N, r, G = shape
    c = Case(M, K, N, r, G, seed=5, layer_id=K + r)
    try:
        R = c.residual()
        ga = c.gpu_act()
        q, s = oracle.quantize_residual(R, G)
        np.testing.assert_array_equal(ga["sx"], s)
        np.testing.assert_array_equal(ga["qx"], q)
        oa = c.oracle_act()
        X = wl.bf16_bits_to_f32(c.Xb).astype(np.float64)
        # the float32 remainder against the float64 one
        err = np.abs(R - oa["Xperp"]).max(axis=1) / np.abs(X).max(axis=1)
        assert err.max() <= 2e-5, err.max()
        # p_hat: the float32 projection differs from the float64 one by a few 1e-6 of the row's
        # largest projection (bf16 hi/lo split of U); after rounding to float16 that is at most
        # one float16 ulp plus that absolute error
        gp = ga["ph"].view(np.float16).astype(np.float64)
        op = oa["ph"].view(np.float16).astype(np.float64)
        ulp = np.spacing(np.maximum(np.abs(gp), np.abs(op)).astype(np.float16)).astype(np.float64)
        tol = ulp + 2e-5 * np.abs(oa["p"]).max(axis=1, keepdims=True)
        assert (np.abs(gp - op) <= tol).all(), np.abs(gp - op).max()
    finally:
        c.close()


@pytest.mark.parametrize("shape", [s for s in SHAPES if s[3] < s[1]], ids=lambda s: "M%d_K%d_N%d_r%d_g%d" % s)
def test_end_to_end_codes_and_output(shape):
    M, K, N, r, G = shape
    c = Case(M, K, N, r, G, seed=6, layer_id=K + r)
    try:
        Y = c.run(fp32=True).cpu().numpy()
        ga, gw = c.gpu_act(), c.gpu_weights()
        oa, ow = c.oracle_act(), c.oracle_weights()
        if r == 0:
            np.testing.assert_array_equal(ga["qx"], oa["qx"])
            np.testing.assert_array_equal(ga["sx"], oa["sx"])
            flip = np.zeros(M, bool)
        else:
            flip = check_int4_act(ga, oa, G)
        tol = gemm_tol(K, -(-r // 16) * 16)
        # the GEMM alone: oracle output from the kernel's own codes, scales and branch input
        Yk = oracle.linear(ga, dict(qw=gw["qw"], sw=gw["sw"], Bh=gw["Bh"]), G)
        assert rowwise_rel_err(Y, Yk).max() <= tol
        # the whole layer against the oracle
        Yo = oracle.linear(oa, ow, G)
        check_layer_output(Y, Yo, Yk, flip, tol)
        # bf16 output is the float32 output rounded once
        Yb = c.run(fp32=False)
        ref = torch.from_numpy(Y).cuda().to(torch.bfloat16)
        assert torch.equal(Yb.view(torch.int16), ref.view(torch.int16))
    finally:
        c.close()


@pytest.mark.parametrize("G", [32, 64])
def test_r_equals_K_gives_the_bf16_gemm(G):
    M, K, N = 96, 64, 64
    c = Case(M, K, N, K, G, seed=7, layer_id=G)
    try:
        Y = c.run(fp32=True).cpu().numpy()
        R = c.residual()
        X = wl.bf16_bits_to_f32(c.Xb).astype(np.float64)
        W = wl.bf16_bits_to_f32(c.Wb).astype(np.float64)
        assert np.abs(R).max() <= 1e-4 * np.abs(X).max()
        assert rowwise_rel_err(Y, X @ W).max() <= 1e-3
    finally:
        c.close()


def test_bounded_wait_reports_timeout_and_context_survives():
    c = Case(64, 128, 64, 16, 64, seed=8)
    try:
        assert asp.qwam_asp_get_error(c.layer.h) == asp.QWAM_OK
        asp.qwam_asp_debug_wait_timeout(c.layer.h, 20000)
        assert asp.qwam_asp_get_error(c.layer.h) == asp.QWAM_ERR_TIMEOUT
        Y = c.run(fp32=True)
        assert asp.qwam_asp_get_error(c.layer.h) == asp.QWAM_OK
        assert torch.isfinite(Y).all()
    finally:
        c.close()


def test_gpu_handles_reject_bad_arguments():
    c = Case(16, 128, 64, 16, 64, seed=9)
    try:
        h, ws = c.layer.h, c.layer.workspace(16)
        Y = torch.empty((16, 64), dtype=torch.float32, device="cuda")
        with pytest.raises(asp.QwamError) as e:
            asp.qwam_asp_linear(c.X, 16, h, Y, 7, ws)
        assert e.value.status == asp.QWAM_ERR_INVALID_ARG
        Xoff = c.X.view(-1)[1:]  # 2-byte offset: not 16-byte aligned
        with pytest.raises(asp.QwamError):
            asp.qwam_asp_quantize_act(Xoff, 8, h, ws)
        asp.qwam_asp_linear(c.X, 0, h, Y, asp.QWAM_Y_FP32, ws)  # M = 0 is a no-op
    finally:
        c.close()


FULL = [  # (name, M, K, N, r, dist, G) in the launch configuration the benchmark times
    ("dit_attn", 4096, 3072, 3072, 32, "outlier", 64),
    ("dit_attn_g32", 4096, 3072, 3072, 32, "outlier", 32),
    ("dit_qkv", 4096, 3072, 9216, 32, "outlier", 64),
    ("dit_qkv_r0", 4096, 3072, 9216, 0, "outlier", 64),    # the sweep's layers without ASP
    ("ffn_up", 4096, 3072, 12288, 32, "outlier", 64),
    ("ffn_down", 4096, 12288, 3072, 32, "student_t", 64),
    ("small_M32_r16", 32, 1024, 1024, 16, "outlier", 64),
    ("small_M128_N4096_r0", 128, 1024, 4096, 0, "outlier", 64),
]


@pytest.mark.parametrize("cfg", FULL, ids=lambda c: c[0])
def test_full_size_sampled_rows(cfg):
    name, M, K, N, r, dist, G = cfg
    c = Case(M, K, N, r, G, seed=0, layer_id=FULL.index(cfg) + 1, dist=dist)
    try:
        Y = c.run(fp32=True).cpu().numpy()
        rows = np.unique(np.random.default_rng(0).choice(M, size=min(M, 48), replace=False))
        rows = np.union1d(rows, [0, M - 1])
        ga = c.gpu_act(rows)
        gw = c.gpu_weights()
        ow = c.oracle_weights()
        np.testing.assert_array_equal(gw["qw"], ow["qw"])
        np.testing.assert_array_equal(gw["sw"], ow["sw"])
        oa = c.oracle_act(rows)
        tol = gemm_tol(K, -(-r // 16) * 16)
        Yk = oracle.linear(ga, dict(qw=gw["qw"], sw=gw["sw"], Bh=gw["Bh"]), G)
        assert rowwise_rel_err(Y[rows], Yk).max() <= tol
        Yo = oracle.linear(oa, ow, G)
        if r == 0:
            np.testing.assert_array_equal(ga["qx"], oa["qx"])
            np.testing.assert_array_equal(ga["sx"], oa["sx"])
            flip = np.zeros(len(rows), bool)
        else:
            flip = check_int4_act(ga, oa, G)
        check_layer_output(Y[rows], Yo, Yk, flip, tol)
    finally:
        c.close()
