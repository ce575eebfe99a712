"""GPU parity of the layer with smoothing and the block Hadamard rotation in front (Sec. 3
Eq. (pair); App. B.1), through the C ABI, against the float64 oracle.

Bars:
  * packing: W~ = H diag(s) W is formed in float64 on the device in the oracle's butterfly order,
    so weight codes, weight scales and branch weights are bit-exact with the oracle's pack of W~,
    and the bf16 hi/lo split of the run-time projection basis diag(s)^-1 H U is bit-exact with
    the same split of the float64 product rounded once to float32;
  * activations: the quantizer applied to the kernel's own float32 rotated remainder
    (qwam_asp_debug_residual) is bit-exact, for r = 0 too (x~ is formed in float32 on the GPU);
    that remainder is within 2e-5 of the float64 one per row (relative to the row's largest
    rotated value); p_hat within one float16 ulp plus 2e-5 of the row's largest projection;
  * end to end, codes may differ from the oracle's only at near-ties of the float64 remainder,
    and the float32 output meets the same per-row bars as the layer without rotation.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_33269_gb300 import asp
from paper_2609_33269_gb300 import workloads as wl

from gpu_helpers import (Case, atoms_to_rows, check_int4_act, check_layer_output, check_nvfp4_activations, gemm_tol,
                         rowwise_rel_err, to_dev_bf16, unpack_e2m1)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2609_33269_gb300 import build
    build.build()
    asp.load()


def smoothing(K, seed, spread=1.0):
    return np.exp(np.random.default_rng(seed).uniform(-spread, spread, K)).astype(np.float32)


def hadamard_block(K):
    b = 1
    while K % (2 * b) == 0 and 2 * b <= 1024:
        b *= 2
    return b


SHAPES = [  # M, K, N, r, G, smoothing
    (256, 512, 512, 16, 64, True),      # the tiny workload's shape, rotated
    (33, 768, 200, 32, 32, True),       # B = 256, ragged M and N
    (1, 256, 136, 0, 64, True),         # one token, r = 0
    (130, 1536, 264, 0, 32, False),     # B = 512, rotation alone
    (200, 1024, 384, 48, 64, True),
    (77, 3072, 128, 32, 64, True),      # B = 1024, three Hadamard blocks
]
IDS = ["M%d_K%d_N%d_r%d_g%d_s%d" % s for s in SHAPES]


def make_case(shape, seed, small=256):
    """small: token counts up to which the small-M kernel runs (0: kernel (a) + rotation kernel)."""
    M, K, N, r, G, sm = shape
    c = Case(M, K, N, r, G, seed=seed, layer_id=K + r, rotate=True, s=smoothing(K, seed) if sm else None)
    asp.qwam_asp_set_small_m(c.layer.h, small)
    return c


PATHS = pytest.mark.parametrize("small", [256, 0], ids=["small_m", "kernel_a"])


@pytest.mark.parametrize("shape", SHAPES, ids=IDS)
def test_rotated_pack_bit_exact(shape):
    M, K, N, r, G, sm = shape
    c = make_case(shape, 3)
    try:
        assert asp.qwam_asp_rotation(c.layer.h) == hadamard_block(K)
        gw, ow = c.gpu_weights(), c.oracle_weights()
        np.testing.assert_array_equal(gw["qw"], ow["qw"])
        np.testing.assert_array_equal(gw["sw"], ow["sw"])
        if r > 0:
            np.testing.assert_array_equal(gw["Bh"], ow["Bh"])
            HU = oracle.fwht_cols(c.U.astype(np.float64))
            s = c.s64() if c.s is not None else np.ones(K)
            Up = (HU / s[:, None]).astype(np.float32)
            hi = wl.f32_to_bf16_bits(Up)
            lo = wl.f32_to_bf16_bits(Up - wl.bf16_bits_to_f32(hi))
            np.testing.assert_array_equal(gw["Uhl"][0][:, :r], hi)
            np.testing.assert_array_equal(gw["Uhl"][1][:, :r], lo)
    finally:
        c.close()


@PATHS
@pytest.mark.parametrize("shape", SHAPES, ids=IDS)
def test_rotated_quantizer_bit_exact_on_kernel_remainder(shape, small):
    M, K, N, r, G, sm = shape
    c = make_case(shape, 4, small)
    try:
        R = c.residual()
        ga = c.gpu_act()
        q, s = oracle.quantize_residual(R, G)
        np.testing.assert_array_equal(ga["sx"].view(np.uint32), s.view(np.uint32))
        np.testing.assert_array_equal(ga["qx"], q)
        oa = c.oracle_act()
        Xt = oracle.rotate_acts(c.Xb, c.s64())
        err = np.abs(R - oa["Xperp"]).max(axis=1) / np.abs(Xt).max(axis=1)
        assert err.max() <= 2e-5, err.max()
        if r > 0:
            gp = ga["ph"].view(np.float16).astype(np.float64)
            op = oa["ph"].view(np.float16).astype(np.float64)
            ulp = np.spacing(np.maximum(np.abs(gp), np.abs(op)).astype(np.float16)).astype(np.float64)
            tol = ulp + 2e-5 * np.abs(oa["p"]).max(axis=1, keepdims=True)
            assert (np.abs(gp - op) <= tol).all(), np.abs(gp - op).max()
    finally:
        c.close()


@PATHS
@pytest.mark.parametrize("shape", SHAPES, ids=IDS)
def test_rotated_end_to_end(shape, small):
    M, K, N, r, G, sm = shape
    c = make_case(shape, 6, small)
    try:
        Y = c.run(fp32=True).cpu().numpy()
        ga, gw = c.gpu_act(), c.gpu_weights()
        oa, ow = c.oracle_act(), c.oracle_weights()
        # the rotated remainder is a float64 value on the oracle's side even at r = 0
        flip = check_int4_act(ga, oa, G)
        tol = gemm_tol(K, -(-r // 16) * 16)
        Yk = oracle.linear(ga, dict(qw=gw["qw"], sw=gw["sw"], Bh=gw["Bh"]), G)
        assert rowwise_rel_err(Y, Yk).max() <= tol
        Yo = oracle.linear(oa, ow, G)
        check_layer_output(Y, Yo, Yk, flip, tol)
        Yb = c.run(fp32=False)
        assert torch.equal(Yb.view(torch.int16), torch.from_numpy(Y).cuda().to(torch.bfloat16).view(torch.int16))
    finally:
        c.close()


def test_rotated_static_entry_matches_the_workspace_call():
    c = make_case((300, 1024, 256, 32, 64, True), 8)
    try:
        Y = c.run(fp32=True)
        Ys = torch.empty_like(Y)
        asp.qwam_asp_linear_static(c.X, c.M, c.layer.h, Ys, asp.QWAM_Y_FP32)
        torch.cuda.synchronize()
        assert torch.equal(Y, Ys)
    finally:
        c.close()


def test_rotated_full_size_sampled_rows():
    """DiT attention projection shape (M = 4096 tokens, K = N = 3072, r = 32, group 64), rotated
    with smoothing, in the bench's launch configuration; sampled rows against the oracle."""
    M, K, N, r, G = 4096, 3072, 3072, 32, 64
    c = Case(M, K, N, r, G, seed=0, layer_id=1, dist="outlier", rotate=True, s=smoothing(K, 0))
    try:
        Y = c.run(fp32=True).cpu().numpy()
        rows = np.union1d(np.random.default_rng(1).choice(M, size=40, replace=False), [0, M - 1])
        ga, gw, ow = c.gpu_act(rows), c.gpu_weights(), c.oracle_weights()
        np.testing.assert_array_equal(gw["qw"], ow["qw"])
        np.testing.assert_array_equal(gw["sw"], ow["sw"])
        np.testing.assert_array_equal(gw["Bh"], ow["Bh"])
        oa = c.oracle_act(rows)
        tol = gemm_tol(K, 32)
        Yk = oracle.linear(ga, dict(qw=gw["qw"], sw=gw["sw"], Bh=gw["Bh"]), G)
        assert rowwise_rel_err(Y[rows], Yk).max() <= tol
        flip = check_int4_act(ga, oa, G)
        check_layer_output(Y[rows], oracle.linear(oa, ow, G), Yk, flip, tol)
    finally:
        c.close()


# ---- NVFP4 variant with the rotation ------------------------------------------------------------

@PATHS
@pytest.mark.parametrize("shape", [(200, 512, 256, 16), (65, 1536, 136, 0), (130, 3072, 128, 32)],
                         ids=lambda s: "M%d_K%d_N%d_r%d" % s)
def test_rotated_nvfp4(shape, small):
    M, K, N, r = shape
    Xb = wl.activations(M, K, seed=9, layer_id=K, dist="outlier")
    Wb = wl.weight(K, N, seed=9, layer_id=K)
    U = wl.basis(K, r, seed=9, layer_id=K)
    s = smoothing(K, 9)
    s64 = s.astype(np.float64)
    X = to_dev_bf16(Xb)
    layer = asp.AspLinear(to_dev_bf16(Wb), torch.from_numpy(U).cuda() if r else None, fmt=asp.QWAM_FMT_NVFP4,
                          rotate=True, s=torch.from_numpy(s).cuda())
    try:
        asp.qwam_asp_set_small_m(layer.h, small)
        e = asp.qwam_asp_export_nvfp4(layer.h)
        gw = dict(qw=unpack_e2m1(e["qw"]), sfw=e["sfw"], sg=e["sg"], Bh=e["Bh"][:, :r].T.copy())
        ow = oracle.pack_nvfp4_f64(oracle.rotate_weights(Wb, s64), U)
        assert gw["sg"].view(np.uint32) == np.float32(ow["sg"]).view(np.uint32)
        np.testing.assert_array_equal(gw["sfw"], ow["sfw"])
        np.testing.assert_array_equal(gw["qw"], ow["qw"])
        if r:
            np.testing.assert_array_equal(gw["Bh"], ow["Bh"])
        Y = layer(X, fp32=True)
        torch.cuda.synchronize()
        Y = Y.cpu().numpy()
        codes, atoms, ph = layer.act_views_nvfp4(M)
        ga = dict(qx=unpack_e2m1(codes.cpu().numpy()), sfx=atoms_to_rows(atoms.cpu().numpy(), M, K),
                  ph=ph.cpu().numpy().view(np.uint16)[:, :r].copy())
        R = torch.empty((M, K), dtype=torch.float32, device="cuda")
        asp.qwam_asp_debug_residual(X, M, layer.h, layer.workspace(M), R)
        torch.cuda.synchronize()
        R = R.cpu().numpy()
        q, sf = oracle.quantize_residual_nvfp4(R)
        np.testing.assert_array_equal(ga["qx"], q)
        np.testing.assert_array_equal(ga["sfx"], sf)
        Yk = oracle.linear_nvfp4(ga, gw)
        assert rowwise_rel_err(Y, Yk).max() <= 1e-5
        Yo, oa, _ = oracle.forward_rotated_nvfp4(Xb, Wb, s64, U)
        same = np.all(ga["qx"] == oa["qx"], axis=1) & np.all(ga["sfx"] == oa["sfx"], axis=1)
        Xrot = oracle.rotate_acts(Xb, s64)
        Xp = oracle.quantize_act_f64(Xrot, U, 32, want_float64=True)["Xperp"] if r else Xrot
        check_nvfp4_activations(ga, oa, Xp, R, Xrot)
        assert rowwise_rel_err(Y[same], Yo[same]).max() <= 1e-3
    finally:
        layer.close()


def test_rotated_pack_rejects_bad_arguments():
    K, N = 576, 64  # K % 256 != 0
    W = to_dev_bf16(wl.weight(K, N, seed=1, layer_id=1))
    with pytest.raises(asp.QwamError) as ei:
        asp.qwam_asp_pack_weights_rotated(W, None, None, K, N, 0, 64)
    assert ei.value.status == asp.QWAM_ERR_INVALID_ARG
    K = 512
    W = to_dev_bf16(wl.weight(K, N, seed=1, layer_id=1))
    for bad in (0.0, -1.0, np.inf, np.nan):
        s = smoothing(K, 1)
        s[17] = bad
        with pytest.raises(asp.QwamError) as ei:
            asp.qwam_asp_pack_weights_rotated(W, torch.from_numpy(s).cuda(), None, K, N, 0, 64)
        assert ei.value.status == asp.QWAM_ERR_RANGE
