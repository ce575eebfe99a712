"""Both activation kernels at small token counts: the small-M CUDA-core kernel (the default for
M <= 256 when K % 256 == 0) and the tensor-core kernel (a) (forced with qwam_asp_set_small_m(h, 0)),
against the oracle, with the bars of the parity tests:

  * the quantizer on the kernel's own float32 remainder: bit-exact; the remainder within 2e-5 of
    the float64 one per row; p_hat within one float16 ulp plus 2e-5 of the row's largest |p|;
  * r = 0: codes and scales bit-exact end to end;
  * outputs within 1e-3 * max |y| per row (rows with a near-tie flip: 1e-5 of the oracle on the
    kernel's own codes), in both formats.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_33269_gb300 import asp
from paper_2609_33269_gb300 import workloads as wl

from gpu_helpers import Case, check_int4_act, check_layer_output, gemm_tol, rowwise_rel_err, to_dev_bf16

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2609_33269_gb300 import build
    build.build()
    asp.load()


SHAPES = [  # M, K, N, r, G
    (32, 1024, 1024, 16, 64),    # the action-expert layer
    (64, 1024, 4096, 0, 64),
    (1, 512, 136, 64, 32),       # one token, the largest rank
    (128, 3072, 256, 32, 64),
    (200, 768, 200, 48, 32),     # ragged M and N
    (256, 2048, 128, 16, 64),
]
IDS = ["M%d_K%d_N%d_r%d_g%d" % s for s in SHAPES]
PATHS = [256, 0]  # small-M kernel, tensor-core kernel (a)


@pytest.mark.parametrize("small", PATHS, ids=["small_m", "kernel_a"])
@pytest.mark.parametrize("shape", SHAPES, ids=IDS)
def test_activation_paths_against_the_oracle(shape, small):
    M, K, N, r, G = shape
    c = Case(M, K, N, r, G, seed=21, layer_id=K + r)
    try:
        asp.qwam_asp_set_small_m(c.layer.h, small)
        R = c.residual()
        ga = c.gpu_act()
        q, s = oracle.quantize_residual(R, G)
        np.testing.assert_array_equal(ga["sx"].view(np.uint32), s.view(np.uint32))
        np.testing.assert_array_equal(ga["qx"], q)
        oa, ow = c.oracle_act(), c.oracle_weights()
        X = wl.bf16_bits_to_f32(c.Xb).astype(np.float64)
        err = np.abs(R - oa["Xperp"]).max(axis=1) / np.abs(X).max(axis=1)
        assert err.max() <= 2e-5, err.max()
        if r == 0:
            np.testing.assert_array_equal(ga["qx"], oa["qx"])
            np.testing.assert_array_equal(ga["sx"], oa["sx"])
            flip = np.zeros(M, bool)
        else:
            gp = ga["ph"].view(np.float16).astype(np.float64)
            op = oa["ph"].view(np.float16).astype(np.float64)
            ulp = np.spacing(np.maximum(np.abs(gp), np.abs(op)).astype(np.float16)).astype(np.float64)
            tol = ulp + 2e-5 * np.abs(oa["p"]).max(axis=1, keepdims=True)
            assert (np.abs(gp - op) <= tol).all(), np.abs(gp - op).max()
            flip = check_int4_act(ga, oa, G)
        Y = c.run(fp32=True).cpu().numpy()
        gw = c.gpu_weights()
        tol = gemm_tol(K, -(-r // 16) * 16)
        Yk = oracle.linear(ga, dict(qw=gw["qw"], sw=gw["sw"], Bh=gw["Bh"]), G)
        assert rowwise_rel_err(Y, Yk).max() <= tol
        check_layer_output(Y, oracle.linear(oa, ow, G), Yk, flip, tol)
    finally:
        c.close()


@pytest.mark.parametrize("small", PATHS, ids=["small_m", "kernel_a"])
@pytest.mark.parametrize("shape", [(32, 1024, 1024, 16), (128, 1024, 4096, 0), (77, 2048, 264, 32)],
                         ids=lambda s: "M%d_K%d_N%d_r%d" % s)
def test_nvfp4_activation_paths(shape, small):
    M, K, N, r = shape
    Xb = wl.activations(M, K, seed=23, layer_id=K, dist="outlier")
    Wb = wl.weight(K, N, seed=23, layer_id=K)
    U = wl.basis(K, r, seed=23, layer_id=K)
    X = to_dev_bf16(Xb)
    layer = asp.AspLinear(to_dev_bf16(Wb), torch.from_numpy(U).cuda() if r else None, fmt=asp.QWAM_FMT_NVFP4)
    try:
        asp.qwam_asp_set_small_m(layer.h, small)
        Y = layer(X, fp32=True)
        torch.cuda.synchronize()
        Y = Y.cpu().numpy()
        codes, atoms, ph = layer.act_views_nvfp4(M)
        p = codes.cpu().numpy()
        qx = np.empty((M, K), np.uint8)
        qx[:, 0::2] = p & 0xF
        qx[:, 1::2] = p >> 4
        a = atoms.cpu().numpy()
        rr = np.arange(M)[:, None]
        b = np.arange(K // 16)[None, :]
        sfx = a[((rr // 128) * (K // 64) + b // 4) * 512 + (rr % 32) * 16 + ((rr % 128) // 32) * 4 + b % 4]
        R = torch.empty((M, K), dtype=torch.float32, device="cuda")
        asp.qwam_asp_debug_residual(X, M, layer.h, layer.workspace(M), R)
        torch.cuda.synchronize()
        q, sf = oracle.quantize_residual_nvfp4(R.cpu().numpy())
        np.testing.assert_array_equal(qx, q)
        np.testing.assert_array_equal(sfx, sf)
        Yo, oa, _ = oracle.forward_nvfp4(Xb, Wb, U)
        if r == 0:
            np.testing.assert_array_equal(qx, oa["qx"])
            np.testing.assert_array_equal(sfx, oa["sfx"])
        same = np.all(qx == oa["qx"], axis=1) & np.all(sfx == oa["sfx"], axis=1)
        assert same.mean() >= 0.9
        assert rowwise_rel_err(Y[same], Yo[same]).max() <= 1e-3
    finally:
        layer.close()


def test_set_small_m_rejects_negative():
    c = Case(8, 256, 64, 0, 64, seed=1, layer_id=1)
    try:
        with pytest.raises(asp.QwamError) as ei:
            asp.qwam_asp_set_small_m(c.layer.h, -1)
        assert ei.value.status == asp.QWAM_ERR_INVALID_ARG
    finally:
        c.close()
