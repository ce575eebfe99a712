"""GPU parity of the NVFP4 variant (App. B.1: E2M1 codes, an E4M3 scale per 16 K, one float32
scale per weight tensor) against the CPU oracle, through the C ABI.

Bars (as for the INT4 layer):
  * weight codes, block scales, the per-tensor scale and the branch weights: bit-exact;
  * activation codes and block scales: bit-exact when r = 0 (the remainder is X itself), and,
    for r > 0, bit-exact given the kernel's own float32 remainder (qwam_asp_debug_residual);
    end to end at r > 0, that remainder within 2e-5 of the oracle's float64 one per row, every
    differing code or block scale a near tie of the oracle's quotient (within 1e-3 of an E2M1 or
    E4M3 midpoint) and at most max(2, 1e-4 * codes) of them;
  * the float32 output within 1e-5 * max |y| per row of the oracle evaluated on the kernel's
    own codes and scales (float32 accumulation order only), and within 1e-3 * max |y| per row
    of the end-to-end oracle for rows whose codes equal the oracle's;
  * the bf16 output equals RN_bf16 of the float32 output bit for bit.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_33269_gb300 import asp
from paper_2609_33269_gb300 import workloads as wl

from gpu_helpers import NvCase, atoms_to_rows, check_nvfp4_activations, rowwise_rel_err, to_dev_bf16, unpack_e2m1

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2609_33269_gb300 import build
    build.build()
    asp.load()


PACK_SHAPES = [(512, 512, 16), (256, 136, 0), (1024, 384, 48), (256, 64, 64), (768, 264, 32)]


@pytest.mark.parametrize("shape", PACK_SHAPES, ids=lambda s: "K%d_N%d_r%d" % s)
def test_nvfp4_pack_bit_exact(shape):
    K, N, r = shape
    c = NvCase(8, K, N, r, seed=5, layer_id=K + r)
    try:
        assert asp.qwam_asp_format(c.layer.h) == asp.QWAM_FMT_NVFP4
        gw, ow = c.gpu_weights(), c.oracle_weights()
        assert gw["sg"].view(np.uint32) == np.float32(ow["sg"]).view(np.uint32)
        np.testing.assert_array_equal(gw["sfw"], ow["sfw"])
        np.testing.assert_array_equal(gw["qw"], ow["qw"])
        if r > 0:
            np.testing.assert_array_equal(gw["Bh"], ow["Bh"])
    finally:
        c.close()


@pytest.mark.parametrize("M", [1, 33, 256, 300])
def test_nvfp4_activation_codes_bit_exact_r0(M):
    c = NvCase(M, 512, 128, 0, seed=6, layer_id=M)
    try:
        c.layer.quantize(c.X)
        ga = c.gpu_act()
        oa = oracle.quantize_act_nvfp4(c.Xb, c.U)
        np.testing.assert_array_equal(ga["sfx"], oa["sfx"])
        np.testing.assert_array_equal(ga["qx"], oa["qx"])
    finally:
        c.close()


@pytest.mark.parametrize("shape", [(128, 512, 128, 16), (100, 1024, 128, 64)], ids=lambda s: "M%d_K%d_N%d_r%d" % s)
def test_nvfp4_quantizer_bit_exact_given_residual(shape):
    M, K, N, r = shape
    c = NvCase(M, K, N, r, seed=7, layer_id=r)
    try:
        R = c.residual()
        ga = c.gpu_act()
        q, sf = oracle.quantize_residual_nvfp4(R)
        np.testing.assert_array_equal(ga["sfx"], sf)
        np.testing.assert_array_equal(ga["qx"], q)
    finally:
        c.close()


LAYER_SHAPES = [  # M, K, N, r
    (256, 512, 512, 16),    # the tiny workload's shape
    (33, 512, 200, 32),     # ragged M and N
    (1, 256, 136, 0),       # one token, r = 0
    (200, 1024, 384, 48),
    (130, 768, 264, 64),
    (300, 2048, 640, 0),    # several tiles per CTA row and column, ragged M
]


@pytest.mark.parametrize("shape", LAYER_SHAPES, ids=lambda s: "M%d_K%d_N%d_r%d" % s)
def test_nvfp4_layer_parity(shape):
    M, K, N, r = shape
    c = NvCase(M, K, N, r, seed=8, layer_id=M + r)
    try:
        Y = c.run(fp32=True).cpu().numpy()
        ga = c.gpu_act()
        gw = c.gpu_weights()
        ow = c.oracle_weights()
        # the oracle's output on the kernel's own codes and scales
        Yk = oracle.linear_nvfp4(ga, dict(qw=gw["qw"], sfw=gw["sfw"], sg=gw["sg"], Bh=ow["Bh"]))
        assert rowwise_rel_err(Y, Yk).max() <= 1e-5
        # end to end: rows whose codes equal the oracle's are within 1e-3 of the oracle
        oa = oracle.quantize_act_nvfp4(c.Xb, c.U)
        Yo = oracle.linear_nvfp4(oa, ow)
        same = np.all(ga["qx"] == oa["qx"], axis=1) & np.all(ga["sfx"] == oa["sfx"], axis=1)
        if r == 0:
            assert same.all()
        else:
            Xp = oracle.quantize_act(c.Xb, c.U, 32, want_float64=True)["Xperp"]
            check_nvfp4_activations(ga, oa, Xp, c.residual(), wl.bf16_bits_to_f32(c.Xb))
        assert rowwise_rel_err(Y[same], Yo[same]).max() <= 1e-3
        # bf16 output = RN_bf16(float32 output)
        Yb = c.run(fp32=False).float().cpu().numpy()
        np.testing.assert_array_equal(Yb, torch.from_numpy(Y).to(torch.bfloat16).float().numpy())
    finally:
        c.close()


def test_nvfp4_full_size_dit_attention_sampled_rows():
    """M = 4096, K = N = 3072, r = 32 (the DiT attention projection), in the launch configuration
    the benchmark times; 48 sampled rows against the oracle."""
    L = wl.dit_attention().layers[0]
    X = to_dev_bf16(L.x())
    layer = asp.AspLinear(to_dev_bf16(L.w()), torch.from_numpy(L.u()).cuda(), fmt=asp.QWAM_FMT_NVFP4)
    try:
        Y = layer(X, fp32=True)
        torch.cuda.synchronize()
        rows = np.sort(np.random.default_rng(0).choice(L.M, 48, replace=False))
        rows[0], rows[-1] = 0, L.M - 1
        Ys = Y[torch.from_numpy(rows).cuda()].cpu().numpy()
        ow = oracle.pack_nvfp4(L.w(), L.u())
        gw = asp.qwam_asp_export_nvfp4(layer.h)
        np.testing.assert_array_equal(unpack_e2m1(gw["qw"]), ow["qw"])
        oa = oracle.quantize_act_nvfp4(L.x()[rows], L.u())
        Yo = oracle.linear_nvfp4(oa, ow)
        codes, atoms, _ = layer.act_views_nvfp4(L.M)
        qx = unpack_e2m1(codes.cpu().numpy()[rows])
        sfx = atoms_to_rows(atoms.cpu().numpy(), L.M, L.K)[rows]
        same = np.all(qx == oa["qx"], axis=1) & np.all(sfx == oa["sfx"], axis=1)
        R = torch.empty((L.M, L.K), dtype=torch.float32, device="cuda")
        asp.qwam_asp_debug_residual(X, L.M, layer.h, layer.workspace(L.M), R)
        torch.cuda.synchronize()
        Xp = oracle.quantize_act(L.x()[rows], L.u(), 32, want_float64=True)["Xperp"]
        check_nvfp4_activations(dict(qx=qx, sfx=sfx), oa, Xp, R[torch.from_numpy(rows).cuda()].cpu().numpy(),
                                wl.bf16_bits_to_f32(L.x()[rows]))
        assert rowwise_rel_err(Ys[same], Yo[same]).max() <= 1e-3
        # rows with a near-tie flip: the oracle on the kernel's own codes
        if (~same).any():
            ph = layer.act_views_nvfp4(L.M)[2].cpu().numpy().view(np.uint16)[rows, :L.r].copy()
            Yk = oracle.linear_nvfp4(dict(qx=qx, sfx=sfx, ph=ph), ow)
            assert rowwise_rel_err(Ys[~same], Yk[~same]).max() <= 1e-5
        assert asp.qwam_asp_get_error(layer.h) == asp.QWAM_OK
    finally:
        layer.close()


def test_nvfp4_empty_input_and_bad_k():
    K, N = 256, 64
    W = to_dev_bf16(wl.weight(K, N, seed=1, layer_id=0))
    layer = asp.AspLinear(W, None, fmt=asp.QWAM_FMT_NVFP4)
    try:
        X = torch.empty((0, K), dtype=torch.bfloat16, device="cuda")
        Y = torch.empty((0, N), dtype=torch.float32, device="cuda")
        ws = torch.zeros(16, dtype=torch.uint8, device="cuda")
        asp.qwam_asp_linear(X, 0, layer.h, Y, asp.QWAM_Y_FP32, ws)
        torch.cuda.synchronize()
        assert asp.qwam_asp_get_error(layer.h) == asp.QWAM_OK
        with pytest.raises(asp.QwamError):  # an INT4 export of an NVFP4 handle is refused
            asp.qwam_asp_export(layer.h)
    finally:
        layer.close()
    W2 = to_dev_bf16(wl.weight(320, N, seed=1, layer_id=0))
    with pytest.raises(asp.QwamError) as ei:  # K must be a multiple of 256
        asp.qwam_asp_pack_weights_nvfp4(W2, None, 320, N, 0)
    assert ei.value.status == asp.QWAM_ERR_INVALID_ARG
