"""The layer's bias, added in the GEMM epilogue (App. B.1), through qwam_asp_set_bias.

Bar: with a bias set, the float32 output is RN_f32(y + b[n]) of the bias-free float32 output y of
the same inputs, bit for bit (one float32 addition in the epilogue), in both 4-bit formats and
for a rotated layer; against the oracle (its output plus the bias, float64) the per-row bar of
the bias-free layer holds; removing the bias restores the bias-free output exactly.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_33269_gb300 import asp
from paper_2609_33269_gb300 import workloads as wl

from gpu_helpers import Case, rowwise_rel_err, to_dev_bf16

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2609_33269_gb300 import build
    build.build()
    asp.load()


def run(layer, X, fp32=True):
    Y = layer(X, fp32=fp32)
    torch.cuda.synchronize()
    return Y


@pytest.mark.parametrize("fmt,rotate", [(asp.QWAM_FMT_INT4, False), (asp.QWAM_FMT_NVFP4, False),
                                        (asp.QWAM_FMT_INT4, True)], ids=["int4", "nvfp4", "int4_rotated"])
@pytest.mark.parametrize("shape", [(200, 512, 264, 16), (33, 1024, 136, 0), (600, 512, 264, 16)],
                         ids=lambda s: "M%d_K%d_N%d_r%d" % s)
def test_bias_is_one_float32_addition(fmt, rotate, shape):
    M, K, N, r = shape
    Xb = wl.activations(M, K, seed=13, layer_id=K, dist="outlier")
    Wb = wl.weight(K, N, seed=13, layer_id=K)
    U = wl.basis(K, r, seed=13, layer_id=K)
    X = to_dev_bf16(Xb)
    layer = asp.AspLinear(to_dev_bf16(Wb), torch.from_numpy(U).cuda() if r else None, 64, fmt=fmt,
                          rotate=rotate)
    try:
        b = (np.random.default_rng(K + N).standard_normal(N) * 0.5).astype(np.float32)
        Y0 = run(layer, X).cpu().numpy()
        asp.qwam_asp_set_bias(layer.h, torch.from_numpy(b).cuda())
        Y1 = run(layer, X).cpu().numpy()
        np.testing.assert_array_equal(Y1.view(np.uint32), (Y0 + b[None, :]).astype(np.float32).view(np.uint32))
        Yb = run(layer, X, fp32=False)
        assert torch.equal(Yb.view(torch.int16), torch.from_numpy(Y1).cuda().to(torch.bfloat16).view(torch.int16))
        # against the oracle, rows whose output meets the bias-free bar keep it with the bias
        if fmt == asp.QWAM_FMT_NVFP4:
            Yo, _, _ = oracle.forward_nvfp4(Xb, Wb, U)
        elif rotate:
            Yo, _, _ = oracle.forward_rotated(Xb, Wb, None, U, 64)
        else:
            Yo, _, _ = oracle.forward(Xb, Wb, U, 64)
        ok = rowwise_rel_err(Y0, Yo) <= 1e-3
        assert ok.mean() >= 0.9
        Yob = Yo + b[None, :].astype(np.float64)
        d = np.abs(Y1 - Yob).max(axis=1)
        bound = 1e-3 * np.abs(Yo).max(axis=1) + 1e-6 * np.abs(Yob).max(axis=1)
        assert (d[ok] <= bound[ok]).all()
        asp.qwam_asp_set_bias(layer.h, None)
        np.testing.assert_array_equal(run(layer, X).cpu().numpy().view(np.uint32), Y0.view(np.uint32))
    finally:
        layer.close()


def test_set_bias_rejects_unaligned():
    c = Case(8, 256, 64, 0, 64, seed=1, layer_id=1)
    try:
        b = torch.zeros(65, dtype=torch.float32, device="cuda")
        with pytest.raises(asp.QwamError) as ei:
            asp.qwam_asp_set_bias(c.layer.h, b[1:])
        assert ei.value.status == asp.QWAM_ERR_INVALID_ARG
    finally:
        c.close()
