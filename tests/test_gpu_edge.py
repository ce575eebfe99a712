"""GPU edge cases of the activation quantizer and the boundary, against the CPU oracle.

* Groups whose absmax is tiny -- down to float32 subnormal scales -- and all-zero groups: with
  r = 0 the remainder is X itself, so scales and codes must equal the oracle's bit for bit
  (Eq. (quant) with the stored scale; a zero scale gives zero codes).  The kernel takes a
  different internal route for scales below 2^-100; this covers it.
* An empty input (M = 0) is accepted and launches nothing, in both formats, with and without the
  rotation.
* Both activation kernels (the small-M one and kernel (a)) take the tiny-group cases.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_33269_gb300 import asp
from paper_2609_33269_gb300 import workloads as wl

from gpu_helpers import Case, rowwise_rel_err

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2609_33269_gb300 import build
    build.build()
    asp.load()


def _tiny_rows(M, K, seed):
    """bf16 bits [M, K]: N(0,1) rows scaled by factors from 1 down to the bf16 subnormal range,
    plus an all-zero row and a row whose groups alternate between zero and tiny values."""
    g = np.random.default_rng(seed)
    x = g.standard_normal((M, K)).astype(np.float32)
    factors = [1.0, 1e-20, 1e-30, 2.0 ** -100, 1e-31, 1e-35, 1e-37, 1e-38, 3e-39, 1e-39, 0.0]
    for i in range(M):
        x[i] *= np.float32(factors[i % len(factors)])
    x[M - 1, ::2] = 0.0
    x[M - 1, 1::2] *= np.float32(1e-38)
    return wl.f32_to_bf16_bits(x)


@pytest.mark.parametrize("small", [256, 0], ids=["small_m", "kernel_a"])
@pytest.mark.parametrize("G", [32, 64])
def test_tiny_and_zero_groups_bit_exact_r0(G, small):
    M, K, N = 24, 512, 128
    c = Case(M, K, N, 0, G, seed=5, layer_id=7, Xb=_tiny_rows(M, K, seed=G))
    try:
        asp.qwam_asp_set_small_m(c.layer.h, small)
        c.layer.quantize(c.X)
        ga = c.gpu_act()
        oa = c.oracle_act(want_float64=False)
        np.testing.assert_array_equal(ga["sx"].view(np.uint32), oa["sx"].view(np.uint32))
        np.testing.assert_array_equal(ga["qx"], oa["qx"])
        assert (ga["qx"][ga["sx"].repeat(G, axis=1) == 0] == 0).all()  # zero scale -> zero codes
        # the layer output, row by row, against the oracle on the same codes
        Y = c.run(fp32=True).cpu().numpy()
        ow = c.oracle_weights()
        Yo = oracle.linear(oa, ow, G)
        nz = np.abs(Yo).max(axis=1) > 0
        assert rowwise_rel_err(Y[nz], Yo[nz]).max() <= 1e-5
        assert np.all(Y[~nz] == 0)
    finally:
        c.close()


@pytest.mark.parametrize("kind", ["int4", "nvfp4", "int4_rotated", "nvfp4_rotated"])
def test_empty_input_launches_nothing(kind):
    K, N, G = 256, 64, 64
    W = torch.from_numpy(wl.weight(K, N, seed=1, layer_id=0).view(np.int16)).cuda().view(torch.bfloat16)
    fmt = asp.QWAM_FMT_NVFP4 if kind.startswith("nvfp4") else asp.QWAM_FMT_INT4
    layer = asp.AspLinear(W, None, G, fmt=fmt, rotate=kind.endswith("rotated"))
    try:
        X = torch.empty((0, K), dtype=torch.bfloat16, device="cuda")
        Y = torch.empty((0, N), dtype=torch.float32, device="cuda")
        ws = torch.zeros(16, dtype=torch.uint8, device="cuda")
        asp.qwam_asp_quantize_act(X, 0, layer.h, ws)
        asp.qwam_asp_gemm(ws, 0, layer.h, Y, asp.QWAM_Y_FP32)
        asp.qwam_asp_linear(X, 0, layer.h, Y, asp.QWAM_Y_FP32, ws)
        torch.cuda.synchronize()
        assert asp.qwam_asp_get_error(layer.h) == asp.QWAM_OK
        assert int(ws.sum()) == 0
    finally:
        layer.close()
