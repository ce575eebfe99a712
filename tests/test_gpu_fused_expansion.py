"""The GEMM's float16 weights written by kernel (a) inside qwam_asp_linear (INT4 layers of 512 or
more tokens with r > 0) against the expansion launch that qwam_asp_gemm runs when called on its
own.

Bar: the two routes give bit-identical outputs (both write the same exact float16 values s_w 2^e_n c
and B_hat 2^e_n, and the GEMM launch is the same), for plain and rotated layers, with the
workspace cleared before each route so that neither can read what the other left; and a workspace
shared by two layers of the same shape, used alternately through both routes, always gives each
layer its own output (no GEMM reads the other layer's float16 weights).
"""
import pytest
import torch

from paper_2609_33269_gb300 import asp
from paper_2609_33269_gb300 import workloads as wl

from gpu_helpers import to_dev_bf16

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2609_33269_gb300 import build
    build.build()
    asp.load()


def make_layer(K, N, r, seed, rotate=False):
    Wb = wl.weight(K, N, seed=seed, layer_id=K)
    U = wl.basis(K, r, seed=seed, layer_id=K) if r else None
    return asp.AspLinear(to_dev_bf16(Wb), torch.from_numpy(U).cuda() if r else None, 64,
                         fmt=asp.QWAM_FMT_INT4, rotate=rotate)


def linear(layer, X, ws):
    M = X.shape[0]
    Y = torch.empty((M, layer.N), dtype=torch.float32, device="cuda")
    asp.qwam_asp_linear(X, M, layer.h, Y, asp.QWAM_Y_FP32, ws)
    torch.cuda.synchronize()
    return Y


def split(layer, X, ws):
    M = X.shape[0]
    Y = torch.empty((M, layer.N), dtype=torch.float32, device="cuda")
    asp.qwam_asp_quantize_act(X, M, layer.h, ws)
    asp.qwam_asp_gemm(ws, M, layer.h, Y, asp.QWAM_Y_FP32)
    torch.cuda.synchronize()
    return Y


def same_bits(a, b):
    return torch.equal(a.view(torch.int32), b.view(torch.int32))


@pytest.mark.parametrize("rotate", [False, True], ids=["plain", "rotated"])
@pytest.mark.parametrize("shape", [(600, 512, 264, 16), (1024, 1024, 520, 48), (4096, 3072, 3072, 32)],
                         ids=lambda s: "M%d_K%d_N%d_r%d" % s)
def test_linear_matches_separate_calls(shape, rotate):
    M, K, N, r = shape
    layer = make_layer(K, N, r, seed=29, rotate=rotate)
    try:
        X = to_dev_bf16(wl.activations(M, K, seed=29, layer_id=K, dist="outlier"))
        ws = layer.workspace(M)
        ws.zero_()
        Y_split = split(layer, X, ws)
        ws.zero_()
        Y_lin = linear(layer, X, ws)
        assert torch.isfinite(Y_lin).all()
        assert same_bits(Y_lin, Y_split)
    finally:
        layer.close()


@pytest.mark.parametrize("r_b", [0, 32], ids=["other_r0", "other_r32"])
def test_shared_workspace_alternating_layers(r_b):
    M, K, N = 1024, 1024, 768
    A = make_layer(K, N, 32, seed=31)
    B = make_layer(K, N, r_b, seed=37)
    try:
        X = to_dev_bf16(wl.activations(M, K, seed=41, layer_id=K, dist="outlier"))
        nbytes = max(asp.qwam_asp_act_workspace_bytes(A.h, M), asp.qwam_asp_act_workspace_bytes(B.h, M))
        ws = torch.zeros(nbytes, dtype=torch.uint8, device="cuda")
        # references, each on a workspace of its own
        Y_a = split(A, X, torch.zeros_like(ws))
        Y_b = split(B, X, torch.zeros_like(ws))
        assert not same_bits(Y_a, Y_b)
        for route_a, route_b in [(linear, linear), (linear, split), (split, linear), (split, split)]:
            assert same_bits(route_a(A, X, ws), Y_a)
            assert same_bits(route_b(B, X, ws), Y_b)
        # the GEMM alone on A's activations right after B's layer: its own expansion, A's weights
        asp.qwam_asp_quantize_act(X, M, A.h, ws)
        linear(B, X, torch.zeros_like(ws))  # B elsewhere, to interleave another layer's launches
        Y = torch.empty((M, N), dtype=torch.float32, device="cuda")
        asp.qwam_asp_gemm(ws, M, A.h, Y, asp.QWAM_Y_FP32)
        torch.cuda.synchronize()
        assert same_bits(Y, Y_a)
    finally:
        A.close()
        B.close()
