"""qwam_asp_linear_static (the layer on the library's static scratch workspace) against
qwam_asp_linear with a caller-provided workspace: same inputs, bit-identical outputs, over two
calls in a row, for both formats (rotated handles included); no device memory taken by the
static calls; and a clear error, before any launch, when the workspace would not fit.
Self-contained (no state from other test files), so it passes alone in a fresh process as well
as after the rest of the suite."""
from __future__ import annotations

import numpy as np
import pytest

pytestmark = pytest.mark.gpu


def _dev_bf16(bits):
    import torch
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).cuda().view(torch.bfloat16)


def _smoothing(K, seed):
    return np.exp(np.random.default_rng(seed).uniform(-1.0, 1.0, K)).astype(np.float32)


def _layer(K, N, r, G, fmt, rotate, seed=3):
    import torch
    from paper_2609_33269_gb300 import asp
    from paper_2609_33269_gb300 import workloads as wl
    W = _dev_bf16(wl.weight(K, N, seed=seed, layer_id=1))
    U = torch.from_numpy(wl.basis(K, r, seed=seed, layer_id=1)).cuda() if r else None
    s = torch.from_numpy(_smoothing(K, seed)).cuda() if rotate else None
    if fmt == "nvfp4":
        return asp.AspLinear(W, U, fmt=asp.QWAM_FMT_NVFP4, rotate=rotate, s=s)
    return asp.AspLinear(W, U, G, rotate=rotate, s=s)


CASES = [  # M, K, N, r, G, format, rotated
    (256, 512, 512, 16, 64, "int4", False),
    (33, 576, 200, 32, 32, "int4", False),
    (4096, 3072, 256, 32, 64, "int4", False),
    (256, 512, 512, 16, 0, "nvfp4", False),
    (4096, 3072, 256, 32, 0, "nvfp4", False),
    (64, 512, 256, 16, 64, "int4", True),
    (64, 512, 256, 16, 0, "nvfp4", True),
    (200, 1024, 136, 0, 0, "nvfp4", True),
]


@pytest.mark.parametrize("M,K,N,r,G,fmt,rot", CASES, ids=lambda v: str(v))
def test_static_workspace_matches_caller_workspace(M, K, N, r, G, fmt, rot):
    import torch
    from paper_2609_33269_gb300 import asp
    from paper_2609_33269_gb300 import workloads as wl
    layer = _layer(K, N, r, G, fmt, rot)
    try:
        assert asp.qwam_asp_act_workspace_bytes(layer.h, M) <= asp.STATIC_WS_BYTES
        # two calls in a row, each on fresh activations, each equal bit for bit to the
        # caller-workspace path (same kernels, same inputs)
        for call in range(2):
            X = _dev_bf16(wl.activations(M, K, seed=10 + call, layer_id=1))
            for fp32 in (True, False):
                ref = layer(X, fp32=fp32)
                out = torch.full_like(ref, float("nan"))
                asp.qwam_asp_linear_static(X, M, layer.h, out, asp.QWAM_Y_FP32 if fp32 else asp.QWAM_Y_BF16)
                torch.cuda.synchronize()
                assert asp.qwam_asp_get_error(layer.h) == asp.QWAM_OK
                assert torch.equal(out, ref), (call, fp32)
    finally:
        layer.close()


@pytest.mark.parametrize("fmt", ["int4", "nvfp4"])
def test_static_calls_take_no_device_memory(fmt):
    import torch
    from paper_2609_33269_gb300 import asp
    from paper_2609_33269_gb300 import workloads as wl
    M, K, N, r = 512, 1024, 384, 32
    layer = _layer(K, N, r, 64, fmt, False)
    try:
        X = _dev_bf16(wl.activations(M, K, seed=5, layer_id=2))
        Y = torch.empty((M, N), dtype=torch.float32, device="cuda")
        asp.qwam_asp_linear_static(X, M, layer.h, Y, asp.QWAM_Y_FP32)  # the first call looks the scratch up
        torch.cuda.synchronize()
        free0 = torch.cuda.mem_get_info()[0]
        for _ in range(4):
            asp.qwam_asp_linear_static(X, M, layer.h, Y, asp.QWAM_Y_FP32)
        torch.cuda.synchronize()
        assert torch.cuda.mem_get_info()[0] == free0
        assert asp.qwam_asp_get_error(layer.h) == asp.QWAM_OK
    finally:
        layer.close()


def _expect_too_large(layer, M, K, N):
    import torch
    from paper_2609_33269_gb300 import asp
    assert asp.qwam_asp_act_workspace_bytes(layer.h, M) > asp.STATIC_WS_BYTES
    X = torch.zeros((M, K), dtype=torch.bfloat16, device="cuda")
    Y = torch.zeros((M, N), dtype=torch.float32, device="cuda")
    with pytest.raises(asp.QwamError) as ei:
        asp.qwam_asp_linear_static(X, M, layer.h, Y, asp.QWAM_Y_FP32)
    assert ei.value.status == asp.QWAM_ERR_TOO_LARGE
    assert "static scratch" in str(ei.value)
    torch.cuda.synchronize()
    assert float(Y.abs().max()) == 0.0  # nothing ran


def test_static_workspace_rejects_oversize_before_launch():
    from paper_2609_33269_gb300 import asp
    K, N = 8192, 64
    layer = _layer(K, N, 0, 64, "int4", False, seed=4)
    try:
        _expect_too_large(layer, asp.STATIC_WS_BYTES // (K // 2) + 1, K, N)  # the packed codes alone
    finally:
        layer.close()


def test_static_workspace_rejects_rotated_remainder_at_dit_size():
    """A rotated handle with r > 0 keeps its float32 remainder (4 K bytes per token) in the
    workspace: at M = 4096, K = 3072 that is 50 MB, above the 24 MiB scratch."""
    layer = _layer(3072, 64, 32, 64, "int4", True, seed=6)
    try:
        _expect_too_large(layer, 4096, 3072, 64)
    finally:
        layer.close()
