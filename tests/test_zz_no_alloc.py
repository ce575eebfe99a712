"""qwam_asp_linear_static (the layer on the library's static scratch workspace) against
qwam_asp_linear with a caller-provided workspace: same inputs, same outputs, over two calls in a
row, and a clear error when the workspace would not fit.  Self-contained (no state from other
test files), so it passes alone in a fresh process as well as after the rest of the suite."""
from __future__ import annotations

import numpy as np
import pytest

pytestmark = pytest.mark.gpu


def _dev_bf16(bits):
    import torch
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).cuda().view(torch.bfloat16)


@pytest.mark.parametrize("M,K,N,r,G", [(256, 512, 512, 16, 64), (33, 576, 200, 32, 32), (4096, 3072, 256, 32, 64)])
def test_static_workspace_matches_caller_workspace(M, K, N, r, G):
    import torch
    from paper_2609_33269_gb300 import asp
    from paper_2609_33269_gb300 import workloads as wl
    W = _dev_bf16(wl.weight(K, N, seed=3, layer_id=1))
    U = torch.from_numpy(wl.basis(K, r, seed=3, layer_id=1)).cuda() if r else None
    layer = asp.AspLinear(W, U, G)
    try:
        assert asp.qwam_asp_act_workspace_bytes(layer.h, M) <= asp.STATIC_WS_BYTES
        # two calls in a row, each on fresh activations, each checked against the caller-workspace path
        for call in range(2):
            X = _dev_bf16(wl.activations(M, K, seed=10 + call, layer_id=1))
            for fp32 in (True, False):
                ref = layer(X, fp32=fp32)
                out = torch.full_like(ref, float("nan"))
                asp.qwam_asp_linear_static(X, M, layer.h, out, asp.QWAM_Y_FP32 if fp32 else asp.QWAM_Y_BF16)
                torch.cuda.synchronize()
                assert asp.qwam_asp_get_error(layer.h) == asp.QWAM_OK
                r_ = ref.float()
                d = (out.float() - r_).abs().max().item()
                assert np.isfinite(d) and d <= 1e-6 * max(r_.abs().max().item(), 1e-30), (call, fp32, d)
    finally:
        layer.close()


def test_static_workspace_rejects_oversize_before_launch():
    import torch
    from paper_2609_33269_gb300 import asp
    from paper_2609_33269_gb300 import workloads as wl
    K, N = 8192, 64
    W = _dev_bf16(wl.weight(K, N, seed=4, layer_id=0))
    layer = asp.AspLinear(W, None, 64)
    try:
        M = asp.STATIC_WS_BYTES // (K // 2) + 1  # the packed codes alone exceed the scratch
        assert asp.qwam_asp_act_workspace_bytes(layer.h, M) > asp.STATIC_WS_BYTES
        X = torch.zeros((M, K), dtype=torch.bfloat16, device="cuda")
        Y = torch.zeros((M, N), dtype=torch.float32, device="cuda")
        with pytest.raises(asp.QwamError) as ei:
            asp.qwam_asp_linear_static(X, M, layer.h, Y, asp.QWAM_Y_FP32)
        assert ei.value.status == asp.QWAM_ERR_TOO_LARGE
        assert "static scratch" in str(ei.value)
        torch.cuda.synchronize()
        assert float(Y.abs().max()) == 0.0  # nothing ran
    finally:
        layer.close()
