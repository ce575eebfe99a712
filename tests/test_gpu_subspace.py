"""GPU parity of the offline choice of what ASP protects (Sec. 4.2-4.3; App. A; App. B.1) against
the float64 oracle (oracle/subspace.py), through the C ABI: smoothing factors, the rotated AOG
G~ = H diag(gamma) G diag(gamma) H, its trace, and its top-r eigenvectors; and a layer packed with
the subspace the GPU chose.

Bars: float32 arithmetic against float64, so relative to the largest entry (G~: 2e-6 of max |G~|),
eigenvalues to 1e-4 relative plus 1e-5 of the largest, and the subspace through its projector (max |VV^T - V_o V_o^T| <=
1e-3) and orthonormality (|V^T V - I| <= 1e-5)."""
import numpy as np
import pytest
import torch

import oracle
from oracle import subspace as sub
from paper_2609_33269_gb300 import asp
from paper_2609_33269_gb300 import workloads as wl

from gpu_helpers import rowwise_rel_err, to_dev_bf16

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2609_33269_gb300 import build
    build.build()
    asp.load()


def psd(rng, d, decay=None, gap_at=None):
    """A symmetric positive semidefinite matrix with a chosen spectrum: Q diag(lam) Q^T."""
    Q, _ = np.linalg.qr(rng.standard_normal((d, d)))
    lam = 10.0 ** (-np.arange(d) / decay) if decay else np.sort(rng.exponential(1.0, d))[::-1]
    if gap_at:
        lam[gap_at:] *= 0.05
    return ((Q * lam) @ Q.T).astype(np.float32), lam


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


@pytest.mark.parametrize("K,N,alpha", [(256, 96, 0.5), (1024, 300, 0.3), (96, 40, 1.0)])
def test_smoothing_factors(K, N, alpha):
    rng = np.random.default_rng(K)
    Wb = wl.weight(K, N, seed=3, layer_id=K)
    xmax = np.exp(rng.uniform(-3, 4, K)).astype(np.float32)
    xmax[5] = 0.0                                 # a dead channel: left unsmoothed
    W = to_dev_bf16(Wb)
    s = torch.empty(K, dtype=torch.float32, device="cuda")
    asp.qwam_asp_smoothing_factors(dev(xmax), W, K, N, alpha, s)
    torch.cuda.synchronize()
    want = sub.smoothing_factors(xmax.astype(np.float64), wl.bf16_bits_to_f32(Wb), alpha).astype(np.float32)
    got = s.cpu().numpy()
    assert got[5] == 1.0
    np.testing.assert_allclose(got, want, rtol=3e-7)


@pytest.mark.parametrize("d", [96, 640, 3072, 80, 7])
def test_rotated_gramian_and_trace(d):
    rng = np.random.default_rng(d)
    G, _ = psd(rng, d)
    gamma = np.exp(rng.uniform(-1, 1, d)).astype(np.float32)
    Gd, Gt, work = dev(G), torch.empty((d, d), dtype=torch.float32, device="cuda"), torch.empty((d, d), dtype=torch.float32, device="cuda")
    asp.qwam_asp_rotated_gramian(Gd, dev(gamma), d, Gt, work)
    torch.cuda.synchronize()
    want = sub.rotated_gramian(G.astype(np.float64), gamma.astype(np.float64))
    got = Gt.cpu().numpy()
    assert np.abs(got - want).max() <= 2e-6 * np.abs(want).max() * max(1.0, np.log2(d))
    tr = asp.qwam_asp_gramian_trace(Gt, d)
    assert tr == pytest.approx(np.trace(want), rel=1e-5)
    # without smoothing: H G H
    asp.qwam_asp_rotated_gramian(Gd, None, d, Gt, work)
    torch.cuda.synchronize()
    want0 = sub.rotated_gramian(G.astype(np.float64))
    assert np.abs(Gt.cpu().numpy() - want0).max() <= 2e-6 * np.abs(want0).max() * max(1.0, np.log2(d))


@pytest.mark.parametrize("d,r,spec", [(256, 16, "decay"), (1024, 32, "gap"), (3072, 32, "decay"), (512, 64, "gap"),
                                      (40, 32, "gap")])
def test_action_subspace_against_the_oracle(d, r, spec):
    rng = np.random.default_rng(d + r)
    if spec == "decay":  # eigenvalues fall by orders of magnitude within a few dozen directions
        G, lam = psd(rng, d, decay=10.0)
    else:
        G, lam = psd(rng, d, gap_at=r)
    Vo, wo = sub.action_subspace(G.astype(np.float64), r)
    Gd = dev(G)
    V = torch.empty((d, r), dtype=torch.float32, device="cuda")
    w = torch.empty(r, dtype=torch.float32, device="cuda")
    work = torch.empty(asp.qwam_asp_subspace_workspace_bytes(d, r), dtype=torch.uint8, device="cuda")
    asp.qwam_asp_action_subspace(Gd, d, r, 40, V, w, work)
    Vg, wg = V.cpu().numpy().astype(np.float64), w.cpu().numpy().astype(np.float64)
    np.testing.assert_allclose(wg, wo, rtol=1e-4, atol=1e-5 * wo[0])
    assert np.abs(Vg.T @ Vg - np.eye(r)).max() <= 1e-5
    assert np.abs(Vg @ Vg.T - Vo @ Vo.T).max() <= 1e-3
    # the Ky Fan value: tr(V^T G~ V) equals the sum of the r largest eigenvalues
    assert np.trace(Vg.T @ G.astype(np.float64) @ Vg) == pytest.approx(wo.sum(), rel=1e-4)


def test_layer_runs_with_the_subspace_the_gpu_chose():
    """End to end at a small size: G -> G~ (with smoothing) -> V on the GPU; the layer packed with
    U = V matches the oracle's layer with the same U."""
    d, N, M, r = 512, 384, 200, 16
    rng = np.random.default_rng(9)
    G, _ = psd(rng, d, decay=8.0)
    gamma = np.exp(rng.uniform(-0.5, 0.5, d)).astype(np.float32)
    Gt = torch.empty((d, d), dtype=torch.float32, device="cuda")
    work = torch.empty((d, d), dtype=torch.float32, device="cuda")
    asp.qwam_asp_rotated_gramian(dev(G), dev(gamma), d, Gt, work)
    V = torch.empty((d, r), dtype=torch.float32, device="cuda")
    w = torch.empty(r, dtype=torch.float32, device="cuda")
    ws = torch.empty(asp.qwam_asp_subspace_workspace_bytes(d, r), dtype=torch.uint8, device="cuda")
    asp.qwam_asp_action_subspace(Gt, d, r, 40, V, w, ws)
    U = V.cpu().numpy()
    Xb = wl.activations(M, d, seed=9, layer_id=1)
    Wb = wl.weight(d, N, seed=9, layer_id=1)
    layer = asp.AspLinear(to_dev_bf16(Wb), V.contiguous(), 64)
    try:
        Y = layer(to_dev_bf16(Xb), fp32=True)
        torch.cuda.synchronize()
        Yo, _, _ = oracle.forward(Xb, Wb, U, 64)
        assert rowwise_rel_err(Y.cpu().numpy(), Yo).max() <= 1e-3
    finally:
        layer.close()


def test_subspace_argument_checks():
    with pytest.raises(asp.QwamError):
        asp.qwam_asp_subspace_workspace_bytes(64, 100)   # r above the 96-vector limit
    with pytest.raises(asp.QwamError):
        asp.qwam_asp_subspace_workspace_bytes(16, 32)    # r above d
    A = torch.zeros((8, 8), dtype=torch.float32, device="cuda")
    with pytest.raises(asp.QwamError):
        asp.qwam_asp_rotated_gramian(A, None, 8, A, A)   # aliasing buffers
