"""Pins of the oracle's offline subspace choice (oracle/subspace.py: Sec. 4.2-4.3, App. A, App. B.1)
against definitions written out here: the Hadamard matrix from its bit formula and from the
butterfly recursion, known spectra, the Ky Fan maximum principle checked against random frames,
the trace and cost identities of the rotation, the smoothing factor's closed forms, and a
hand-worked expert selection."""
from __future__ import annotations

import numpy as np
import pytest

from oracle import subspace as sub


def hadamard_bits(b: int) -> np.ndarray:
    """H[i, j] = (-1)^popcount(i & j): the Sylvester matrix, from its closed form."""
    i = np.arange(b)[:, None]
    j = np.arange(b)[None, :]
    pc = np.vectorize(lambda v: bin(int(v)).count("1"))(i & j)
    return np.where(pc % 2 == 0, 1.0, -1.0)


def fwht(v: np.ndarray, b: int) -> np.ndarray:
    """Block fast Walsh-Hadamard transform (butterflies), normalised by 1/sqrt(b), along the last
    axis in blocks of b."""
    v = np.array(v, np.float64)
    shape = v.shape
    v = v.reshape(-1, b)
    h = 1
    while h < b:
        v = v.reshape(-1, b // (2 * h), 2, h)
        a, c = v[:, :, 0, :].copy(), v[:, :, 1, :].copy()
        v[:, :, 0, :], v[:, :, 1, :] = a + c, a - c
        v = v.reshape(-1, b)
        h *= 2
    return (v / np.sqrt(b)).reshape(shape)


def random_orthonormal(rng, d, r):
    q, _ = np.linalg.qr(rng.standard_normal((d, r)))
    return q


@pytest.mark.parametrize("d,b", [(3072, 1024), (12288, 1024), (1024, 1024), (2048, 1024), (96, 32),
                                 (80, 16), (7, 1), (640, 128)])
def test_hadamard_block_size(d, b):
    assert sub.hadamard_block_size(d) == b


@pytest.mark.parametrize("b", [1, 2, 8, 64])
def test_sylvester_matches_bit_formula(b):
    np.testing.assert_array_equal(sub.sylvester(b), hadamard_bits(b))
    np.testing.assert_array_equal(sub.sylvester(b) @ sub.sylvester(b).T, b * np.eye(b))


@pytest.mark.parametrize("d", [96, 640, 3072])
def test_block_hadamard_is_symmetric_orthogonal_and_the_fwht(d):
    H = sub.block_hadamard(d)
    np.testing.assert_allclose(H, H.T, atol=0)
    np.testing.assert_allclose(H @ H, np.eye(d), atol=1e-12)
    rng = np.random.default_rng(d)
    x = rng.standard_normal((3, d))
    np.testing.assert_allclose(x @ H, fwht(x, sub.hadamard_block_size(d)), atol=1e-12)


def test_smoothing_factor_closed_forms_and_exactness():
    rng = np.random.default_rng(1)
    d, dp = 64, 24
    W = rng.standard_normal((d, dp))
    xmax = np.exp(rng.uniform(-2, 3, d))
    wmax = np.abs(W).max(axis=1)
    np.testing.assert_allclose(sub.smoothing_factors(xmax, W, 0.5), np.sqrt(xmax / wmax), rtol=1e-14)
    np.testing.assert_allclose(sub.smoothing_factors(xmax, W, 1.0), xmax, rtol=1e-14)
    np.testing.assert_allclose(sub.smoothing_factors(xmax, W, 0.0), 1.0 / wmax, rtol=1e-14)
    # a channel with a zero maximum is left unsmoothed
    W0 = W.copy()
    W0[3] = 0.0
    xm0 = xmax.copy()
    xm0[5] = 0.0
    s0 = sub.smoothing_factors(xm0, W0, 0.5)
    assert s0[3] == 1.0 and s0[5] == 1.0
    np.testing.assert_allclose(np.delete(s0, [3, 5]), np.delete(np.sqrt(xm0 / np.abs(W0).max(axis=1).clip(1e-300)), [3, 5]),
                               rtol=1e-14)
    # Eq. (pair): x~ = H diag(s)^-1 x and W~ = H diag(s) W leave W^T x unchanged
    s = sub.smoothing_factors(xmax, W, 0.5)
    H = sub.block_hadamard(d)
    x = rng.standard_normal(d) * xmax
    xt, Wt = H @ (x / s), H @ (s[:, None] * W)
    np.testing.assert_allclose(Wt.T @ xt, W.T @ x, rtol=1e-12, atol=1e-12)


def test_rotated_gramian_identities():
    rng = np.random.default_rng(2)
    d = 96
    A = rng.standard_normal((d, 2 * d))
    G = A @ A.T / d
    gamma = np.exp(rng.uniform(-1, 1, d))
    Gt = sub.rotated_gramian(G, gamma)
    np.testing.assert_allclose(Gt, Gt.T, atol=1e-12)
    # the trace is that of diag(gamma) G diag(gamma): sum_j gamma_j^2 G_jj
    np.testing.assert_allclose(np.trace(Gt), np.sum(gamma ** 2 * np.diag(G)), rtol=1e-12)
    # a rounding error delta of x~ moves x by diag(gamma) H delta and costs delta^T G~ delta
    S = np.diag(gamma) @ sub.block_hadamard(d)
    for _ in range(5):
        delta = rng.standard_normal(d)
        xs = S @ delta
        np.testing.assert_allclose(delta @ Gt @ delta, xs @ G @ xs, rtol=1e-12)
    # positive semidefinite
    assert np.linalg.eigvalsh(Gt).min() > -1e-10


@pytest.mark.parametrize("d,r", [(64, 8), (128, 32)])
def test_action_subspace_recovers_a_known_spectrum(d, r):
    rng = np.random.default_rng(d + r)
    Q = random_orthonormal(rng, d, d)
    lam = np.sort(10.0 ** rng.uniform(-3, 2, d))[::-1]
    lam[r:] *= 0.1  # a clear gap after the r-th eigenvalue
    G = (Q * lam) @ Q.T
    V, w = sub.action_subspace(G, r)
    np.testing.assert_allclose(w, lam[:r], rtol=1e-10)
    np.testing.assert_allclose(V.T @ V, np.eye(r), atol=1e-12)
    np.testing.assert_allclose(V @ V.T, Q[:, :r] @ Q[:, :r].T, atol=1e-9)
    assert np.all(np.diff(w) <= 0)


def test_ky_fan_top_eigenvectors_are_the_best_rank_r_protection():
    """App. A: over V with orthonormal columns, tr(V^T G~ V) is at most the sum of the r largest
    eigenvalues and the top-r eigenvectors attain it; so the residual damage tr((I - VV^T) G~) is
    least for them and equals the sum of the remaining eigenvalues."""
    rng = np.random.default_rng(3)
    d, r = 48, 6
    A = rng.standard_normal((d, d)) * np.exp(-np.arange(d) / 6.0)[None, :]
    Gt = A @ A.T
    V, w = sub.action_subspace(Gt, r)
    top = np.sort(np.linalg.eigvalsh(Gt))[::-1]
    best = np.trace(V.T @ Gt @ V)
    np.testing.assert_allclose(best, top[:r].sum(), rtol=1e-12)
    np.testing.assert_allclose(np.trace(Gt) - best, top[r:].sum(), rtol=1e-9)
    for _ in range(200):
        P = random_orthonormal(rng, d, r)
        assert np.trace(P.T @ Gt @ P) <= best * (1 + 1e-12)


def test_action_mass_is_the_sum_of_traces_and_rotation_invariant():
    rng = np.random.default_rng(4)
    gs = []
    for d in (32, 64, 96):
        A = rng.standard_normal((d, d))
        gs.append(A @ A.T)
    assert sub.action_mass(gs) == pytest.approx(sum(np.trace(g) for g in gs), rel=1e-14)
    assert sub.action_mass([sub.rotated_gramian(g) for g in gs]) == pytest.approx(sub.action_mass(gs), rel=1e-12)


def test_expert_selection_by_mass_per_added_value():
    # branch cost r (d + d') per layer
    assert sub.branch_cost([(1024, 1024), (1024, 4096)], 16) == 16 * (2048 + 5120)
    masses = [89.3, 10.0, 0.7]
    costs = [100.0, 400.0, 10.0]
    # ratios 0.893, 0.025, 0.07 -> order 0, 2, 1
    assert sub.select_experts(masses, costs, 110.0) == [0, 2]
    assert sub.select_experts(masses, costs, 509.0) == [0, 2]      # expert 1 does not fit
    assert sub.select_experts(masses, costs, 510.0) == [0, 2, 1]
    assert sub.select_experts(masses, costs, 50.0) == [2]          # 0 does not fit, 2 does
    assert sub.select_experts(masses, costs, 0.0) == []
    assert sub.select_experts([1.0, 2.0], [1.0, 2.0], 1.5) == [0]  # equal ratios: lower index first
