"""CPU oracle for the offline choice of what ASP protects (Q-WAM Sec. 4.2 and 3.3; App. B.1).

TEST INFRASTRUCTURE ONLY, like the rest of ``oracle``: the tests and the smoke check load it; the
library never imports it.  Everything is float64 numpy; the one library routine used as a step is
the symmetric eigendecomposition ``numpy.linalg.eigh``.

The steps, in the paper's order and notation (d = the layer's input width, row-major W [d, d']):

* smoothing factor per input channel j (App. B.1): s_j = max|X_j|^alpha / max|W_j,:|^(1 - alpha),
  with max|X_j| the channel's calibration maximum and max|W_j,:| the largest weight of that input
  channel (the row of W that multiplies x_j here, the paper's "matching weight column");
* block Hadamard rotation H (Sec. 3 Eq. (pair); App. B.1): block-diagonal, each block the
  Sylvester Hadamard matrix of size B divided by sqrt(B), B the largest power of two that divides
  d, at most 1024.  H is symmetric and orthogonal;
* the AOG in the rotated coordinates (Sec. 4.2): G~ = H diag(gamma) G diag(gamma) H;
* the action subspace (Sec. 4.2, Eq. (gtilde)): the eigenvectors of the r largest eigenvalues of
  G~, which the Ky Fan maximum principle (App. A) makes the best rank-r protection;
* the action mass of an expert E (Sec. 4.3, Eq. (mass)): mu_E = sum over its layers of tr G~;
* which experts to protect (Sec. 4.3): those with the largest action mass per added 16-bit value,
  read here as a greedy choice in decreasing mu_E / c_E while the added values fit a budget
  (c_E = the 16-bit values the branches of E add, r (d + d') per layer).
"""
from __future__ import annotations

import numpy as np


def hadamard_block_size(d: int) -> int:
    """The largest power of two that divides d, capped at 1024 (App. B.1)."""
    b = 1
    while d % (2 * b) == 0 and 2 * b <= 1024:
        b *= 2
    return b


def sylvester(b: int) -> np.ndarray:
    """The b x b Sylvester Hadamard matrix (entries +-1), b a power of two."""
    h = np.ones((1, 1))
    while h.shape[0] < b:
        h = np.block([[h, h], [h, -h]])
    return h


def block_hadamard(d: int) -> np.ndarray:
    """The rotation H of Eq. (pair): block diagonal with blocks sylvester(B) / sqrt(B)."""
    b = hadamard_block_size(d)
    return np.kron(np.eye(d // b), sylvester(b) / np.sqrt(b))


def smoothing_factors(xmax: np.ndarray, W: np.ndarray, alpha: float = 0.5) -> np.ndarray:
    """App. B.1: s_j = max|X_j|^alpha / max|W_j,:|^(1 - alpha) for W [d, d'] (row j = channel j).
    A channel whose activation or weight maximum is zero carries nothing and is left unsmoothed
    (s_j = 1): the factor is undefined there and the paper does not say."""
    wmax = np.abs(np.asarray(W, np.float64)).max(axis=1)
    xm = np.asarray(xmax, np.float64)
    ok = (xm > 0) & (wmax > 0)
    s = np.ones_like(xm)
    s[ok] = xm[ok] ** alpha / wmax[ok] ** (1.0 - alpha)
    return s


def rotated_gramian(G: np.ndarray, gamma: np.ndarray | None = None) -> np.ndarray:
    """Sec. 4.2: G~ = H diag(gamma) G diag(gamma) H (gamma = 1 when None)."""
    G = np.asarray(G, np.float64)
    d = G.shape[0]
    g = np.ones(d) if gamma is None else np.asarray(gamma, np.float64)
    H = block_hadamard(d)
    return H @ (g[:, None] * G * g[None, :]) @ H


def action_subspace(Gt: np.ndarray, r: int):
    """Sec. 4.2: the top-r eigenvectors V [d, r] (columns in decreasing eigenvalue order) and the
    eigenvalues lambda_1 >= ... >= lambda_r of the symmetric matrix G~."""
    w, Q = np.linalg.eigh(np.asarray(Gt, np.float64))
    order = np.argsort(w)[::-1][:r]
    return Q[:, order], w[order]


def action_mass(gramians) -> float:
    """Sec. 4.3 Eq. (mass): mu_E = sum of tr G~ over the layers of the expert."""
    return float(sum(np.trace(np.asarray(g, np.float64)) for g in gramians))


def branch_cost(shapes, r: int) -> int:
    """16-bit values the rank-r branches of an expert add: V [d, r] and V^T W~ [r, d'] per layer."""
    return int(sum(r * (d + dp) for d, dp in shapes))


def select_experts(masses, costs, budget: float):
    """Sec. 4.3: protect in decreasing order of action mass per added 16-bit value, while the added
    values fit the budget; an expert that does not fit is skipped and the next one is tried.
    Returns the indices chosen, in the order chosen."""
    order = sorted(range(len(masses)), key=lambda i: (-masses[i] / costs[i], i))
    chosen, used = [], 0.0
    for i in order:
        if used + costs[i] <= budget:
            chosen.append(i)
            used += costs[i]
    return chosen
