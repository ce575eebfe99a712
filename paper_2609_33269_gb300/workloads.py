"""Seeded synthetic inputs for the ASP linear layer, shared by the tests, the smoke check and the
benchmark.

This module draws inputs only; it holds none of the layer's arithmetic.  The paper measures on
trained World Action Models over RoboTwin 2.0, which are not available here; these generators
stand in for its DiT / action-expert linear layers (shapes of Sec. 5 and App. B.1: rank r = 32,
group-wise 4-bit quantization).  Every array comes from NumPy's PCG64 seeded with
``[seed, layer_id, step]`` so that both sides of a comparison see the same bytes.

Recipe (also stated in the design notes):
  X  token activations, bf16 [M, K]: N(0, 1), with a seeded set of outlier channels scaled by a
     factor drawn from U(lo, hi) (1% of channels, x10..30), or Student-t(nu=4) for the input of
     an FFN down projection (heavy-tailed, GELU-like).
  W  weight, bf16 [K, N]: N(0, 1/K).
  U  orthonormal basis [K, r] float32: Q factor of a Householder QR (float64) of a seeded
     N(0, 1) [K, r] matrix, column signs chosen so that diag(R) > 0.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np


def f32_to_bf16_bits(a: np.ndarray) -> np.ndarray:
    """float32 -> bfloat16 bit patterns (uint16), round to nearest even (finite inputs)."""
    u = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32)
    bias = ((u >> 16) & 1) + np.uint32(0x7FFF)
    return ((u + bias) >> 16).astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def rng(seed: int, layer_id: int = 0, step: int = 0) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64([seed, layer_id, step]))


def activations(M: int, K: int, *, seed: int, layer_id: int = 0, step: int = 0,
                dist: str = "outlier", n_outlier: int | None = None,
                outlier_lo: float = 10.0, outlier_hi: float = 30.0) -> np.ndarray:
    """bf16 bits [M, K].  dist: 'outlier' (N(0,1) with scaled outlier channels) or 'student_t'."""
    g = rng(seed, layer_id, step)
    if dist == "student_t":
        x = g.standard_t(4.0, size=(M, K)).astype(np.float32)
    elif dist == "outlier":
        x = g.standard_normal((M, K), dtype=np.float32)
        n_out = max(1, K // 100) if n_outlier is None else n_outlier
        if n_out:
            ch = g.choice(K, size=n_out, replace=False)
            factor = (g.uniform(outlier_lo, outlier_hi, size=n_out).astype(np.float32)
                      if outlier_hi > outlier_lo else np.full(n_out, outlier_lo, np.float32))
            x[:, ch] *= factor
    elif dist == "normal":
        x = g.standard_normal((M, K), dtype=np.float32)
    else:
        raise ValueError(dist)
    return f32_to_bf16_bits(x)


def weight(K: int, N: int, *, seed: int, layer_id: int = 0) -> np.ndarray:
    """bf16 bits [K, N] drawn from N(0, 1/K)."""
    g = rng(seed, layer_id, 1_000_003)
    w = (g.standard_normal((K, N), dtype=np.float32) * np.float32(1.0 / np.sqrt(K)))
    return f32_to_bf16_bits(w)


def basis(K: int, r: int, *, seed: int, layer_id: int = 0) -> np.ndarray:
    """float32 [K, r] with orthonormal columns (empty [K, 0] for r == 0)."""
    if r == 0:
        return np.zeros((K, 0), np.float32)
    g = rng(seed, layer_id, 2_000_003)
    a = g.standard_normal((K, r))
    q, rr = np.linalg.qr(a)
    q = q * np.sign(np.diag(rr))[None, :]
    return q.astype(np.float32)


@dataclass
class Layer:
    """One linear layer of a workload."""
    name: str
    M: int
    K: int
    N: int
    r: int
    G: int = 64
    dist: str = "outlier"
    n_outlier: int | None = None
    outlier_lo: float = 10.0
    outlier_hi: float = 30.0
    seed: int = 0
    layer_id: int = 0

    @property
    def flops(self) -> float:
        return 2.0 * self.M * self.N * self.K

    def x(self, step: int = 0) -> np.ndarray:
        return activations(self.M, self.K, seed=self.seed, layer_id=self.layer_id, step=step,
                           dist=self.dist, n_outlier=self.n_outlier,
                           outlier_lo=self.outlier_lo, outlier_hi=self.outlier_hi)

    def w(self) -> np.ndarray:
        return weight(self.K, self.N, seed=self.seed, layer_id=self.layer_id)

    def u(self) -> np.ndarray:
        return basis(self.K, self.r, seed=self.seed, layer_id=self.layer_id)


@dataclass
class Workload:
    name: str
    layers: list = field(default_factory=list)
    steps: int = 1
    note: str = ""


def tiny() -> Workload:
    """Single ASP linear, M=256, K=N=512, r=16, G=64, 8 outlier channels x20, seed 0."""
    return Workload("asp_linear_tiny_M256_K512_N512_r16_g64",
                    [Layer("tiny", 256, 512, 512, 16, 64, "outlier", n_outlier=8,
                           outlier_lo=20.0, outlier_hi=20.0, seed=0)])


def dit_attention() -> Workload:
    """DiT attention projection: M=4096 tokens, K=N=3072, r=32, G=64, 1% outlier channels x10..30."""
    return Workload("dit_attn_proj_M4096_K3072_N3072_r32_g64",
                    [Layer("attn_proj", 4096, 3072, 3072, 32, 64, "outlier", seed=0, layer_id=1)])


def dit_ffn() -> Workload:
    """DiT FFN pair at M=4096: up 3072->12288 (outlier inputs), down 12288->3072 (Student-t)."""
    return Workload("dit_ffn_M4096_3072x12288_r32_g64",
                    [Layer("ffn_up", 4096, 3072, 12288, 32, 64, "outlier", seed=0, layer_id=2),
                     Layer("ffn_down", 4096, 12288, 3072, 32, 64, "student_t", seed=0, layer_id=3)])


def action_expert_small_m() -> Workload:
    """Action-expert small-M path: M in {32,64,128}, 1024->1024 and 1024->4096, r in {16, 0}."""
    layers = []
    lid = 10
    for M in (32, 64, 128):
        for N in (1024, 4096):
            for r in (16, 0):
                layers.append(Layer(f"act_M{M}_N{N}_r{r}", M, 1024, N, r, 64, "outlier", seed=0, layer_id=lid))
                lid += 1
    return Workload("action_expert_smallM_K1024", layers)


def denoise_sweep(blocks: int = 30, steps: int = 10) -> Workload:
    """30 DiT blocks x {qkv 3072->9216, o 3072->3072, up 3072->12288, down 12288->3072} at M=4096;
    ASP (r=32) on a seeded third of the blocks, r=0 elsewhere; fresh activations every step."""
    asp_blocks = set(np.random.Generator(np.random.PCG64(0)).choice(blocks, blocks // 3, replace=False).tolist())
    layers = []
    for b in range(blocks):
        r = 32 if b in asp_blocks else 0
        base = 100 + 4 * b
        layers += [Layer(f"b{b}_qkv", 4096, 3072, 9216, r, 64, "outlier", seed=0, layer_id=base),
                   Layer(f"b{b}_o", 4096, 3072, 3072, r, 64, "outlier", seed=0, layer_id=base + 1),
                   Layer(f"b{b}_up", 4096, 3072, 12288, r, 64, "outlier", seed=0, layer_id=base + 2),
                   Layer(f"b{b}_down", 4096, 12288, 3072, r, 64, "student_t", seed=0, layer_id=base + 3)]
    return Workload("denoise_sweep_30blocks_M4096", layers, steps=steps,
                    note=f"ASP blocks {sorted(asp_blocks)}")


ALL = {
    "tiny": tiny,
    "dit_attn": dit_attention,
    "dit_ffn": dit_ffn,
    "small_m": action_expert_small_m,
    "sweep": denoise_sweep,
}
