"""The synthetic input recipe (CPU): the workload shapes and the statistics of the seeded inputs
that stand in for the paper's DiT / action-expert activations, weights and protected bases.

Checks what the recipe promises, independently of how it draws: the shapes of the five
workloads, the fraction and scale of the outlier channels, the N(0, 1/K) weights, the heavy tails
of the Student-t(4) inputs, orthonormal bases, the third of the sweep's blocks that carries ASP,
and that the same seed gives the same bytes.
"""
import numpy as np

from paper_2609_33269_gb300 import workloads as wl


def test_workload_shapes():
    t = wl.tiny().layers
    assert [(L.M, L.K, L.N, L.r, L.G) for L in t] == [(256, 512, 512, 16, 64)]
    a = wl.dit_attention().layers
    assert [(L.M, L.K, L.N, L.r, L.G) for L in a] == [(4096, 3072, 3072, 32, 64)]
    f = wl.dit_ffn().layers
    assert [(L.M, L.K, L.N, L.r, L.dist) for L in f] == [(4096, 3072, 12288, 32, "outlier"),
                                                          (4096, 12288, 3072, 32, "student_t")]
    s = wl.action_expert_small_m().layers
    assert sorted({L.M for L in s}) == [32, 64, 128] and {L.K for L in s} == {1024}
    assert {L.N for L in s} == {1024, 4096} and {L.r for L in s} == {0, 16}
    sw = wl.denoise_sweep()
    assert len(sw.layers) == 120 and sw.steps == 10
    kinds = [(L.K, L.N) for L in sw.layers[:4]]
    assert kinds == [(3072, 9216), (3072, 3072), (3072, 12288), (12288, 3072)]
    asp_blocks = {i // 4 for i, L in enumerate(sw.layers) if L.r == 32}
    assert len(asp_blocks) == 10 and all(L.r in (0, 32) for L in sw.layers)
    # every layer of a block has the same rank
    for b in range(30):
        assert len({L.r for L in sw.layers[4 * b:4 * b + 4]}) == 1


def test_outlier_channels_fraction_and_scale():
    M, K = 512, 3072
    x = wl.bf16_bits_to_f32(wl.activations(M, K, seed=3, layer_id=1)).astype(np.float64)
    rms = np.sqrt((x ** 2).mean(axis=0))
    out = rms > 5.0
    assert out.sum() == K // 100                      # 1 % of the channels
    assert 8.0 < rms[out].min() and rms[out].max() < 33.0  # scaled x10 .. x30
    assert 0.9 < np.median(rms[~out]) < 1.1           # the rest N(0, 1)


def test_weights_and_student_t_inputs():
    K, N = 3072, 512
    w = wl.bf16_bits_to_f32(wl.weight(K, N, seed=1, layer_id=2)).astype(np.float64)
    assert abs(w.std() * np.sqrt(K) - 1.0) < 0.02 and abs(w.mean()) < 1e-3
    x = wl.bf16_bits_to_f32(wl.activations(256, 4096, seed=1, layer_id=3, dist="student_t")).astype(np.float64)
    # t(4): variance nu / (nu - 2) = 2, and heavier tails than a Gaussian of that variance
    assert abs(x.var() - 2.0) < 0.3
    assert (np.abs(x) > 6.0).mean() > 10 * 2 * (1 - 0.9999999)


def test_bases_are_orthonormal_and_seeded_inputs_repeat():
    for K, r in ((512, 16), (3072, 32), (1024, 64)):
        U = wl.basis(K, r, seed=0, layer_id=K).astype(np.float64)
        np.testing.assert_allclose(U.T @ U, np.eye(r), atol=1e-6)
    assert wl.basis(64, 0, seed=0).shape == (64, 0)
    a = wl.activations(8, 256, seed=5, layer_id=9)
    b = wl.activations(8, 256, seed=5, layer_id=9)
    c = wl.activations(8, 256, seed=5, layer_id=9, step=1)
    assert np.array_equal(a, b) and not np.array_equal(a, c)
