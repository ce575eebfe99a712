"""The expert choice of Sec. 4.3 (qwam_asp_select_experts, host-only, no GPU needed) against the
oracle: decreasing action mass per added 16-bit value while the additions fit the budget."""
import numpy as np
import pytest

from oracle import subspace as sub


@pytest.fixture(scope="module")
def asp():
    from paper_2609_33269_gb300 import asp as a
    from paper_2609_33269_gb300 import build
    try:
        build.build()
        a.load()
    except Exception as e:  # the library needs nvcc to build; the host call itself needs no GPU
        pytest.skip("library not buildable here: %s" % e)
    return a


def test_select_experts_matches_the_oracle(asp):
    rng = np.random.default_rng(0)
    for trial in range(200):
        n = int(rng.integers(0, 9))
        mass = rng.exponential(1.0, n) * (rng.random(n) < 0.9)
        cost = rng.integers(1, 50, n).astype(np.float64)
        budget = float(rng.uniform(0, cost.sum() + 1)) if n else 3.0
        assert asp.qwam_asp_select_experts(mass, cost, budget) == sub.select_experts(list(mass), list(cost), budget)


def test_select_experts_hand_cases_and_errors(asp):
    assert asp.qwam_asp_select_experts([89.3, 10.0, 0.7], [100.0, 400.0, 10.0], 110.0) == [0, 2]
    assert asp.qwam_asp_select_experts([1.0, 2.0], [1.0, 2.0], 1.5) == [0]
    assert asp.qwam_asp_select_experts([], [], 5.0) == []
    with pytest.raises(asp.QwamError):
        asp.qwam_asp_select_experts([1.0], [0.0], 5.0)  # a cost must be positive
