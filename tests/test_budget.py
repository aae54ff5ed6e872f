"""Rank and storage budgets (host functions of the library, no GPU) against the oracle: block boundaries, the
smallest rank reaching a target energy, and the greedy per-matrix allocation, on random curves including
non-concave ones where greedy is not optimal but both sides must still choose the same ranks."""
import os
import shutil

import numpy as np
import pytest

from oracle import externd_next as N


@pytest.fixture(scope="module")
def X():
    if shutil.which("nvcc") is None and not os.path.exists("/usr/local/cuda/bin/nvcc"):
        pytest.skip("nvcc not available")
    import paper_2607_13511_gb300 as X
    from paper_2607_13511_gb300 import build
    build.build()
    X.load()
    return X


@pytest.mark.parametrize("m,n,mu,block", [(256, 256, 2.0, 1), (2048, 2048, 3.0, 64), (2560, 9728, 3.0, 128),
                                          (4096, 4096, 2.5, 128), (10, 7, 0.5, 1), (100, 37, 1.3, 4)])
def test_block_boundaries(X, m, n, mu, block):
    assert X.block_boundaries(m, n, mu, block) == N.block_boundaries(m, n, mu, block)


def test_rank_for_energy_on_random_traces(X):
    rng = np.random.default_rng(0)
    for trial in range(200):
        m, n = int(rng.integers(8, 300)), int(rng.integers(8, 300))
        mu = float(rng.choice([0.5, 1.0, 1.5, 3.0]))
        block = int(rng.choice([1, 4, 8, 64]))
        ranks = N.block_boundaries(m, n, mu, block)
        trace = list(np.cumsum(rng.random(len(ranks))) / (len(ranks) * rng.uniform(0.5, 1.2)))
        for target in (0.0, 0.3, 0.9, float(trace[len(trace) // 2]), 2.0):
            assert X.rank_for_energy(trace, m, n, mu, block, target) == N.rank_for_energy(trace, ranks, target)


def test_rank_for_energy_rejects_a_trace_of_the_wrong_length(X):
    with pytest.raises(X.ExterndError):
        X.rank_for_energy([0.1, 0.2], 64, 64, 1.0, 8, 0.15)


@pytest.mark.parametrize("concave", [True, False])
def test_allocation_matches_the_oracle(X, concave):
    rng = np.random.default_rng(1 if concave else 2)
    for trial in range(150):
        nm = int(rng.integers(1, 6))
        curves = []
        for _ in range(nm):
            npt = int(rng.integers(0, 7))
            step = int(rng.integers(1, 9))
            gains = rng.random(npt)
            if concave:
                gains = np.sort(gains)[::-1]
            e = np.cumsum(gains) / max(1e-9, gains.sum() * 1.05)
            curves.append([(step * (i + 1), float(e[i])) for i in range(npt)])
        costs = [float(c) for c in rng.uniform(0.5, 3.0, nm)]
        weights = None if trial % 2 else [float(w) for w in rng.uniform(0.2, 2.0, nm)]
        budget = float(rng.uniform(0, 60))
        assert X.allocate_ranks(curves, costs, budget, weights) == N.allocate_ranks(curves, costs, budget, weights)


def test_allocation_from_real_traces(X):
    """Curves from oracle runs of three matrices of different difficulty, allocated under (m + n)-bit costs."""
    from oracle import externd_oracle as O
    from paper_2607_13511_gb300 import workloads as W
    mats = [W.gaussian(48, 64, 0.02, 1), W.student_t(48, 64, 5.0, 0.015, 2), W.gaussian_with_outliers(48, 64, 0.02, 0.01, 20.0, 3)]
    curves, costs = [], []
    for A in mats:
        res = O.block_als(A, 2.0, 0.7, 4, 2)
        ranks = N.block_boundaries(48, 64, 2.0, 4)
        curves.append(list(zip(ranks, res.trace)))
        costs.append(48.0 + 64.0)
    for budget in (500.0, 3000.0, 9000.0):
        assert X.allocate_ranks(curves, costs, budget) == N.allocate_ranks(curves, costs, budget)
