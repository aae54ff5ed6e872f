"""Pins of the oracle's second part (rank budgets, packing, the Prop. 2 safeguard, refinement sweeps), each
checked against something other than the oracle restating itself: the method's greedy-prefix structure, exhaustive
search, Eq. 5's bit count from an actual packing, the Prop. 2 bound, and explicit reconstruction."""
import itertools
import warnings

import numpy as np
import pytest

import oracle as O
from paper_2607_13511_gb300 import workloads as W


# ------------------------------------------------------------------------------------------- rank budgets
@pytest.mark.parametrize("block", [1, 8])
def test_smaller_rank_is_a_prefix_of_a_larger_one(block):
    """§2.3/§2.4: sequential deflation means a run at a smaller inner rank is the prefix of a longer run."""
    A = W.gaussian(48, 64, 0.02, 31)
    b = O.block_width(48, 64, block)
    big = O.decompose(A, 1.5, 0.7, block, 3)
    k1 = 3 * b
    small = O.decompose(A, k1 / 48, 0.7, block, 3)
    assert small.B.shape[1] == k1
    np.testing.assert_array_equal(small.B, big.B[:, :k1])
    np.testing.assert_array_equal(small.C, big.C[:k1])
    np.testing.assert_array_equal(small.D, big.D[:k1])
    assert small.trace == big.trace[:len(small.trace)]


def test_rank_for_energy_matches_reconstructed_energies():
    A = W.student_t(40, 72, 5.0, 0.015, 7)
    res = O.block_als(A, 2.0, 0.7, 8, 3)
    ranks = O.block_boundaries(40, 72, 2.0, 8)
    assert len(ranks) == len(res.trace)
    energies = [O.energy(A, res.B[:, :k], res.D[:k], res.C[:k]) for k in ranks]   # from the factors alone
    np.testing.assert_allclose(energies, res.trace, rtol=0, atol=1e-10)
    # "reaches the target" includes equality: every boundary's own energy as a target
    for target in (0.3, 0.8, 0.95, 0.999, 1.5, *res.trace):
        brute = next((k for k, e in zip(ranks, energies) if e >= target - 1e-12), None)
        assert O.rank_for_energy(res.trace, ranks, target) == brute


def test_allocation_is_optimal_on_concave_curves():
    """Greedy by marginal gain per cost is optimal when every curve is concave and blocks cost the same."""
    rng = np.random.default_rng(5)
    for trial in range(25):
        nm = int(rng.integers(2, 4))
        curves = []
        for _ in range(nm):
            gains = np.sort(rng.random(int(rng.integers(1, 5))))[::-1]   # decreasing gains: concave
            e = np.cumsum(gains) / (gains.sum() * 1.1)
            curves.append([(4 * (i + 1), float(e[i])) for i in range(len(e))])
        costs = [1.0] * nm
        budget = float(4 * rng.integers(1, 9))
        got = O.allocate_ranks(curves, costs, budget)
        best = -1.0
        for choice in itertools.product(*[range(len(c) + 1) for c in curves]):
            cost = sum(4 * ch for ch in choice)
            if cost > budget:
                continue
            val = sum(0.0 if ch == 0 else curves[j][ch - 1][1] for j, ch in enumerate(choice))
            best = max(best, val)
        got_val = sum(0.0 if k == 0 else dict(curves[j])[k] for j, k in enumerate(got))
        assert sum(got) <= budget
        assert got_val == pytest.approx(best, abs=1e-12)


# ------------------------------------------------------------------------------------------------ packing
def test_mask_sign_packing_roundtrip_and_eq5():
    A = W.gaussian(48, 80, 0.02, 11)
    mu = 1.5
    res = O.block_als(A, mu, 0.7, 8, 3)
    bits = 0
    zeros = 0
    for T in (res.B, res.C):
        mask, sign = O.pack_mask_sign(T)
        np.testing.assert_array_equal(O.unpack_mask_sign(mask, sign, T.shape), T)
        assert len(mask) == T.size and len(sign) == int(np.count_nonzero(T))
        bits += len(mask) + len(sign)
        zeros += T.size - int(np.count_nonzero(T))
    sparsity = zeros / (res.B.size + res.C.size)
    assert bits / A.size == pytest.approx(O.bpw_eff(mu, 48, 80, sparsity), rel=1e-12)


def test_ternary_apply_matches_dense_reconstruction():
    A = W.gaussian(30, 50, 0.02, 12)
    res = O.block_als(A, 1.2, 0.7, 4, 2)
    x = np.random.default_rng(2).standard_normal(50)
    dense = (res.B.astype(np.float64) * res.D[None, :]) @ res.C.astype(np.float64)
    np.testing.assert_allclose(O.ternary_apply(res.B, res.D, res.C, x), dense @ x, rtol=1e-12, atol=1e-14)


# ------------------------------------------------------------------------------------------------ Prop. 2
def test_best_single_entry_brute_force():
    R = np.random.default_rng(4).standard_normal((6, 5))
    h = np.random.default_rng(5).random(5) + 0.1
    i, j, rij, removed = O.best_single_entry(R, h)
    best = max((h[c] * R[r, c] ** 2, -r, -c) for r in range(6) for c in range(5))
    assert (i, j) == (-best[1], -best[2]) and removed == pytest.approx(best[0]) and rij == R[i, j]
    # the pair u = e_i, v = sgn e_j with d = |R_ij| removes exactly h_j R_ij^2
    U = np.zeros((6, 1), np.int8); U[i, 0] = 1
    V = np.zeros((1, 5), np.int8); V[0, j] = 1 if rij >= 0 else -1
    after = O.deflate(R, U, np.array([abs(rij)]), V)
    assert O.weighted_norm2(R, h) - O.weighted_norm2(after, h) == pytest.approx(removed, rel=1e-12)


@pytest.mark.parametrize("seed", range(6))
def test_safeguard_geometric_bound(seed):
    """Prop. 2: with the safeguard, ||R_k||^2 <= (1 - 1/(mn))^k ||A||^2 after every component."""
    rng = np.random.default_rng(seed)
    m, n = int(rng.integers(3, 8)), int(rng.integers(3, 8))
    A = rng.standard_normal((m, n)) * np.exp(rng.standard_normal((m, n)))
    tau = float(rng.choice([0.0, 0.7, 2.0]))
    res, _ = O.decompose_safeguarded(A, 3.0, tau, 1, 3)
    for k, e in enumerate(res.trace, start=1):
        assert 1.0 - e <= (1.0 - 1.0 / (m * n)) ** k + 1e-12


def test_safeguard_activates_on_a_spike_in_noise():
    """tau = 0 keeps every entry, so the fitted component is a dense sign pattern; one large entry in small
    noise is then removed better by the single-entry pair."""
    rng = np.random.default_rng(1)
    A = 0.01 * rng.standard_normal((8, 8))
    A[3, 5] = 1.0
    res, act = O.decompose_safeguarded(A, 0.25, 0.0, 1, 3)
    assert act >= 1
    assert res.B[3, 0] == 1 and np.count_nonzero(res.B[:, 0]) == 1
    assert res.C[0, 5] == 1 and np.count_nonzero(res.C[0]) == 1
    assert res.D[0] == pytest.approx(1.0)
    plain = O.decompose(A, 0.25, 0.0, 1, 3)
    assert res.energy > plain.energy


def test_safeguard_inactive_is_the_plain_method():
    A = W.gaussian(32, 40, 0.02, 9)
    for block in (1, 4):
        res, act = O.decompose_safeguarded(A, 1.0, 0.7, block, 3)
        plain = O.decompose(A, 1.0, 0.7, block, 3)
        assert act == 0
        np.testing.assert_array_equal(res.B, plain.B)
        np.testing.assert_array_equal(res.C, plain.C)
        np.testing.assert_allclose(res.D, plain.D, rtol=1e-12)


# ----------------------------------------------------------------------------------------- refinement sweeps
@pytest.mark.parametrize("block", [1, 8])
def test_refinement_is_monotone_and_consistent(block):
    A = W.student_t(40, 64, 5.0, 0.015, 3)
    res = O.decompose(A, 1.5, 1.0, block, 3)
    ref, replaced = O.refine(A, res, 1.0, block, 3, 4)
    energies = [res.energy] + ref.trace
    assert all(b >= a - 1e-12 for a, b in zip(energies, energies[1:]))
    assert ref.energy == pytest.approx(O.energy(A, ref.B, ref.D, ref.C), abs=1e-10)
    assert set(np.unique(ref.B)) <= {-1, 0, 1} and set(np.unique(ref.C)) <= {-1, 0, 1}
    assert len(replaced) == 4


def test_refinement_never_lowers_the_energy_on_random_matrices():
    """§2.4's sweeps may only improve a decomposition: a refit is kept only if it removes at least as much as the
    block it replaces. Small heavy-tailed matrices over tau, block width and iteration counts include refits that
    remove less (ALS from a warm start is not monotone there), so the keep rule is what holds the energy up."""
    rng = np.random.default_rng(0)
    for _ in range(120):
        m, n = int(rng.integers(4, 12)), int(rng.integers(4, 12))
        A = rng.standard_normal((m, n)) * np.exp(rng.standard_normal((m, n)))
        tau = float(rng.choice([0.0, 0.7, 1.5, 2.5, 4.0]))
        block = int(rng.choice([1, 2, 4]))
        iters = int(rng.choice([1, 2]))
        mu = float(rng.choice([0.5, 1.0, 2.0]))
        res = O.decompose(A, mu, tau, block, 3)
        ref, _ = O.refine(A, res, tau, block, iters, 2)
        energies = [res.energy] + ref.trace
        assert all(b >= a - 1e-12 for a, b in zip(energies, energies[1:])), (m, n, tau, block, iters, mu)


@pytest.mark.parametrize("block", [4, 8])
def test_refinement_improves_single_iteration_fits(block):
    """Blocks fitted with one ALS iteration are far from their best; refitting each one on the residual with
    the block added back (§2.4) must raise the energy."""
    A = W.student_t(40, 64, 5.0, 0.015, 3)
    res = O.decompose(A, 1.0, 1.0, block, 1)
    ref, replaced = O.refine(A, res, 1.0, block, 1, 3)
    assert sum(replaced) > 0
    assert ref.energy > res.energy + 1e-3


def test_refinement_gain_on_a_hard_matrix_soft():
    """§2.4 reports about +0.4 points of energy after 10 sweeps on hard matrices (LLM weights); synthetic data
    only gets a warning if the gain differs in size."""
    A = W.student_t(64, 96, 5.0, 0.015, 21)
    res = O.block_als(A, 1.0, 1.0, 8, 4)
    ref, _ = O.refine(A, res, 1.0, 8, 4, 10)
    gain = 100.0 * (ref.energy - res.energy)
    assert gain >= 0.0
    if not 0.05 <= gain <= 2.0:
        warnings.warn(f"refinement gain {gain:.3f} points on synthetic data (paper: ~0.4 on LLM matrices)")
