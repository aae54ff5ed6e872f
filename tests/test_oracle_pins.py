"""Pins of the CPU oracle against what the ExTernD paper and plain mathematics fix.

Each test checks the oracle against something other than itself: closed forms, brute force on tiny inputs,
an independent least-squares solve (numpy lstsq on the vectorised problem), the paper's printed figures, or
identities proved in the paper (Prop. 1). A plausible slip in the oracle (a dropped term, a wrong sign, a
transposed operand, the weights applied on the wrong step) fails at least one of them.
"""
import itertools
import json
import math
import os
import warnings

import numpy as np
import pytest

from oracle import externd_oracle as O
from paper_2607_13511_gb300 import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ---------------------------------------------------------------------------------------------- sizes (§2.1, §2.4)
def test_inner_rank_of_the_workloads():
    assert O.inner_rank(256, 256, 2.0) == 512
    assert O.inner_rank(2048, 2048, 3.0) == 6144
    assert O.inner_rank(2560, 9728, 3.0) == 7680
    assert O.inner_rank(4096, 4096, 2.5) == 10240
    assert O.inner_rank(2560, 1024, 3.0) == 3072
    assert O.inner_rank(10, 7, 0.5) == 4          # 3.5 rounds half up
    assert O.inner_rank(10, 7, 0.2) == 1          # 1.4


def test_block_width_cap():
    assert O.block_width(2048, 2048, 64) == 64
    assert O.block_width(2560, 1024, 256) == 128   # floor(1024 / 8)
    assert O.block_width(256, 256, 1) == 1
    assert O.block_width(12, 40, 64) == 1          # cap floor(12/8) = 1
    assert O.block_width(7, 7, 16) == 1            # cap 0 -> at least 1


# ---------------------------------------------------------------------------------------------- Eq. 2
def test_ternarize_hand_cases():
    # S = 6.5, L = 4, threshold 0.7 * 1.625 = 1.1375: keep 3 and -2.
    assert O.ternarize([3.0, -1.0, 0.5, -2.0], 0.7).tolist() == [1, 0, 0, -1]
    # Equal magnitudes at tau = 1: nothing is strictly above the mean -> keep the first largest entry.
    assert O.ternarize([1.0, -1.0, 1.0, -1.0], 1.0).tolist() == [1, 0, 0, 0]
    assert O.ternarize([-2.0, 2.0, 1.0], 3.0).tolist() == [-1, 0, 0]
    # Zero vector: the fallback keeps index 0 with sign +1.
    assert O.ternarize([0.0, 0.0, 0.0], 0.7).tolist() == [1, 0, 0]
    # tau = 0 keeps every nonzero entry; zeros never pass.
    assert O.ternarize([0.5, 0.0, -1e-30], 0.0).tolist() == [1, 0, -1]
    # Scale invariance (T is invariant to positive scaling).
    x = np.random.default_rng(0).standard_normal(101)
    assert (O.ternarize(x, 0.7) == O.ternarize(37.5 * x, 0.7)).all()
    assert (O.ternarize(x, 0.7) == -O.ternarize(-x, 0.7)).all()


def test_ternarize_mean_counts_zeros():
    # Eq. 2's mean runs over the vector's whole length, zeros included: |x| = (3, 1.2, 0, 0) has mean 4.2 / 4 =
    # 1.05, so 1.2 passes at tau = 1 (over the nonzeros, or over L - 1 = 3 entries, it would not).
    assert O.ternarize([3.0, -1.2, 0.0, 0.0], 1.0).tolist() == [1, -1, 0, 0]
    assert O.ternarize([0.0, 0.0, 1.2, -3.0], 1.0).tolist() == [0, 0, 1, -1]


def test_ternarize_strict_threshold_boundary():
    # mean |x| = 1 exactly; at tau = 2 the entry equal to the threshold (2.0) must not pass.
    x = np.array([2.0, 0.5, 0.5, 1.0])
    assert O.ternarize(x, 2.0).tolist() == [1, 0, 0, 0]      # fallback (nothing > 2)
    assert O.ternarize(x, 1.999).tolist() == [1, 0, 0, 0]     # 2.0 > 1.999
    assert O.ternarize(np.array([2.0, 0.5, 0.5, 1.0, 2.0, 0.0]), 2.0 * 6 / 6.0).tolist() == [1, 0, 0, 0, 0, 0]


@pytest.mark.parametrize("tau", [0.7, 1.0, 2.0])
def test_tau_zero_fraction_gaussian_closed_form_and_paper(tau):
    # For x ~ N(0, 1): mean |x| = sqrt(2/pi), so P(zero) = P(|x| <= tau sqrt(2/pi)) = erf(tau / sqrt(pi)).
    closed = math.erf(tau / math.sqrt(math.pi))
    x = np.random.default_rng(11).standard_normal((40, 5000))
    zeros = float((O.ternarize_rows(x, tau) == 0).mean())
    assert abs(zeros - closed) < 0.005
    paper = json.load(open(os.path.join(GOLDEN, "tau_zero_fraction.json")))["zero_percent"][str(tau)] / 100
    assert abs(zeros - paper) < 0.025


def test_optimal_projection_matches_brute_force():
    rng = np.random.default_rng(5)
    for length in (1, 2, 5, 7):
        for _ in range(5):
            u = rng.standard_normal(length)
            best = min(
                float(np.sum((u - (u @ t) / (t @ t) * t) ** 2))
                for t in (np.array(c, float) for c in itertools.product((-1, 0, 1), repeat=length))
                if np.any(t)
            )
            t, alpha = O.ternary_projection(u)
            assert abs(float(np.sum((u - alpha * t) ** 2)) - best) < 1e-12


# ---------------------------------------------------------------------------------------------- Prop. 1, §2.3
def _lstsq_scales(R, U, Cb, h, ridge):
    """min_d sum_ij h_j (R - sum_a d_a u_a v_a^T)_ij^2 + ridge ||d||^2, solved by lstsq on the vectorised problem."""
    sh = np.sqrt(h)[None, :]
    phi = np.stack([(np.outer(U[:, a], Cb[a]) * sh).ravel() for a in range(U.shape[1])], axis=1)
    y = (R * sh).ravel()
    if ridge > 0:
        phi = np.vstack([phi, math.sqrt(ridge) * np.eye(U.shape[1])])
        y = np.concatenate([y, np.zeros(U.shape[1])])
    return np.linalg.lstsq(phi, y, rcond=None)[0], phi


def test_prop1_identity_and_scale_is_least_squares():
    rng = np.random.default_rng(1)
    for trial in range(20):
        m, n = rng.integers(1, 9, size=2)
        R = rng.standard_normal((m, n))
        u = W.ternary(m, 1, 0.6, trial)[:, 0].astype(float)
        v = W.ternary(1, n, 0.6, 100 + trial)[0].astype(float)
        if not u.any() or not v.any():
            continue
        d = O.block_scales(u[:, None], v[None, :], R @ v[:, None])
        d_ls, _ = _lstsq_scales(R, u[:, None], v[None, :], np.ones(n), 0.0)
        assert np.allclose(d, d_ls, rtol=1e-12, atol=1e-14)
        Rn = O.deflate(R, u[:, None], d, v[None, :])
        drop = (u @ R @ v) ** 2 / ((u @ u) * (v @ v))
        assert abs(O.weighted_norm2(Rn) - (O.weighted_norm2(R) - drop)) < 1e-12 * max(1.0, O.weighted_norm2(R))


def test_sequential_first_component_vs_brute_force():
    # Enumerate every nonzero ternary pair (u, v) on tiny matrices: the best possible one-component decrease.
    rng = np.random.default_rng(2)
    for m, n in ((3, 3), (4, 3), (4, 4), (5, 4)):
        A = rng.standard_normal((m, n))
        us = [np.array(c, float) for c in itertools.product((-1, 0, 1), repeat=m) if any(c)]
        vs = [np.array(c, float) for c in itertools.product((-1, 0, 1), repeat=n) if any(c)]
        Um, Vm = np.array(us), np.array(vs)
        num = (Um @ A @ Vm.T) ** 2
        best = float(np.max(num / np.outer((Um ** 2).sum(1), (Vm ** 2).sum(1))))
        res = O.sequential_als(A, 1.0 / min(m, n), 0.7, 15)
        u, v, d = res.B[:, 0].astype(float), res.C[0].astype(float), res.D[0]
        decrease = O.weighted_norm2(A) - O.weighted_norm2(res.R)
        assert decrease <= best + 1e-12
        assert abs(decrease - (u @ A @ v) ** 2 / ((u @ u) * (v @ v))) < 1e-12
        # the scale is the brute-force least-squares optimum for that pair
        ds = np.linspace(d - 1, d + 1, 2001)
        errs = [np.sum((A - t * np.outer(u, v)) ** 2) for t in ds]
        assert abs(ds[int(np.argmin(errs))] - d) <= 1e-3


def test_planted_ternary_rank_one_is_recovered():
    rng = np.random.default_rng(3)
    for trial in range(5):
        m, n = 17, 23
        u = W.ternary(m, 1, 0.5, 10 + trial)[:, 0]
        v = W.ternary(1, n, 0.5, 20 + trial)[0]
        u[0], v[0] = 1, -1
        A = 0.37 * np.outer(u, v).astype(float)
        res = O.sequential_als(A, 1.0 / min(m, n), 0.7, 4)
        assert res.energy > 1 - 1e-12
        assert abs(abs(res.D[0]) - 0.37) < 1e-12


def test_initial_columns_hand_case():
    # Reading (the paper does not say where u starts): the w columns of largest h_j ||R_:j||^2, ties to the
    # lower index, returned in ascending order. Column energies here are [1, 9, 4, 1].
    R = np.array([[1.0, 0.0, 2.0, 0.0], [0.0, 3.0, 0.0, 1.0]])
    assert O.initial_columns(R, 1, np.ones(4)).tolist() == [1]
    assert O.initial_columns(R, 2, np.ones(4)).tolist() == [1, 2]
    assert O.initial_columns(R, 3, np.ones(4)).tolist() == [0, 1, 2]          # tie 0 vs 3 -> 0
    assert O.initial_columns(R, 2, np.array([10.0, 1.0, 1.0, 1.0])).tolist() == [0, 1]
    assert O.initial_columns(R, 4, np.ones(4)).tolist() == [0, 1, 2, 3]


# ---------------------------------------------------------------------------------------------- Eq. 3, Eq. 4, §2.5
def test_vstep_target_is_ridge_least_squares():
    rng = np.random.default_rng(4)
    m, n, w = 40, 30, 5
    R = rng.standard_normal((m, n))
    U = W.ternary(m, w, 0.6, 4).astype(float)
    X = O.vstep_target(R, U)
    eps = O.EPS_REL * np.trace(U.T @ U) / w
    X_ls = np.linalg.lstsq(np.vstack([U, math.sqrt(eps) * np.eye(w)]), np.vstack([R, np.zeros((w, n))]),
                           rcond=None)[0]
    assert np.allclose(X, X_ls, rtol=1e-10, atol=1e-12)


def test_ustep_target_is_weighted_ridge_least_squares():
    rng = np.random.default_rng(5)
    m, n, w = 30, 40, 6
    R = rng.standard_normal((m, n))
    Cb = W.ternary(w, n, 0.6, 5).astype(float)
    h = W.importance(n, 5).astype(float)
    Y = O.ustep_target(R, Cb, h)
    V = Cb.T
    eps = O.EPS_REL * np.sum(h[:, None] * V * V) / w
    sh = np.sqrt(h)[:, None]
    Yt = np.linalg.lstsq(np.vstack([sh * V, math.sqrt(eps) * np.eye(w)]), np.vstack([sh * R.T, np.zeros((w, m))]),
                         rcond=None)[0]
    assert np.allclose(Y, Yt.T, rtol=1e-10, atol=1e-12)


def test_weights_cancel_in_the_exact_vstep():
    # §2.5: in a column-weighted objective the importances cancel in the V-step, so its exact target is plain R.
    rng = np.random.default_rng(6)
    m, n, w = 25, 20, 4
    R = rng.standard_normal((m, n))
    U = W.ternary(m, w, 0.6, 6).astype(float)
    h = W.importance(n, 6).astype(float)
    # min_X sum_ij h_j (R - U X)_ij^2, one column j at a time, solved by lstsq with the weights applied
    X_w = np.stack([np.linalg.lstsq(math.sqrt(h[j]) * U, math.sqrt(h[j]) * R[:, j], rcond=None)[0]
                    for j in range(n)], axis=1)
    assert np.allclose(O.vstep_target(R, U), X_w, rtol=2e-3, atol=1e-6)   # ridge 1e-4 relative


@pytest.mark.parametrize("weighted", [False, True])
def test_block_scales_are_weighted_least_squares(weighted):
    rng = np.random.default_rng(7)
    m, n, w = 20, 18, 5
    R = rng.standard_normal((m, n))
    U = W.ternary(m, w, 0.6, 7).astype(float)
    Cb = W.ternary(w, n, 0.6, 8).astype(float)
    h = W.importance(n, 7).astype(float) if weighted else np.ones(n)
    d = O.block_scales(U, Cb, O.ustep_product(R, Cb, h if weighted else None), h if weighted else None)
    K = (U.T @ U) * (Cb @ (h[:, None] * Cb.T))
    d_ls, _ = _lstsq_scales(R, U, Cb, h, O.EPS_REL * np.trace(K) / w)
    assert np.allclose(d, d_ls, rtol=1e-9, atol=1e-12)
    # exact decrease of the ridge least-squares step: ||R||^2 - r^T d - eps ||d||^2
    Rn = O.deflate(R, U, d, Cb)
    r = np.sum(U * O.ustep_product(R, Cb, h), axis=0)
    eps = O.EPS_REL * np.trace(K) / w
    lhs = O.weighted_norm2(Rn, h)
    rhs = O.weighted_norm2(R, h) - r @ d - eps * d @ d
    assert abs(lhs - rhs) < 1e-10 * O.weighted_norm2(R, h)


# ---------------------------------------------------------------------------------------------- algorithms
def test_block_width_one_is_the_sequential_algorithm():
    A = W.gaussian(48, 40, 0.02, 9)
    h = W.importance(40, 9)
    for weights in (None, h):
        s = O.sequential_als(A, 2.0, 0.7, 4, weights)
        b = O.block_als(A, 2.0, 0.7, 1, 4, weights)
        assert (s.B == b.B).all() and (s.C == b.C).all()
        assert np.allclose(s.D, b.D, rtol=1e-12, atol=0)


@pytest.mark.parametrize("block,weighted", [(1, False), (1, True), (8, False), (8, True)])
def test_energy_trace_is_monotone_and_matches_reconstruction(block, weighted):
    A = W.student_t(64, 80, 5.0, 0.015, 10)
    h = W.importance(80, 10) if weighted else None
    res = O.decompose(A, 2.0, 0.7, block, 4, h)
    assert np.all(np.diff(res.trace) >= -1e-13)
    assert abs(res.energy - O.energy(A, res.B, res.D, res.C, h)) < 1e-10
    assert set(np.unique(res.B)) <= {-1, 0, 1} and set(np.unique(res.C)) <= {-1, 0, 1}
    assert (np.abs(res.B).sum(0) > 0).all() and (np.abs(res.C).sum(1) > 0).all()   # no empty factor


def test_energy_approaches_one_as_mu_grows():
    # Corollary (Appendix A): the residual can be driven below any epsilon by adding components.
    A = W.gaussian(6, 5, 1.0, 12)
    res = O.sequential_als(A, 30.0, 0.7, 4)   # k = 150
    assert np.all(np.diff(res.trace) >= -1e-13)
    assert res.energy > 1 - 1e-6


def test_tail_block_and_rank():
    A = W.gaussian(40, 33, 0.02, 13)
    res = O.block_als(A, 1.3, 0.7, 4, 2)         # k = 43, b = 4 -> 10 blocks of 4 and one of 3
    assert res.B.shape == (40, 43) and res.C.shape == (43, 33) and res.D.shape == (43,)
    assert len(res.trace) == 11
    assert np.all(res.D != 0)


def test_importance_scaling_does_not_change_the_factors():
    A = W.gaussian(40, 48, 0.02, 14)
    h = W.importance(48, 14)
    a = O.block_als(A, 1.5, 0.7, 6, 3, h)
    b = O.block_als(A, 1.5, 0.7, 6, 3, (h * 8.0))   # power of two: exactly the same relative ridge
    assert (a.B == b.B).all() and (a.C == b.C).all()
    assert np.allclose(a.D, b.D, rtol=1e-12)


# ---------------------------------------------------------------------------------------------- soft checks (§2.4, §2.5)
def _naive_block(A, mu, tau, block, iters, weights=None, naive_v=False, naive_w=False):
    """Variants the paper argues against, built from the oracle's steps: no decorrelation (naive_v) or the
    V-step solved against W = R (.) h (naive_w)."""
    R = np.array(A, dtype=np.float64)
    m, n = R.shape
    h = np.ones(n) if weights is None else np.asarray(weights, float)
    k, b = O.inner_rank(m, n, mu), O.block_width(m, n, block)
    norm_a = O.weighted_norm2(R, h)
    for j0 in range(0, k, b):
        w = min(b, k - j0)
        U = O.ternarize_cols(R[:, O.initial_columns(R, w, h)], tau)
        for _ in range(iters):
            if naive_v:
                Cb = O.ternarize_rows((R.T @ U).T, tau)
                PU = O.ustep_product(R, Cb, h)
                U = O.ternarize_cols(PU, tau)
            else:
                target = R * h[None, :] if naive_w else R
                Cb = O.ternarize_rows(O.vstep_target(target, U), tau)
                PU = O.ustep_product(R, Cb, h)
                U = O.ternarize_cols(O.ustep_solve(PU, Cb, h), tau)
        R = O.deflate(R, U, O.block_scales(U, Cb, PU, h), Cb)
    return 1 - O.weighted_norm2(R, h) / norm_a


def test_decorrelated_blocks_match_sequential_and_naive_blocks_collapse():
    A = W.student_t(128, 160, 5.0, 0.015, 15)
    seq = O.sequential_als(A, 1.5, 0.7, 4).energy
    blk = O.block_als(A, 1.5, 0.7, 16, 4).energy
    naive = _naive_block(A, 1.5, 0.7, 16, 4, naive_v=True)
    # §3.1 Table 1: batched matches sequential within +-0.2 points on LLM matrices.
    if abs(blk - seq) > 0.002:
        warnings.warn(f"block vs sequential differ by {100 * (blk - seq):.2f} points on synthetic data")
    assert abs(blk - seq) < 0.02
    # §2.4: ternarizing R^T U column-wise without decorrelation collapses.
    assert naive < blk - 0.05


def test_weighted_vstep_correction_beats_naive_weighted_vstep():
    A = W.gaussian(96, 128, 0.02, 16)
    h = W.importance(128, 16)
    corrected = O.block_als(A, 1.5, 0.7, 12, 4, h).energy
    naive = _naive_block(A, 1.5, 0.7, 12, 4, h, naive_w=True)
    # §2.5: the naive weighted V-step loses 0.3-1.8 points of weighted energy.
    assert corrected > naive


# ---------------------------------------------------------------------------------------------- a block step by hand
def test_hand_computed_two_component_block_step():
    """One block of w = 2 (§2.4, Eq. 3 and Eq. 4) worked out by hand on a 4 x 4 residual, tau = 0.7.

    Start (largest column energies 32 and 18: columns 0 and 1): U = [e0 + e1, e2 + e3].
    V-step: U^T U = 2 I, eps = 1e-4 * 4 / 2, so X = (R[0] + R[1], R[2] + R[3]) / 2.0002 = ([8,0,0,0], [0,6,0,1])
    / 2.0002; means of |x| 2 and 1.75 (times 1 / 2.0002) give thresholds 1.4 and 1.225 (same scale): V = e0, e1.
    U-step: V^T V = I, eps = 1e-4, Y = R V / 1.0001 = ([4,4,0,0], [0,0,3,3]) / 1.0001: U stays [e0 + e1, e2 + e3].
    Eq. 4: K = (U^T U) .* (V^T V) = 2 I, eps = 1e-4 * 4 / 2 = 2e-4, r = (8, 6): d = (8, 6) / 2.0002.
    Deflation leaves 4 - d0 in R[0:2, 0], 3 - d1 in R[2:4, 1] and the three unit entries."""
    R = np.array([[4.0, 0.0, 1.0, 0.0],
                  [4.0, 0.0, -1.0, 0.0],
                  [0.0, 3.0, 0.0, 0.0],
                  [0.0, 3.0, 0.0, 1.0]])
    U0 = np.array([[1, 0], [1, 0], [0, 1], [0, 1]], dtype=np.int8)
    assert O.initial_columns(R, 2, np.ones(4)).tolist() == [0, 1]
    assert (O.ternarize_cols(R[:, [0, 1]], 0.7) == U0).all()
    X = O.vstep_target(R, U0)
    assert np.allclose(X, np.array([[8.0, 0, 0, 0], [0, 6.0, 0, 1.0]]) / 2.0002, rtol=1e-14, atol=0)
    Cb = O.ternarize_rows(X, 0.7)
    assert (Cb == np.array([[1, 0, 0, 0], [0, 1, 0, 0]])).all()
    PU = O.ustep_product(R, Cb)
    assert np.array_equal(PU, np.array([[4.0, 0], [4.0, 0], [0, 3.0], [0, 3.0]]))
    Y = O.ustep_solve(PU, Cb)
    assert np.allclose(Y, PU / 1.0001, rtol=1e-14, atol=0)
    U1 = O.ternarize_cols(Y, 0.7)
    assert (U1 == U0).all()
    d = O.block_scales(U1, Cb, PU)
    assert np.allclose(d, [8 / 2.0002, 6 / 2.0002], rtol=1e-14, atol=0)
    R1 = O.deflate(R, U1, d, Cb)
    expect = R.copy()
    expect[0:2, 0] = 4 - 8 / 2.0002
    expect[2:4, 1] = 3 - 6 / 2.0002
    assert np.allclose(R1, expect, rtol=0, atol=1e-14)


# ---------------------------------------------------------------------------------------------- block loop properties
def _block_residuals(A, res, b):
    """The residual each block of a block_als result was fitted to, rebuilt from the returned factors alone."""
    R = np.asarray(A, dtype=np.float64).copy()
    out = []
    for j0 in range(0, res.D.size, b):
        j1 = min(res.D.size, j0 + b)
        out.append((R.copy(), j0, j1))
        R = R - (res.B[:, j0:j1] * res.D[j0:j1]) @ res.C[j0:j1].astype(np.float64)
    return out


@pytest.mark.parametrize("weighted", [False, True])
def test_block_loop_scales_are_ridge_least_squares_for_each_block(weighted):
    # Eq. 4 for the factors block_als returns: each block's D is the ridge least-squares scale of its own U and V
    # against the residual it was fitted to (lstsq on the vectorised problem, independent of the oracle's solver).
    A = W.student_t(40, 48, 5.0, 0.015, 21)
    h = W.importance(48, 21).astype(float) if weighted else None
    hh = np.ones(48) if h is None else h
    res = O.block_als(A, 0.6, 0.7, 8, 3, h)
    for R, j0, j1 in _block_residuals(A, res, 5):
        U, Cb = res.B[:, j0:j1].astype(float), res.C[j0:j1].astype(float)
        K = (U.T @ U) * (Cb @ (hh[:, None] * Cb.T))
        eps = O.EPS_REL * np.trace(K) / (j1 - j0) if j1 - j0 > 1 else 0.0
        d_ls, _ = _lstsq_scales(R, U, Cb, hh, eps)
        assert np.allclose(res.D[j0:j1], d_ls, rtol=1e-9, atol=1e-12), (j0, j1)


@pytest.mark.parametrize("weighted", [False, True])
def test_block_loop_final_u_is_the_ustep_of_the_final_v(weighted):
    # The last step of every block is the U-step (Eq. 3 right, §2.5): U = T_tau of the weighted ridge
    # least-squares target of the block's final V against the residual it was fitted to (lstsq, column-weighted).
    A = W.gaussian(40, 48, 0.02, 22)
    h = W.importance(48, 22).astype(float) if weighted else None
    hh = np.ones(48) if h is None else h
    res = O.block_als(A, 0.6, 0.7, 8, 3, h)
    for R, j0, j1 in _block_residuals(A, res, 5):
        V = res.C[j0:j1].astype(float).T
        w = j1 - j0
        eps = O.EPS_REL * np.sum(hh[:, None] * V * V) / w
        sh = np.sqrt(hh)[:, None]
        Yt = np.linalg.lstsq(np.vstack([sh * V, math.sqrt(eps) * np.eye(w)]),
                             np.vstack([sh * R.T, np.zeros((w, R.shape[0]))]), rcond=None)[0]
        assert (O.ternarize_cols(Yt.T, 0.7) == res.B[:, j0:j1]).all(), (j0, j1)
