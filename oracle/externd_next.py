"""ExTernD oracle, second part: the uses and extensions of the decomposition (fp64, numpy).

TEST INFRASTRUCTURE ONLY, like ``externd_oracle``: only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import it; the product path never does, and the two share no code.

* Rank and energy budgets (§3 iso-energy comparisons, §5 "per-matrix rank allocation"): because the method is
  greedy with sequential deflation (§2.3, §2.4), the factors of a run at inner rank k1 are the first k1
  components of a run at any k2 > k1 (for k1 a multiple of the block width), so one run at the largest rank
  gives the energy at every block boundary.
* Mask+sign packing and the inference product (§2.6, Eq. 5): y = B (diag(D) (C x)).
* The convergence safeguard of Prop. 2 (appendix): take the best single-entry pair whenever it removes more
  than the fitted component.
* Refinement sweeps (§2.4): revisit each block, add it back, refit, deflate again.

Readings taken where the paper is silent:

* Safeguard with importance weights: the single-entry pair u = e_i, v = sgn(R_ij) e_j removes h_j R_ij^2 from
  the weighted residual, so the best pair is the argmax of h_j R_ij^2 (ties to the lowest row, then column).
  For a block of w components the comparison is between the block's decrease (the drop of the weighted squared
  norm of the residual when it is deflated) and that maximum; when the pair wins, the block becomes the pair followed by w - 1 zero
  components (zero factor columns and rows, scale 0). With b = 1 it is Prop. 2 as stated.
* Refinement sweep: the blocks are revisited in order; a revisited block is refitted by `iters` ALS
  iterations warm-started from its current U (no column selection), and the refit replaces the block only if
  it removes at least as much from the added-back residual as the block it replaces (both measured as the
  drop of the weighted squared norm of that residual), so the energy never decreases.
"""
from __future__ import annotations

import math

import numpy as np

from .externd_oracle import (Result, block_scales, block_width, deflate, initial_columns, inner_rank, ternarize,
                             ternarize_cols, ternarize_rows, ustep_product, ustep_solve, vstep_target,
                             weighted_norm2)


# ----------------------------------------------------------------------------------------------------------
# Rank and energy budgets
# ----------------------------------------------------------------------------------------------------------
def block_boundaries(m: int, n: int, mu: float, block: int) -> list[int]:
    """The inner ranks at which a run at (mu, block) finishes a block (§2.4): b, 2b, ..., k."""
    k, b = inner_rank(m, n, mu), block_width(m, n, block)
    return [min(j, k) for j in range(b, k + b, b)]


def rank_for_energy(trace, ranks, target: float):
    """Smallest inner rank among ``ranks`` (the block boundaries of one run) whose energy reaches ``target``;
    None when the run never does."""
    for e, k in zip(trace, ranks):
        if e >= target:
            return k
    return None


def allocate_ranks(curves, costs, budget: float, weights=None):
    """Per-matrix rank allocation under a storage budget. ``curves[j]`` lists (k, E_j(k)) at matrix j's block
    boundaries (from one run each); choosing boundary i of matrix j costs ``costs[j] * k``. Greedy: repeatedly
    take the next block of the matrix with the largest weighted energy gain per unit cost that still fits (ties
    to the lower matrix index). Returns the chosen rank of every matrix (0 for none). Optimal when every curve
    is concave in k (decreasing gains), as greedy deflation curves are."""
    nm = len(curves)
    wts = [1.0] * nm if weights is None else list(weights)
    idx = [0] * nm               # blocks taken per matrix
    spent = 0.0
    while True:
        best, best_j = None, -1
        for j in range(nm):
            if idx[j] >= len(curves[j]):
                continue
            k_prev, e_prev = (0, 0.0) if idx[j] == 0 else curves[j][idx[j] - 1]
            k_next, e_next = curves[j][idx[j]]
            cost = costs[j] * (k_next - k_prev)
            if spent + cost > budget + 1e-12:
                continue
            gain = wts[j] * (e_next - e_prev) / cost
            if best is None or gain > best:
                best, best_j = gain, j
        if best_j < 0:
            break
        k_prev = 0 if idx[best_j] == 0 else curves[best_j][idx[best_j] - 1][0]
        spent += costs[best_j] * (curves[best_j][idx[best_j]][0] - k_prev)
        idx[best_j] += 1
    return [0 if idx[j] == 0 else curves[j][idx[j] - 1][0] for j in range(nm)]


# ----------------------------------------------------------------------------------------------------------
# §2.6, Eq. 5: mask+sign packing and the inference product
# ----------------------------------------------------------------------------------------------------------
def pack_mask_sign(T):
    """Sparse mask+sign packing of a ternary matrix (§2.6): one mask bit per element in row-major order (1 =
    nonzero) and one sign bit per nonzero in the same order (1 = negative). Returns (mask bits, sign bits) as
    uint8 arrays of 0/1 values (one entry per bit, kept unpacked for clarity)."""
    t = np.asarray(T).reshape(-1)
    mask = (t != 0).astype(np.uint8)
    sign = (t[t != 0] < 0).astype(np.uint8)
    return mask, sign


def unpack_mask_sign(mask, sign, shape):
    """Inverse of pack_mask_sign."""
    t = np.zeros(len(mask), np.int8)
    nz = np.flatnonzero(mask)
    t[nz] = np.where(np.asarray(sign) == 1, -1, 1).astype(np.int8)
    return t.reshape(shape)


def bpw_eff(mu: float, m: int, n: int, sparsity: float) -> float:
    """Eq. 5: storage per original weight of the mask+sign packed factors."""
    return mu * (m + n) / max(m, n) * (2.0 - sparsity)


def ternary_apply(B, D, C, x):
    """§2.6: y = B (diag(D) (C x)) in float64."""
    z = np.asarray(D, np.float64) * (np.asarray(C, np.float64) @ np.asarray(x, np.float64))
    return np.asarray(B, np.float64) @ z


# ----------------------------------------------------------------------------------------------------------
# Prop. 2: the convergence safeguard
# ----------------------------------------------------------------------------------------------------------
def best_single_entry(R, h=None):
    """The single-entry pair of Prop. 2 under column weights h: (i, j, R_ij, removed = h_j R_ij^2), the first
    (row-major) maximizer."""
    hh = np.ones(R.shape[1]) if h is None else np.asarray(h, np.float64)
    score = hh[None, :] * R * R
    flat = int(np.argmax(score))
    i, j = divmod(flat, R.shape[1])
    return i, j, float(R[i, j]), float(score[i, j])


def _block_fit(R, U, tau, iters, h):
    """`iters` ALS iterations of §2.4 from the ternary U; returns (U, V, d, decrease), the decrease being the
    drop of the weighted squared norm of R when the block is deflated."""
    for _ in range(iters):
        Cb = ternarize_rows(vstep_target(R, U), tau)
        PU = ustep_product(R, Cb, h)
        U = ternarize_cols(ustep_solve(PU, Cb, h), tau)
    d = block_scales(U, Cb, PU, h)
    return U, Cb, d, weighted_norm2(R, h) - weighted_norm2(deflate(R, U, d, Cb), h)


def _seq_fit(R, u, tau, iters, h):
    """`iters` sequential ALS iterations of §2.3 from u; returns (u, v, d, decrease)."""
    hh = np.ones(R.shape[1]) if h is None else h
    for _ in range(iters):
        v = ternarize(R.T @ u, tau)
        u = ternarize(R @ (hh * v), tau)
    uf, vf = u.astype(np.float64), v.astype(np.float64)
    num = uf @ R @ (hh * vf)
    den = (uf @ uf) * (vf @ (hh * vf))
    d = num / den
    return u, v, d, num * num / den


def decompose_safeguarded(A, mu: float, tau: float, block: int, iters: int, weights=None):
    """The method with Prop. 2's safeguard: every component (b = 1) or block (b > 1) is compared with the best
    single-entry pair and replaced by it when the pair removes more. Returns (Result, activations)."""
    R = np.array(A, dtype=np.float64)
    m, n = R.shape
    h = None if weights is None else np.asarray(weights, dtype=np.float64)
    hh = np.ones(n) if h is None else h
    k = inner_rank(m, n, mu)
    b = block_width(m, n, block)
    B = np.zeros((m, k), np.int8)
    C = np.zeros((k, n), np.int8)
    D = np.zeros(k)
    norm_a = weighted_norm2(R, h)
    trace, act = [], 0
    j0 = 0
    while j0 < k:
        w = min(b, k - j0)
        U0 = ternarize_cols(R[:, initial_columns(R, w, hh)], tau)
        if b == 1:
            u, v, d, dec = _seq_fit(R, U0[:, 0], tau, iters, h)
            U, Cb, dv = u[:, None], v[None, :], np.array([d])
        else:
            U, Cb, dv, dec = _block_fit(R, U0, tau, iters, h)
        i, j, rij, single = best_single_entry(R, h)
        if single > dec:
            act += 1
            U = np.zeros((m, w), np.int8)
            Cb = np.zeros((w, n), np.int8)
            dv = np.zeros(w)
            U[i, 0] = 1
            Cb[0, j] = 1 if rij >= 0 else -1
            dv[0] = abs(rij)
        R = deflate(R, U, dv, Cb)
        B[:, j0:j0 + w], C[j0:j0 + w], D[j0:j0 + w] = U, Cb, dv
        trace.append(1.0 - weighted_norm2(R, h) / norm_a)
        j0 += w
    return Result(B, D, C, trace[-1] if trace else 0.0, trace, R), act


# ----------------------------------------------------------------------------------------------------------
# §2.4: refinement sweeps
# ----------------------------------------------------------------------------------------------------------
def refine(A, res: Result, tau: float, block: int, iters: int, sweeps: int, weights=None):
    """`sweeps` refinement sweeps over the blocks of ``res`` (same block layout as the run that produced it).
    Returns (Result, replaced blocks per sweep)."""
    A64 = np.asarray(A, dtype=np.float64)
    m, n = A64.shape
    h = None if weights is None else np.asarray(weights, dtype=np.float64)
    B, C, D = res.B.copy(), res.C.copy(), res.D.astype(np.float64).copy()
    k = B.shape[1]
    b = block_width(m, n, block)
    R = A64 - B.astype(np.float64) @ (D[:, None] * C.astype(np.float64))
    norm_a = weighted_norm2(A64, h)
    trace, replaced = [], []
    for _ in range(sweeps):
        count = 0
        for j0 in range(0, k, b):
            w = min(b, k - j0)
            U, Cb, d = B[:, j0:j0 + w], C[j0:j0 + w], D[j0:j0 + w]
            Radd = R + U.astype(np.float64) @ (d[:, None] * Cb.astype(np.float64))
            if w == 1:
                u2, v2, d2, _ = _seq_fit(Radd, U[:, 0].copy(), tau, iters, h)
                U2, C2, dv2 = u2[:, None], v2[None, :], np.array([d2])
            else:
                U2, C2, dv2, _ = _block_fit(Radd, U.copy(), tau, iters, h)
            # what each block removes from the added-back residual, as a change of the weighted norm
            base = weighted_norm2(Radd, h)
            old = base - weighted_norm2(deflate(Radd, U, d, Cb), h)
            new = base - weighted_norm2(deflate(Radd, U2, dv2, C2), h)
            if new >= old:
                B[:, j0:j0 + w], C[j0:j0 + w], D[j0:j0 + w] = U2, C2, dv2
                count += 1
            R = deflate(Radd, B[:, j0:j0 + w], D[j0:j0 + w], C[j0:j0 + w])
        replaced.append(count)
        trace.append(1.0 - weighted_norm2(R, h) / norm_a)
    return Result(B, D, C, trace[-1] if trace else res.energy, trace, R), replaced
