"""ExTernD oracle: a plain, slow, fp64 CPU restatement of the factorization method.

TEST INFRASTRUCTURE ONLY. This module exists to check the CUDA library. Only ``tests/``,
``__graft_entry__.smoke()`` and the CPU-baseline leg of ``bench.py`` may import it; the product path (the
CUDA library and its Python binding) never does, and the two share no code.

Every function follows the ExTernD paper (arxiv 2607.13511, "Expanded-Rank Ternary Decomposition") and cites
the section or equation it restates. Everything is computed in float64 with numpy; a numpy library primitive
(matmul, solve, sort) serves as a single step, with no blocking or reordering beyond what the paper states.

Readings taken where the paper is silent:

* Ridge in Eq. 3: ``eps = EPS_REL * trace(G) / w`` (relative, so scaling the importances does not change the
  factors). Eq. 4 gets the same relative ridge when the block has ``w > 1`` components; a 1x1 system is
  solved exactly (it is Prop. 1's closed form, always positive).
* Eq. 2: the mean is over the vector's own length L; the kept set is ``|x_i| > tau * (S / L)`` with
  ``S = sum_j |x_j|`` summed exactly (``math.fsum``) and the product/quotient taken in float64; sign(0) never
  passes; the all-zero fallback keeps the first index of maximal magnitude, with sign +1 when that entry is 0.
* Initial ternary factor of each component/block (the paper starts at "v <- T(R^T u)" without saying where
  u comes from): the w columns of R with the largest weighted energy ``h_j * ||R[:, j]||^2`` (ties to the
  lower column index), in ascending column order, each ternarized with Eq. 2.
* One ALS iteration is a V-step followed by a U-step; ``iters`` iterations, no early exit; the scales use
  the final U, the final V and the last U-step's product R H V.
* The inner rank is ``k = floor(mu * min(m, n) + 0.5)``; the block width is ``min(block, floor(min(m,n)/8))``
  but at least 1; the last block is ``k mod b`` wide when that is non-zero.
* Importance weighting (§2.5): ``weights`` is h~ itself (the caller forms h/max(h) + lambda); columns index
  input channels.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

EPS_REL = 1e-4


# ----------------------------------------------------------------------------------------------------------
# §2.1, §2.4: sizes
# ----------------------------------------------------------------------------------------------------------
def inner_rank(m: int, n: int, mu: float) -> int:
    """§2.1: inner rank k = mu * min(m, n), rounded to the nearest integer (halves up)."""
    return int(math.floor(mu * min(m, n) + 0.5))


def block_width(m: int, n: int, block: int) -> int:
    """§2.4: block width, capped at floor(min(m, n) / 8); at least 1."""
    return max(1, min(int(block), min(m, n) // 8))


# ----------------------------------------------------------------------------------------------------------
# §2.2, Eq. 2: ternarization
# ----------------------------------------------------------------------------------------------------------
def ternarize(x, tau: float) -> np.ndarray:
    """Eq. 2: T_tau(x)_i = sign(x_i) * 1[|x_i| > tau * (1/L) * sum_j |x_j|].

    If no entry passes, the single largest-magnitude entry is kept (§2.2)."""
    x = np.asarray(x, dtype=np.float64).reshape(-1)
    length = x.size
    mag = np.abs(x)
    theta = tau * (math.fsum(mag.tolist()) / length)
    keep = mag > theta
    t = np.zeros(length, dtype=np.int8)
    t[keep] = np.where(x[keep] < 0, -1, 1)
    if not keep.any():
        i = int(np.argmax(mag))
        t[i] = -1 if x[i] < 0 else 1
    return t


def ternarize_rows(X, tau: float) -> np.ndarray:
    """Eq. 2 applied to every row of X (each row is one vector)."""
    X = np.asarray(X, dtype=np.float64)
    return np.stack([ternarize(X[i], tau) for i in range(X.shape[0])]).astype(np.int8)


def ternarize_cols(Y, tau: float) -> np.ndarray:
    """Eq. 2 applied to every column of Y (each column is one vector)."""
    return np.ascontiguousarray(ternarize_rows(np.asarray(Y).T, tau).T)


def ternary_projection(u) -> tuple[np.ndarray, float]:
    """§2.2: the optimal ternary projection argmin_{t, alpha} ||u - alpha t||_2.

    Sort |u| in decreasing order and keep the prefix of length s* that maximises (1/sqrt(s)) sum_{i<=s} |u|_(i);
    t = sign(u) on the kept entries and alpha = mean of the kept |u|."""
    u = np.asarray(u, dtype=np.float64).reshape(-1)
    order = np.argsort(-np.abs(u), kind="stable")
    prefix = np.cumsum(np.abs(u)[order])
    s = np.arange(1, u.size + 1)
    best = int(np.argmax(prefix / np.sqrt(s))) + 1
    t = np.zeros(u.size, dtype=np.int8)
    kept = order[:best]
    t[kept] = np.where(u[kept] < 0, -1, 1)
    return t, float(prefix[best - 1] / best)


# ----------------------------------------------------------------------------------------------------------
# Start of each component / block (reading: the paper does not say how u is initialised)
# ----------------------------------------------------------------------------------------------------------
def initial_columns(R, w: int, h) -> np.ndarray:
    """Indices of the w columns of R with the largest h_j * ||R[:, j]||^2 (ties -> lower j), ascending."""
    energy = np.asarray(h, dtype=np.float64) * np.sum(np.asarray(R, dtype=np.float64) ** 2, axis=0)
    order = np.lexsort((np.arange(energy.size), -energy))
    return np.sort(order[:w])


# ----------------------------------------------------------------------------------------------------------
# §2.4 Eq. 3, §2.5: decorrelated block targets
# ----------------------------------------------------------------------------------------------------------
def ridge(G) -> float:
    """The +eps I of Eq. 3: EPS_REL times the mean diagonal of the Gram matrix."""
    G = np.asarray(G, dtype=np.float64)
    return EPS_REL * float(np.trace(G)) / G.shape[0]


def vstep_product(R, U) -> np.ndarray:
    """The V-step residual product U^T R (w x n); U is m x w. Plain R even when weighted (§2.5)."""
    return np.asarray(U, dtype=np.float64).T @ np.asarray(R, dtype=np.float64)


def ustep_product(R, Cb, h=None) -> np.ndarray:
    """The U-step residual product R diag(h) V (m x w), with V = Cb^T and Cb the w x n block of C (§2.5)."""
    R = np.asarray(R, dtype=np.float64)
    V = np.asarray(Cb, dtype=np.float64).T
    if h is not None:
        V = np.asarray(h, dtype=np.float64)[:, None] * V
    return R @ V


def gram_u(U) -> np.ndarray:
    """U^T U (w x w), the Gram matrix of the V-step in Eq. 3."""
    U = np.asarray(U, dtype=np.float64)
    return U.T @ U


def gram_v(Cb, h=None) -> np.ndarray:
    """V^T diag(h) V (w x w) with V = Cb^T: the Gram matrix of the U-step (Eq. 3, §2.5)."""
    V = np.asarray(Cb, dtype=np.float64).T
    HV = V if h is None else np.asarray(h, dtype=np.float64)[:, None] * V
    return V.T @ HV


def vstep_solve(PV, U) -> np.ndarray:
    """Eq. 3 (left) given PV = U^T R: X = (U^T U + eps I)^{-1} PV, w x n."""
    G = gram_u(U)
    return np.linalg.solve(G + ridge(G) * np.eye(G.shape[0]), np.asarray(PV, dtype=np.float64))


def ustep_solve(PU, Cb, h=None) -> np.ndarray:
    """Eq. 3 (right) given PU = R H V: Y = PU (V^T H V + eps I)^{-1}, m x w (the Gram is symmetric)."""
    G = gram_v(Cb, h)
    return np.linalg.solve(G + ridge(G) * np.eye(G.shape[0]), np.asarray(PU, dtype=np.float64).T).T


def vstep_target(R, U) -> np.ndarray:
    """Eq. 3 (left): X = (U^T U + eps I)^{-1} U^T R, w x n. Row a of X is component a's V target."""
    return vstep_solve(vstep_product(R, U), U)


def ustep_target(R, Cb, h=None) -> np.ndarray:
    """Eq. 3 (right) with §2.5 weighting: Y = R H V (V^T H V + eps I)^{-1}, m x w. Column a targets u_a."""
    return ustep_solve(ustep_product(R, Cb, h), Cb, h)


# ----------------------------------------------------------------------------------------------------------
# §2.3, §2.4 Eq. 4, §2.5: scales and deflation
# ----------------------------------------------------------------------------------------------------------
def block_scales(U, Cb, PU, h=None) -> np.ndarray:
    """Eq. 4 with §2.5 weighting: [(U^T U) * (V^T H V)] d = diag(U^T R H V), where PU = R H V.

    A 1x1 system is Prop. 1's scale u^T R H v / (||u||^2 v^T H v); larger systems get the relative ridge."""
    K = gram_u(U) * gram_v(Cb, h)
    r = np.sum(np.asarray(U, dtype=np.float64) * np.asarray(PU, dtype=np.float64), axis=0)
    if K.shape[0] > 1:
        K = K + ridge(K) * np.eye(K.shape[0])
    return np.linalg.solve(K, r)


def deflate(R, U, d, Cb) -> np.ndarray:
    """§2.3 step 3 / §2.4: R - U diag(d) V^T (returns a new array)."""
    U = np.asarray(U, dtype=np.float64)
    return np.asarray(R, dtype=np.float64) - (U * np.asarray(d, dtype=np.float64)) @ np.asarray(Cb, dtype=np.float64)


def weighted_norm2(R, h=None) -> float:
    """sum_ij h_j R_ij^2 (h = 1 when unweighted): the objective of §2.5 / the Frobenius norm of Eq. 1."""
    col = np.sum(np.asarray(R, dtype=np.float64) ** 2, axis=0)
    return float(col.sum() if h is None else np.dot(np.asarray(h, dtype=np.float64), col))


def energy(A, B, D, C, h=None) -> float:
    """Eq. 1: E = 1 - ||A - B diag(D) C||^2 / ||A||^2 (weighted form of §2.5 when h is given)."""
    A = np.asarray(A, dtype=np.float64)
    Ahat = (np.asarray(B, dtype=np.float64) * np.asarray(D, dtype=np.float64)) @ np.asarray(C, dtype=np.float64)
    return 1.0 - weighted_norm2(A - Ahat, h) / weighted_norm2(A, h)


# ----------------------------------------------------------------------------------------------------------
# Algorithms
# ----------------------------------------------------------------------------------------------------------
@dataclass
class Result:
    B: np.ndarray                # m x k int8
    D: np.ndarray                # k float64
    C: np.ndarray                # k x n int8
    energy: float                # 1 - ||R||_H^2 / ||A||_H^2 from the tracked residual
    trace: list = field(default_factory=list)   # energy after each component (b = 1) or block (b > 1)
    R: np.ndarray | None = None  # final residual


def sequential_als(A, mu: float, tau: float, iters: int, weights=None) -> Result:
    """§2.3 greedy sequential ALS (with the §2.5 weighting: U-step on W = R (.) h~, V-step on plain R)."""
    R = np.array(A, dtype=np.float64)
    m, n = R.shape
    h = np.ones(n) if weights is None else np.asarray(weights, dtype=np.float64)
    k = inner_rank(m, n, mu)
    B = np.zeros((m, k), np.int8)
    C = np.zeros((k, n), np.int8)
    D = np.zeros(k)
    norm_a = weighted_norm2(R, h)
    trace = []
    for i in range(k):
        u = ternarize(R[:, initial_columns(R, 1, h)[0]], tau)
        for _ in range(iters):
            v = ternarize(R.T @ u, tau)               # step 1: v <- T(R^T u)
            u = ternarize(R @ (h * v), tau)           # step 1: u <- T(R v), weighted target R H v
        uf, vf = u.astype(np.float64), v.astype(np.float64)
        d = (uf @ R @ (h * vf)) / ((uf @ uf) * (vf @ (h * vf)))   # step 2 / Prop. 1
        R -= d * np.outer(uf, vf)                                   # step 3
        B[:, i], C[i], D[i] = u, v, d
        trace.append(1.0 - weighted_norm2(R, h) / norm_a)
    return Result(B, D, C, trace[-1] if trace else 0.0, trace, R)


def block_als(A, mu: float, tau: float, block: int, iters: int, weights=None) -> Result:
    """§2.4 batched block ALS with decorrelated targets (Eq. 3), joint scales (Eq. 4) and sequential
    deflation across blocks; §2.5 weighting (V-step on plain R, U-step and scales with h~)."""
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
    trace = []
    j0 = 0
    while j0 < k:
        w = min(b, k - j0)
        U = ternarize_cols(R[:, initial_columns(R, w, hh)], tau)
        for _ in range(iters):
            Cb = ternarize_rows(vstep_target(R, U), tau)        # V <- T([(U^T U + eps I)^-1 U^T R]^T)
            PU = ustep_product(R, Cb, h)                        # R H V
            U = ternarize_cols(ustep_solve(PU, Cb, h), tau)     # U <- T(R H V (V^T H V + eps I)^-1)
        d = block_scales(U, Cb, PU, h)                          # Eq. 4
        R = deflate(R, U, d, Cb)                                # R <- R - U diag(d) V^T
        B[:, j0:j0 + w], C[j0:j0 + w], D[j0:j0 + w] = U, Cb, d
        trace.append(1.0 - weighted_norm2(R, h) / norm_a)
        j0 += w
    return Result(B, D, C, trace[-1] if trace else 0.0, trace, R)


def decompose(A, mu: float, tau: float, block: int, iters: int, weights=None) -> Result:
    """ExTernD: A ~ B diag(D) C (Eq. 1). Block width 1 is the sequential algorithm of §2.3, wider blocks the
    batched algorithm of §2.4."""
    A = np.asarray(A)
    if block_width(A.shape[0], A.shape[1], block) == 1:
        return sequential_als(A, mu, tau, iters, weights)
    return block_als(A, mu, tau, block, iters, weights)
