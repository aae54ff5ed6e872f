"""Seeded synthetic inputs shaped like the ExTernD paper's workloads.

This module only draws random numbers: it holds none of the method's arithmetic, so both the CPU oracle
(tests) and the CUDA path (tests, bench) can take their inputs from it without sharing any computation.

The paper decomposes real LLM weight matrices (Gemma-4-E2B, Qwen3.5-4B, Granite; §3) and uses llama.cpp
imatrix statistics as channel importances (§2.5). None of those are available here, so each workload below
is a synthetic stand-in of the same shape and a similar value distribution:

* ``gaussian``       i.i.d. N(0, std^2) entries.
* ``outliers``       0.1 % of the entries (chosen without replacement) replaced by ``s * 20 * |x|`` with a
                     uniformly random sign ``s``: the outlier channels of LLM weights.
* ``student_t``      Student-t (nu = 5) entries rescaled to the requested standard deviation: the heavy tails of
                     LLM MLP weights.
* ``importance``     per-input-channel second moments ``h_j = exp(N(0, 1))`` (log-normal, an imatrix-like skew),
                     returned already normalised as ``h / max(h)`` (lambda = 0 in §2.5).

Every generator uses numpy's PCG64 (``numpy.random.default_rng(seed)``) and draws in a fixed order, so a seed
fixes the matrix bit for bit on every machine.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Iterator

import numpy as np


def gaussian(m: int, n: int, std: float, seed: int) -> np.ndarray:
    """m x n fp32 matrix with i.i.d. N(0, std^2) entries."""
    rng = np.random.default_rng(seed)
    return (rng.standard_normal((m, n)) * std).astype(np.float32)


def gaussian_with_outliers(m: int, n: int, std: float, frac: float, factor: float, seed: int) -> np.ndarray:
    """N(0, std^2) matrix where ``round(frac*m*n)`` entries become ``s * factor * |x|`` with random sign s."""
    rng = np.random.default_rng(seed)
    a = rng.standard_normal((m, n)) * std
    count = int(round(frac * m * n))
    pos = rng.choice(m * n, size=count, replace=False)
    sign = rng.choice(np.array([-1.0, 1.0]), size=count)
    flat = a.reshape(-1)
    flat[pos] = sign * factor * np.abs(flat[pos])
    return a.astype(np.float32)


def student_t(m: int, n: int, nu: float, std: float, seed: int) -> np.ndarray:
    """Student-t(nu) entries scaled to standard deviation ``std`` (variance of t(nu) is nu/(nu-2))."""
    rng = np.random.default_rng(seed)
    a = rng.standard_t(nu, size=(m, n)) * (std / math.sqrt(nu / (nu - 2.0)))
    return a.astype(np.float32)


def importance(n: int, seed: int) -> np.ndarray:
    """Log-normal(0, 1) per-column importances, normalised to max 1 (h/max(h), lambda = 0)."""
    rng = np.random.default_rng(seed)
    h = np.exp(rng.standard_normal(n))
    return (h / h.max()).astype(np.float32)


def ternary(rows: int, cols: int, density: float, seed: int) -> np.ndarray:
    """Random int8 matrix in {-1, 0, +1} with P(nonzero) = density and equiprobable signs."""
    rng = np.random.default_rng(seed)
    nz = rng.random((rows, cols)) < density
    sign = np.where(rng.random((rows, cols)) < 0.5, -1, 1)
    return (nz * sign).astype(np.int8)


@dataclasses.dataclass(frozen=True)
class Workload:
    """One decomposition problem: the matrix recipe plus the method's parameters."""

    name: str
    m: int
    n: int
    mu: float
    tau: float
    block: int
    iters: int
    kind: str            # "gaussian" | "outliers" | "student_t"
    std: float
    seed: int
    weighted: bool = False

    def matrix(self) -> np.ndarray:
        if self.kind == "gaussian":
            return gaussian(self.m, self.n, self.std, self.seed)
        if self.kind == "outliers":
            return gaussian_with_outliers(self.m, self.n, self.std, 1e-3, 20.0, self.seed)
        if self.kind == "student_t":
            return student_t(self.m, self.n, 5.0, self.std, self.seed)
        raise ValueError(self.kind)

    def weights(self) -> np.ndarray | None:
        # The importances take their own stream (seed + 7919) so the matrix does not depend on them.
        return importance(self.n, self.seed + 7919) if self.weighted else None


# The five benchmark problems: a 256x256 sequential case, a 2048x2048 matrix with outliers, an MLP
# up-projection, an importance-weighted attention projection and a whole 36-layer 4B-class decoder.
SEQUENTIAL_256 = Workload("seq256_gauss_mu2_b1", 256, 256, 2.0, 0.7, 1, 4, "gaussian", 0.02, 0)
OUTLIER_2048 = Workload("outlier2048_mu3_b64", 2048, 2048, 3.0, 0.7, 64, 4, "outliers", 0.02, 1)
MLP_UP_2560x9728 = Workload("up2560x9728_t5_mu3_tau1_b128", 2560, 9728, 3.0, 1.0, 128, 4, "student_t", 0.015, 2)
ATTN_4096_WEIGHTED = Workload("attn4096_weighted_mu2.5_b128", 4096, 4096, 2.5, 0.7, 128, 4, "gaussian", 0.02, 3,
                              weighted=True)

DECODER_LAYERS = 36
DECODER_SHAPES = (("q", 2560, 4096), ("k", 2560, 1024), ("v", 2560, 1024), ("o", 4096, 2560),
                  ("gate", 2560, 9728), ("up", 2560, 9728), ("down", 9728, 2560))


def decoder_conversion(layers: int = DECODER_LAYERS) -> Iterator[Workload]:
    """The 36-layer decoder, matrix by matrix; seed = 1000 + 10*layer + index of the projection name."""
    for layer in range(layers):
        for idx, (name, m, n) in enumerate(DECODER_SHAPES):
            yield Workload(f"L{layer}.{name}", m, n, 3.0, 0.7, 128, 4, "student_t", 0.015, 1000 + 10 * layer + idx)


WORKLOADS = {w.name: w for w in (SEQUENTIAL_256, OUTLIER_2048, MLP_UP_2560x9728, ATTN_4096_WEIGHTED)}
