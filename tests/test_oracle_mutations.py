"""The oracle's pins catch plausible slips: each mutation below plants one mistake in a copy of the oracle
(oracle/externd_oracle.py), and at least one pin of tests/test_oracle_pins.py must then fail.

The mutations are the slips a restatement of §2.2-§2.5 could plausibly contain: a wrong or missing term, a
swapped row/column orientation, a stale intermediate, a wrong sign, an off-by-one in a mean, a dropped weight.
Nothing here touches the CUDA path; the oracle module itself is never modified (each mutant is a fresh module
built from the source text).
"""
import inspect
import itertools
import os
import sys
import types
import warnings

import pytest

import tests.test_oracle_pins as PINS
from oracle import externd_oracle as O

SOURCE = open(os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "oracle",
                           "externd_oracle.py")).read()

# name -> list of (old text, new text) replacements, each old text occurring exactly once in the oracle
MUTATIONS = {
    "eq2 non-strict threshold": [("keep = mag > theta", "keep = mag >= theta")],
    "eq2 mean over L - 1": [("theta = tau * (math.fsum(mag.tolist()) / length)",
                             "theta = tau * (math.fsum(mag.tolist()) / max(1, length - 1))")],
    "eq2 fallback drops the sign": [("t[i] = -1 if x[i] < 0 else 1", "t[i] = 1")],
    "eq2 fallback keeps the last maximum": [("i = int(np.argmax(mag))", "i = int(mag.size - 1 - np.argmax(mag[::-1]))")],
    "initial columns of smallest energy": [("order = np.lexsort((np.arange(energy.size), -energy))",
                                            "order = np.lexsort((np.arange(energy.size), energy))")],
    "initial columns ties to the higher index": [("order = np.lexsort((np.arange(energy.size), -energy))",
                                                  "order = np.lexsort((-np.arange(energy.size), -energy))")],
    "eq3 ridge missing": [("return EPS_REL * float(np.trace(G)) / G.shape[0]", "return 0.0 * float(np.trace(G))")],
    "eq3 ridge not relative": [("return EPS_REL * float(np.trace(G)) / G.shape[0]", "return EPS_REL")],
    "eq4 ridge on a single component": [("    if K.shape[0] > 1:\n        K = K + ridge(K)",
                                         "    if K.shape[0] >= 1:\n        K = K + ridge(K)")],
    "eq4 without the V gram": [("K = gram_u(U) * gram_v(Cb, h)", "K = gram_u(U) * np.eye(gram_u(U).shape[0])")],
    "eq4 r from the wrong product axis": [("r = np.sum(np.asarray(U, dtype=np.float64) * np.asarray(PU, dtype=np.float64), axis=0)",
                                           "r = np.sum(np.asarray(U, dtype=np.float64), axis=0) * np.sum(np.asarray(PU, dtype=np.float64), axis=0) / np.asarray(U).shape[0]")],
    "deflation with the wrong sign": [("return np.asarray(R, dtype=np.float64) - (U * np.asarray(d, dtype=np.float64))",
                                       "return np.asarray(R, dtype=np.float64) + (U * np.asarray(d, dtype=np.float64))")],
    "sec25 weighted v-step (correction dropped)": [("Cb = ternarize_rows(vstep_target(R, U), tau)        # V",
                                                    "Cb = ternarize_rows(vstep_solve(np.asarray(U, dtype=np.float64).T @ (R * hh[None, :]), U), tau)        # V")],
    "sec25 u-step unweighted": [("PU = ustep_product(R, Cb, h)                        # R H V",
                                 "PU = ustep_product(R, Cb, None)                        # R H V")],
    "block v ternarized along columns": [("Cb = ternarize_rows(vstep_target(R, U), tau)        # V",
                                          "Cb = ternarize_cols(vstep_target(R, U), tau)        # V")],
    "block u ternarized along rows": [("U = ternarize_cols(ustep_solve(PU, Cb, h), tau)     # U",
                                       "U = ternarize_rows(ustep_solve(PU, Cb, h), tau)     # U")],
    "block scales from the initial U (stale)": [
        ("        U = ternarize_cols(R[:, initial_columns(R, w, hh)], tau)\n",
         "        U = ternarize_cols(R[:, initial_columns(R, w, hh)], tau)\n        U0 = U\n"),
        ("d = block_scales(U, Cb, PU, h)                          # Eq. 4",
         "d = block_scales(U0, Cb, PU, h)                          # Eq. 4")],
    "block scales from the first iteration's product (stale PU)": [
        ("            PU = ustep_product(R, Cb, h)                        # R H V\n",
         "            PU = ustep_product(R, Cb, h)                        # R H V\n"
         "            PU_first = PU if _ == 0 else PU_first\n"),
        ("d = block_scales(U, Cb, PU, h)                          # Eq. 4",
         "d = block_scales(U, Cb, PU_first, h)                          # Eq. 4")],
    "sequential scale without the v norm": [("d = (uf @ R @ (h * vf)) / ((uf @ uf) * (vf @ (h * vf)))",
                                             "d = (uf @ R @ (h * vf)) / (uf @ uf)")],
    "sequential v-step on the weighted residual": [("v = ternarize(R.T @ u, tau)", "v = ternarize((R * h[None, :]).T @ u, tau)")],
    "energy before deflation": [("        trace.append(1.0 - weighted_norm2(R, h) / norm_a)\n        j0 += w",
                                 "        trace.append(1.0 - weighted_norm2(R + (U * d) @ Cb, h) / norm_a)\n        j0 += w")],
    "block width cap at min / 4": [("return max(1, min(int(block), min(m, n) // 8))",
                                    "return max(1, min(int(block), min(m, n) // 4))")],
    "inner rank truncated": [("return int(math.floor(mu * min(m, n) + 0.5))", "return int(math.floor(mu * min(m, n)))")],
    "eq3 v-step without the gram inverse (naive batching)": [("    return vstep_solve(vstep_product(R, U), U)",
                                                              "    return vstep_product(R, U)")],
    "eq3 u-step without the gram inverse": [
        ("    return np.linalg.solve(G + ridge(G) * np.eye(G.shape[0]), np.asarray(PU, dtype=np.float64).T).T",
         "    return np.asarray(PU, dtype=np.float64)")],
    "sec25 u-step gram unweighted": [("    G = gram_v(Cb, h)\n    return np.linalg.solve",
                                      "    G = gram_v(Cb, None)\n    return np.linalg.solve")],
    "initial columns by unweighted energy": [
        ("energy = np.asarray(h, dtype=np.float64) * np.sum(np.asarray(R, dtype=np.float64) ** 2, axis=0)",
         "energy = np.sum(np.asarray(R, dtype=np.float64) ** 2, axis=0)")],
    "eq2 threshold from the largest magnitude": [("theta = tau * (math.fsum(mag.tolist()) / length)",
                                                  "theta = tau * float(mag.max())")],
    "deflation without the scales": [
        ("return np.asarray(R, dtype=np.float64) - (U * np.asarray(d, dtype=np.float64)) @ np.asarray(Cb, dtype=np.float64)",
         "return np.asarray(R, dtype=np.float64) - U @ np.asarray(Cb, dtype=np.float64)")],
    "weighted energy over the unweighted norm of A": [
        ("return 1.0 - weighted_norm2(A - Ahat, h) / weighted_norm2(A, h)",
         "return 1.0 - weighted_norm2(A - Ahat, h) / weighted_norm2(A, None)")],
    "sequential u-step on the unweighted residual": [("u = ternarize(R @ (h * v), tau)", "u = ternarize(R @ v, tau)")],
    "eq4 r without U": [("r = np.sum(np.asarray(U, dtype=np.float64) * np.asarray(PU, dtype=np.float64), axis=0)",
                         "r = np.sum(np.asarray(PU, dtype=np.float64), axis=0)")],
    "eq3 ridge over the trace, not its mean": [("return EPS_REL * float(np.trace(G)) / G.shape[0]",
                                                 "return EPS_REL * float(np.trace(G))")],
}


def mutant(name):
    src = SOURCE
    for old, new in MUTATIONS[name]:
        assert src.count(old) == 1, (name, old)
        src = src.replace(old, new)
    mod = types.ModuleType(f"oracle_mutant_{abs(hash(name))}")
    sys.modules[mod.__name__] = mod   # the oracle's dataclass looks its module up while being defined
    try:
        exec(compile(src, f"<mutant {name}>", "exec"), mod.__dict__)
    finally:
        del sys.modules[mod.__name__]
    return mod


def pin_cases():
    """Every test of test_oracle_pins with its parametrizations, as (label, callable, kwargs)."""
    for fname, fn in inspect.getmembers(PINS, inspect.isfunction):
        if not fname.startswith("test_"):
            continue
        marks = [m for m in getattr(fn, "pytestmark", []) if m.name == "parametrize"]
        if not marks:
            yield fname, fn, {}
            continue
        grids = []
        for m in marks:
            names = [s.strip() for s in m.args[0].split(",")] if isinstance(m.args[0], str) else list(m.args[0])
            grids.append([dict(zip(names, v if len(names) > 1 else (v,))) for v in m.args[1]])
        for combo in itertools.product(*grids):
            kw = {}
            for part in combo:
                kw.update(part)
            yield f"{fname}{kw}", fn, kw


def first_failing_pin(mod):
    saved = PINS.O
    PINS.O = mod
    try:
        for label, fn, kw in pin_cases():
            try:
                with warnings.catch_warnings():
                    warnings.simplefilter("ignore")
                    fn(**kw)
            except Exception:   # an assertion, or the mutant breaking a shape: either way the pin caught it
                return label
        return None
    finally:
        PINS.O = saved


def test_the_unmutated_oracle_passes_every_pin():
    assert first_failing_pin(O) is None


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_planted_slip_fails_a_pin(name):
    assert first_failing_pin(mutant(name)) is not None, f"no pin catches: {name}"
