"""The pins of the oracle's second part catch plausible slips: each mutation below plants one mistake in a copy
of oracle/externd_next.py (rank budgets, mask+sign packing and the inference product, Prop. 2's safeguard,
refinement sweeps), and at least one pin of tests/test_oracle_next.py must then fail.

The oracle module itself is never modified: each mutant is a fresh module built from the source text, whose
functions stand in for the originals in the `oracle` package namespace while the pins run.
"""
import inspect
import itertools
import os
import sys
import types
import warnings

import pytest

import oracle
import tests.test_oracle_next as PINS

SOURCE = open(os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "oracle",
                           "externd_next.py")).read()

# name -> list of (old text, new text) replacements, each old text occurring exactly once in the source
MUTATIONS = {
    "rank for energy: strictly above the target": [("        if e >= target:\n            return k",
                                                    "        if e > target:\n            return k")],
    "rank for energy: the boundary before": [("    for e, k in zip(trace, ranks):\n        if e >= target:\n            return k",
                                              "    prev = None\n    for e, k in zip(trace, ranks):\n        if e >= target:\n"
                                              "            return prev if prev is not None else k\n        prev = k")],
    "block boundaries from the uncapped block": [("k, b = inner_rank(m, n, mu), block_width(m, n, block)",
                                                  "k, b = inner_rank(m, n, mu), max(1, int(block))")],
    "allocation ignores the budget": [("            if spent + cost > budget + 1e-12:\n                continue\n",
                                       "")],
    "allocation picks the smallest gain": [("            if best is None or gain > best:",
                                                                     "            if best is None or gain < best:")],
    "packing: a sign bit for every element": [("sign = (t[t != 0] < 0).astype(np.uint8)",
                                               "sign = (t < 0).astype(np.uint8)")],
    "packing: sign bit set for positives": [("sign = (t[t != 0] < 0).astype(np.uint8)",
                                             "sign = (t[t != 0] > 0).astype(np.uint8)")],
    "eq5 without the sign bits": [("return mu * (m + n) / max(m, n) * (2.0 - sparsity)",
                                   "return mu * (m + n) / max(m, n) * (1.0 - sparsity)")],
    "eq5 over min(m, n)": [("return mu * (m + n) / max(m, n) * (2.0 - sparsity)",
                            "return mu * (m + n) / min(m, n) * (2.0 - sparsity)")],
    "inference product without D": [("z = np.asarray(D, np.float64) * (np.asarray(C, np.float64) @ np.asarray(x, np.float64))",
                                     "z = np.asarray(C, np.float64) @ np.asarray(x, np.float64)")],
    "inference product with x reversed": [("(np.asarray(C, np.float64) @ np.asarray(x, np.float64))",
                                            "(np.asarray(C, np.float64) @ np.asarray(x, np.float64)[::-1])")],
    "best single entry ignores the weights": [("score = hh[None, :] * R * R", "score = R * R")],
    "best single entry by |R| not R^2": [("score = hh[None, :] * R * R", "score = hh[None, :] * np.abs(R)")],
    "safeguard takes the pair when it removes less": [("        if single > dec:", "        if single < dec:")],
    "safeguard pair without its sign": [("Cb[0, j] = 1 if rij >= 0 else -1", "Cb[0, j] = 1")],
    "safeguard pair scaled by R_ij^2": [("dv[0] = abs(rij)", "dv[0] = rij * rij")],
    "sequential fit without the v norm": [("den = (uf @ uf) * (vf @ (hh * vf))", "den = (uf @ uf)")],
    "refinement keeps every refit": [("            if new >= old:", "            if True:")],
    "refinement starts from A": [("R = A64 - B.astype(np.float64) @ (D[:, None] * C.astype(np.float64))",
                                  "R = A64.copy()")],
    "refinement refits the residual without the block added back": [
        ("                U2, C2, dv2, _ = _block_fit(Radd, U.copy(), tau, iters, h)",
         "                U2, C2, dv2, _ = _block_fit(R, U.copy(), tau, iters, h)")],
}


def mutant(name):
    src = SOURCE
    for old, new in MUTATIONS[name]:
        assert src.count(old) == 1, (name, old)
        src = src.replace(old, new)
    mod = types.ModuleType(f"oracle.next_mutant_{abs(hash(name))}")
    mod.__package__ = "oracle"   # the relative import of the first part
    sys.modules[mod.__name__] = mod
    try:
        exec(compile(src, f"<mutant {name}>", "exec"), mod.__dict__)
    finally:
        del sys.modules[mod.__name__]
    return mod


def pin_cases():
    """Every test of test_oracle_next with its parametrizations, as (label, callable, kwargs)."""
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


NAMES = ["block_boundaries", "rank_for_energy", "allocate_ranks", "pack_mask_sign", "unpack_mask_sign", "bpw_eff",
         "ternary_apply", "best_single_entry", "decompose_safeguarded", "refine"]


def first_failing_pin(mod):
    saved = {nm: getattr(oracle, nm) for nm in NAMES}
    for nm in NAMES:
        setattr(oracle, nm, getattr(mod, nm))
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
        for nm, f in saved.items():
            setattr(oracle, nm, f)


def test_the_unmutated_oracle_passes_every_pin():
    import oracle.externd_next as N
    assert first_failing_pin(N) is None


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_planted_slip_fails_a_pin(name):
    assert first_failing_pin(mutant(name)) is not None, f"no pin catches: {name}"
