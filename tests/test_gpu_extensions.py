"""The two extensions of the block loop on the GPU against the oracle: Prop. 2's safeguard and §2.4's refinement.

End to end the bar is the energy (|dE| <= 1e-4, as for the plain method: a near-tie trit may flip between float32
and float64), plus what holds for any valid run: Prop. 2's geometric bound after every component, the plain result
when the safeguard never fires, a monotone refinement trace, and the energy recomputed from the returned factors
equal to the tracked one within 1e-5.
"""
import numpy as np
import pytest

from oracle import externd_next as N
from oracle import externd_oracle as O
from paper_2607_13511_gb300 import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def X():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2607_13511_gb300 as X
    from paper_2607_13511_gb300 import build
    build.build()
    X.load()
    return X


def cuda(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def host(res):
    return res.B.cpu().numpy(), res.D.cpu().numpy(), res.C.cpu().numpy()


def spiky(m, n, seed, spikes=3):
    """Small noise with a few large isolated entries: tau = 0 fits dense sign patterns the pairs beat."""
    rng = np.random.default_rng(seed)
    A = 0.01 * rng.standard_normal((m, n))
    for _ in range(spikes):
        A[rng.integers(m), rng.integers(n)] = rng.choice([-1.0, 1.0]) * rng.uniform(0.5, 1.5)
    return A.astype(np.float32)


# ------------------------------------------------------------------------------------------------- Prop. 2
@pytest.mark.parametrize("seed", range(6))
def test_safeguard_geometric_bound(X, seed):
    rng = np.random.default_rng(seed)
    m, n = int(rng.integers(3, 8)), int(rng.integers(3, 8))
    A = (rng.standard_normal((m, n)) * np.exp(rng.standard_normal((m, n)))).astype(np.float32)
    tau = float(rng.choice([0.0, 0.7, 2.0]))
    res, _ = X.decompose_safeguarded(cuda(A), 3.0, tau, 1, 3)
    for k, e in enumerate(res.trace, start=1):
        assert 1.0 - e <= (1.0 - 1.0 / (m * n)) ** k + 1e-6
    ref, _ = N.decompose_safeguarded(A.astype(np.float64), 3.0, tau, 1, 3)
    assert abs(res.energy - ref.energy) <= 1e-4


@pytest.mark.parametrize("m,n,block", [(8, 8, 1), (40, 56, 1), (64, 96, 8), (128, 160, 16)])
def test_safeguard_matches_oracle_on_spikes(X, m, n, block):
    A = spiky(m, n, m + n)
    res, act = X.decompose_safeguarded(cuda(A), 0.25, 0.0, block, 3)
    ref, ref_act = N.decompose_safeguarded(A.astype(np.float64), 0.25, 0.0, block, 3)
    assert ref_act >= 1 and act == ref_act
    B, D, C = host(res)
    np.testing.assert_array_equal(B, ref.B)
    np.testing.assert_array_equal(C, ref.C)
    np.testing.assert_allclose(D, ref.D, rtol=1e-5, atol=1e-7)
    assert abs(res.energy - ref.energy) <= 1e-4
    e2 = X.energy(cuda(A), res.B, res.D, res.C)
    assert abs(e2 - res.energy) <= 1e-5


@pytest.mark.parametrize("block", [1, 8, 32])
def test_safeguard_inactive_is_the_plain_method(X, block):
    A = W.gaussian(96, 200, 0.02, 9).astype(np.float32)
    res, act = X.decompose_safeguarded(cuda(A), 1.0, 0.7, block, 3)
    plain = X.decompose_traced(cuda(A), 1.0, 0.7, block, 3)
    torch.cuda.synchronize()
    assert act == 0
    assert torch.equal(res.B, plain.B) and torch.equal(res.C, plain.C) and torch.equal(res.D, plain.D)
    assert res.trace == plain.trace


def test_safeguard_weighted(X):
    A = spiky(48, 64, 5, spikes=4)
    h = W.importance(64, 3).astype(np.float32)
    res, act = X.decompose_safeguarded(cuda(A), 0.5, 0.0, 4, 3, cuda(h))
    ref, ref_act = N.decompose_safeguarded(A.astype(np.float64), 0.5, 0.0, 4, 3, h.astype(np.float64))
    assert act == ref_act >= 1
    assert abs(res.energy - ref.energy) <= 1e-4
    e2 = X.energy(cuda(A), res.B, res.D, res.C, cuda(h))
    assert abs(e2 - res.energy) <= 1e-5


# ------------------------------------------------------------------------------------------ refinement sweeps
REFINE_CASES = [  # m, n, mu, tau, block, iters, sweeps, weighted
    (40, 64, 1.5, 1.0, 1, 3, 3, False),
    (96, 128, 1.5, 1.0, 8, 3, 3, False),
    (200, 150, 1.3, 1.0, 16, 3, 2, False),
    (130, 257, 1.2, 0.7, 32, 2, 2, True),
    (44, 33, 1.3, 0.7, 4, 2, 2, False),      # tail block of 3
]


@pytest.mark.parametrize("case", REFINE_CASES, ids=lambda c: f"{c[0]}x{c[1]}_b{c[4]}{'_w' if c[7] else ''}")
def test_refine_matches_oracle(X, case):
    m, n, mu, tau, block, iters, sweeps, weighted = case
    A = W.student_t(m, n, 5.0, 0.015, m * 7 + n).astype(np.float32)
    h = W.importance(n, m).astype(np.float32) if weighted else None
    hc = None if h is None else cuda(h)
    dec = X.decompose_traced(cuda(A), mu, tau, block, iters, hc)
    ref_in = O.Result(*host(dec), dec.energy, dec.trace, None)
    out, replaced = X.refine(cuda(A), dec, tau, block, iters, sweeps, hc)
    ref, ref_replaced = N.refine(A.astype(np.float64), ref_in, tau, block, iters, sweeps,
                                 None if h is None else h.astype(np.float64))
    assert len(out.trace) == sweeps and len(replaced) == sweeps
    energies = [dec.energy] + out.trace
    assert all(b >= a - 1e-6 for a, b in zip(energies, energies[1:]))
    assert abs(out.energy - ref.energy) <= 1e-4
    for e_gpu, e_ref in zip(out.trace, ref.trace):
        assert abs(e_gpu - e_ref) <= 1e-4
    B, D, C = host(out)
    assert set(np.unique(B)) <= {-1, 0, 1} and set(np.unique(C)) <= {-1, 0, 1}
    e2 = X.energy(cuda(A), out.B, out.D, out.C, hc)
    assert abs(e2 - out.energy) <= 1e-5
    assert sum(replaced) >= 1 and sum(ref_replaced) >= 1


def test_refine_leaves_input_and_repeats(X):
    A = W.student_t(96, 160, 5.0, 0.015, 4).astype(np.float32)
    dec = X.decompose(cuda(A), 1.5, 1.0, 8, 3)
    B0 = dec.B.clone()
    out1, rep1 = X.refine(cuda(A), dec, 1.0, 8, 3, 2)
    out2, rep2 = X.refine(cuda(A), dec, 1.0, 8, 3, 2)
    torch.cuda.synchronize()
    assert torch.equal(dec.B, B0)
    assert torch.equal(out1.B, out2.B) and torch.equal(out1.C, out2.C) and torch.equal(out1.D, out2.D)
    assert out1.trace == out2.trace and rep1 == rep2
