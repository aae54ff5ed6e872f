"""End-to-end parity of externd_decompose with the oracle, and the C-ABI's error conventions, on the GPU.

The ALS trajectory depends on every thresholding decision, and float32 (GPU) and float64 (oracle) arithmetic can
flip a near-tie trit, after which both sides follow different but equally valid trajectories. So end to end the
bar is the final energy, |E_gpu - E_oracle| <= 1e-4 (the paper's method, measured), plus properties that hold for
any valid trajectory: ternary factors, no empty component, monotone energy trace, and the energy recomputed from
the returned factors (externd_energy) equal to the tracked one within 1e-5.
"""
import json
import os

import numpy as np
import pytest

from oracle import externd_oracle as O
from paper_2607_13511_gb300 import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "oracle_energies.json")


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


def check_valid(X, A, res, h, k):
    B, D, C = res.B.cpu().numpy(), res.D.cpu().numpy(), res.C.cpu().numpy()
    assert B.shape[1] == k and C.shape[0] == k and D.shape == (k,)
    assert set(np.unique(B)) <= {-1, 0, 1} and set(np.unique(C)) <= {-1, 0, 1}
    assert (np.abs(B).sum(0) > 0).all() and (np.abs(C).sum(1) > 0).all()
    assert np.all(np.isfinite(D))
    if res.trace is not None:
        assert np.all(np.diff(res.trace) >= -1e-6)
    e2 = X.energy(cuda(A), res.B, res.D, res.C, None if h is None else cuda(h))
    assert abs(e2 - res.energy) <= 1e-5
    return B, D, C


CASES = [  # m, n, mu, tau, block, iters, kind, weighted
    (64, 48, 2.0, 0.7, 1, 4, "gaussian", False),
    (96, 200, 1.5, 0.7, 8, 4, "gaussian", False),
    (200, 150, 1.3, 1.0, 16, 3, "student_t", False),
    (300, 517, 1.2, 0.7, 32, 4, "outliers", False),
    (160, 160, 1.5, 0.7, 20, 4, "gaussian", True),
    (257, 130, 1.7, 0.7, 16, 2, "student_t", True),
    (40, 33, 1.3, 0.7, 4, 2, "gaussian", False),       # tail block of 3
    (7, 5, 3.0, 0.7, 16, 4, "gaussian", False),         # min < 8: cap 0, sequential
    (1, 9, 2.0, 0.7, 1, 4, "gaussian", False),          # a single row
    (520, 64, 2.0, 0.7, 8, 4, "student_t", True),
    (640, 768, 1.2, 0.7, 80, 3, "student_t", False),   # tensor-core targets (w = 80), tail 48
    (576, 700, 1.1, 0.7, 72, 3, "gaussian", True),     # tensor-core targets weighted (w = 72), tail 57
    (1000, 1100, 0.3, 0.7, 128, 2, "gaussian", False), # block capped to 125, tail 50
]


@pytest.mark.parametrize("case", CASES, ids=lambda c: "x".join(map(str, c[:2])) + f"_b{c[4]}_{c[6]}{'_w' if c[7] else ''}")
def test_decompose_matches_oracle(X, case):
    m, n, mu, tau, block, iters, kind, weighted = case
    wl = W.Workload("t", m, n, mu, tau, block, iters, kind, 0.02, m * 31 + n)
    A = wl.matrix()
    h = W.importance(n, m + n) if weighted else None
    ref = O.decompose(A, mu, tau, block, iters, h)
    res = X.decompose(cuda(A), mu, tau, block, iters, None if h is None else cuda(h))
    check_valid(X, A, res, h, ref.D.size)
    assert abs(res.energy - ref.energy) <= 1e-4
    # the traced entry point runs the same method: identical factors, and a monotone trace ending at E
    tr = X.decompose_traced(cuda(A), mu, tau, block, iters, None if h is None else cuda(h))
    check_valid(X, A, tr, h, ref.D.size)
    assert torch.equal(tr.B, res.B) and torch.equal(tr.C, res.C) and torch.equal(tr.D, res.D)
    assert tr.energy == res.energy == tr.trace[-1]
    assert len(tr.trace) == len(ref.trace)


def test_block_width_one_first_components_match_exactly(X):
    # Before any near-tie flip the two sides take identical decisions: the first components agree bit for bit.
    A = W.gaussian(128, 96, 0.02, 5)
    ref = O.decompose(A, 0.1, 0.7, 1, 4)          # k = 10 components
    res = X.decompose(cuda(A), 0.1, 0.7, 1, 4)
    assert (res.B.cpu().numpy() == ref.B).all() and (res.C.cpu().numpy() == ref.C).all()
    assert np.allclose(res.D.cpu().numpy(), ref.D, rtol=1e-5)


@pytest.mark.parametrize("m,n,w", [(128, 160, 16), (256, 320, 24), (400, 416, 48), (640, 768, 80)])
def test_first_block_matches_exactly(X, m, n, w):
    # one block of w components: the FMA inverse beside the product (w = 16), the cluster inverse (w > 16), the
    # tensor-core targets (w > 64)
    A = W.student_t(m, n, 5.0, 0.015, 6)
    ref = O.block_als(A, w / min(m, n), 0.7, w, 2)
    res = X.decompose(cuda(A), w / min(m, n), 0.7, w, 2)
    assert (res.B.cpu().numpy() == ref.B).all() and (res.C.cpu().numpy() == ref.C).all()
    assert np.allclose(res.D.cpu().numpy(), ref.D, rtol=1e-4)


def test_repeatable_and_graph_replay(X):
    A = cuda(W.gaussian(300, 260, 0.02, 7))
    r1 = X.decompose(A, 1.5, 0.7, 16, 4)
    r2 = X.decompose(A, 1.5, 0.7, 16, 4)
    assert r1.energy == r2.energy
    assert torch.equal(r1.B, r2.B) and torch.equal(r1.C, r2.C) and torch.equal(r1.D, r2.D)


def test_repeatable_at_full_size_tensor_core_path(X):
    # 2560 x 9728, blocks of 128: the TMA products (stream-K, A in tensor memory) and the fused targets grid run
    # every half-step. Every decision is taken in a fixed order, so repeated runs agree bit for bit.
    wl = W.WORKLOADS["up2560x9728_t5_mu3_tau1_b128"]
    A = cuda(wl.matrix())
    ref = X.decompose_traced(A, wl.mu, wl.tau, wl.block, wl.iters)
    for _ in range(3):
        r = X.decompose_traced(A, wl.mu, wl.tau, wl.block, wl.iters)
        assert r.trace == ref.trace
        assert torch.equal(r.B, ref.B) and torch.equal(r.C, ref.C) and torch.equal(r.D, ref.D)


def test_host_entry_point_matches_device(X):
    A = W.gaussian(200, 180, 0.02, 8)
    h = W.importance(180, 8)
    dev = X.decompose(cuda(A), 1.5, 0.7, 16, 4, cuda(h))
    host = X.decompose_host(torch.from_numpy(A), 1.5, 0.7, 16, 4, torch.from_numpy(h))
    assert host.energy == dev.energy
    assert torch.equal(host.B, dev.B.cpu()) and torch.equal(host.C, dev.C.cpu())


def test_zero_matrix_does_not_fail(X):
    A = torch.zeros((64, 64), dtype=torch.float32, device="cuda")
    res = X.decompose(A, 0.5, 0.7, 8, 2)
    assert torch.all(res.D == 0)


@pytest.mark.parametrize("name", ["seq256_gauss_mu2_b1", "outlier2048_mu3_b64", "up2560x9728_t5_mu3_tau1_b128",
                                  "attn4096_weighted_mu2.5_b128"])
def test_full_workloads_match_oracle_energy(X, name):
    golden = json.load(open(GOLDEN))
    if name not in golden:
        pytest.skip(f"{name} not in golden table")
    wl = W.WORKLOADS[name]
    A = wl.matrix()
    h = wl.weights()
    res = X.decompose(cuda(A), wl.mu, wl.tau, wl.block, wl.iters, None if h is None else cuda(h))
    check_valid(X, A, res, h, golden[name]["k"])
    assert abs(res.energy - golden[name]["energy"]) <= 1e-4


@pytest.mark.parametrize("layer", [0, 17, 35])
def test_decoder_layers_match_oracle_energy(X, layer):
    """Every projection of decoder layers 0, 17 and 35 of the 36-layer conversion, at full size."""
    golden = json.load(open(GOLDEN))
    wls = [wl for wl in W.decoder_conversion() if wl.name.startswith(f"L{layer}.")]
    if not any(wl.name in golden for wl in wls):
        pytest.skip(f"decoder layer {layer} not in golden table")
    for wl in wls:
        if wl.name not in golden:
            continue
        A = wl.matrix()
        res = X.decompose(cuda(A), wl.mu, wl.tau, wl.block, wl.iters)
        assert res.D.numel() == golden[wl.name]["k"], wl.name
        assert abs(res.energy - golden[wl.name]["energy"]) <= 1e-4, wl.name


# ------------------------------------------------------------------------------------------------ error conventions
def test_error_conventions(X):
    import ctypes
    lib = X.load()
    A = cuda(W.gaussian(32, 32, 0.02, 1))
    B = torch.empty((32, 32), dtype=torch.int8, device="cuda")
    D = torch.empty((32,), dtype=torch.float32, device="cuda")
    C = torch.empty((32, 32), dtype=torch.int8, device="cuda")
    e = ctypes.c_double()

    def call(Ap, m, n, mu, tau, block, iters, Bp=B.data_ptr(), Dp=D.data_ptr(), Cp=C.data_ptr()):
        return lib.externd_decompose(Ap, m, n, mu, tau, block, iters, None, Bp, Dp, Cp, ctypes.byref(e))

    assert call(A.data_ptr(), 32, 32, 1.0, 0.7, 4, 2) == 0
    assert call(A.data_ptr(), 0, 32, 1.0, 0.7, 4, 2) == -1          # bad size
    assert call(A.data_ptr(), 32, 32, -1.0, 0.7, 4, 2) == -1        # mu <= 0
    assert call(A.data_ptr(), 32, 32, 1.0, -0.1, 4, 2) == -1        # tau < 0
    assert call(A.data_ptr(), 32, 32, 1.0, 0.7, 0, 2) == -1         # block < 1
    assert call(A.data_ptr(), 32, 32, 1.0, 0.7, 4, 0) == -1         # iters < 1
    assert call(None, 32, 32, 1.0, 0.7, 4, 2) == -1                 # NULL
    host = np.zeros((32, 32), np.float32)
    assert call(host.ctypes.data, 32, 32, 1.0, 0.7, 4, 2) == -2     # host pointer where device memory is needed
    with pytest.raises(X.ExterndError):
        X.decompose(A.cpu(), 1.0, 0.7, 4, 2)
