"""Per-kernel parity: each step of the CUDA path, called through the C ABI, against the CPU oracle on the same
seeded inputs.

Bars (derived from the arithmetic of each step):
* Eq. 2 ternarization: bit-exact (both sides decide |x| > tau * mean|x| for the same float32 x).
* Residual products U^T R and R H V: ||dP||_F / ||P||_F <= 1e-5 and |dP_ij| <= 1e-5 * (|U|^T |R|)_ij elementwise.
* Decorrelated targets (Eq. 3) and scales (Eq. 4): relative Frobenius error <= 2e-5 + 4 kappa 2^-24, kappa the
  condition number of the ridge system (a float32 solve loses about kappa units of roundoff; the paper's cap
  b <= min(m, n)/8 keeps kappa small, the (129, 1031, 128) case deliberately breaks it).
* Deflation: |dR_ij| <= 2^-22 * (|R_ij| + sum_a |u_ia d_a v_aj|) + float32 rounding of the result.
"""
import numpy as np
import pytest

from oracle import externd_oracle as O
from paper_2607_13511_gb300 import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

SHAPES = [  # (m, n, w): several 64x128 tiles with ragged tails, a GEMV, a tiny case, the widest block
    (300, 517, 70),
    (256, 512, 64),
    (33, 47, 5),
    (1000, 777, 1),
    (129, 1031, 128),
    (640, 300, 256),
    (300, 9728, 32),    # V-step grid of 76 tiles x 2 splits = every SM: the stream plan over SMs - 1 CTAs
    (9728, 300, 32),    # the same for the U-step
]


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


def solve_tol(G):
    Gr = G + O.ridge(G) * np.eye(G.shape[0])
    return 2e-5 + 4 * np.linalg.cond(Gr) * 2.0 ** -24


def rel_fro(a, b):
    return float(np.linalg.norm(np.asarray(a, np.float64) - b) / max(np.linalg.norm(b), 1e-300))


# ------------------------------------------------------------------------------------------------ Eq. 2
@pytest.mark.parametrize("rows,cols", [(1, 1), (3, 7), (64, 1000), (130, 4099), (1000, 129)])
@pytest.mark.parametrize("tau", [0.0, 0.7, 1.0, 2.0, 50.0])
def test_ternarize_rows_and_columns_bit_exact(X, rows, cols, tau):
    x = W.student_t(rows, cols, 5.0, 1.0, rows * 1000 + cols)
    t_rows = X.ternarize(cuda(x), tau, axis=1).cpu().numpy()
    t_cols = X.ternarize(cuda(x), tau, axis=0).cpu().numpy()
    assert (t_rows == O.ternarize_rows(x, tau)).all()
    assert (t_cols == O.ternarize_cols(x, tau)).all()


def test_ternarize_fallback_ties_and_zeros(X):
    x = np.zeros((4, 9), np.float32)
    x[1] = 1.0                                     # all equal: at tau = 1 nothing passes -> first index
    x[2, 5] = -3.0                                 # single nonzero, negative
    x[3] = np.array([2, -2, 1, 0, 0, 2, -2, 0, 0], np.float32)
    for tau in (0.7, 1.0, 3.0):
        assert (X.ternarize(cuda(x), tau).cpu().numpy() == O.ternarize_rows(x, tau)).all()


# ------------------------------------------------------------------------------------------------ products
def _product_bars(P_gpu, P_ref, bound):
    assert rel_fro(P_gpu, P_ref) <= 1e-5
    assert np.all(np.abs(P_gpu - P_ref) <= 1e-5 * bound + 1e-30)


@pytest.mark.parametrize("m,n,w", SHAPES)
def test_vstep_product(X, m, n, w):
    R = W.gaussian(m, n, 0.02, m + n + w)
    U = W.ternary(m, w, 0.6, w)
    P = X.vstep_product(cuda(R), cuda(U)).cpu().numpy()
    _product_bars(P, O.vstep_product(R, U), np.abs(U).T.astype(np.float64) @ np.abs(R.astype(np.float64)))


@pytest.mark.parametrize("m,n,w", SHAPES)
@pytest.mark.parametrize("weighted", [False, True])
def test_ustep_product(X, m, n, w, weighted):
    R = W.student_t(m, n, 5.0, 0.015, m * n + w)
    Cb = W.ternary(w, n, 0.55, w + 1)
    h = W.importance(n, w + 2) if weighted else None
    P = X.ustep_product(cuda(R), cuda(Cb), None if h is None else cuda(h)).cpu().numpy()
    hh = np.ones(n) if h is None else h.astype(np.float64)
    bound = np.abs(R.astype(np.float64)) @ (hh[:, None] * np.abs(Cb.T))
    _product_bars(P, O.ustep_product(R, Cb, h), bound)


# ------------------------------------------------------------------------------------------------ Eq. 3, Eq. 4
@pytest.mark.parametrize("m,n,w", SHAPES)
def test_vstep_target(X, m, n, w):
    R = W.gaussian(m, n, 0.02, 7 * m + n)
    U = W.ternary(m, w, 0.6, 3 * w)
    Xg = X.vstep_target(cuda(R), cuda(U)).cpu().numpy()
    ref = O.vstep_product(R, U) if w == 1 else O.vstep_target(R, U)
    assert rel_fro(Xg, ref) <= solve_tol(O.gram_u(U))


@pytest.mark.parametrize("m,n,w", SHAPES)
@pytest.mark.parametrize("weighted", [False, True])
def test_ustep_target(X, m, n, w, weighted):
    R = W.gaussian(m, n, 0.02, 5 * m + n)
    Cb = W.ternary(w, n, 0.6, 5 * w)
    h = W.importance(n, 9) if weighted else None
    Y = X.ustep_target(cuda(R), cuda(Cb), None if h is None else cuda(h)).cpu().numpy()
    ref = O.ustep_product(R, Cb, h) if w == 1 else O.ustep_target(R, Cb, h)
    assert rel_fro(Y, ref) <= solve_tol(O.gram_v(Cb, h))


@pytest.mark.parametrize("m,n,w", SHAPES)
@pytest.mark.parametrize("weighted", [False, True])
def test_block_scales(X, m, n, w, weighted):
    R = W.gaussian(m, n, 0.02, 11 * m + n)
    U = W.ternary(m, w, 0.6, 11 * w)
    Cb = W.ternary(w, n, 0.6, 13 * w)
    h = W.importance(n, 10) if weighted else None
    d = X.block_scales(cuda(R), cuda(U), cuda(Cb), None if h is None else cuda(h)).cpu().numpy()
    ref = O.block_scales(U, Cb, O.ustep_product(R, Cb, h), h)
    assert rel_fro(d, ref) <= solve_tol(O.gram_u(U) * O.gram_v(Cb, h))


@pytest.mark.parametrize("m,n,w", SHAPES)
@pytest.mark.parametrize("weighted", [False, True])
def test_deflate(X, m, n, w, weighted):
    R = W.gaussian(m, n, 0.02, 17 * m + n)
    U = W.ternary(m, w, 0.6, 17 * w)
    Cb = W.ternary(w, n, 0.6, 19 * w)
    d = (np.random.default_rng(w).standard_normal(w) * 0.01).astype(np.float32)
    h = W.importance(n, 12) if weighted else None
    Rg = cuda(R)
    norm2 = X.deflate(Rg, cuda(U), cuda(d), cuda(Cb), None if h is None else cuda(h))
    ref = O.deflate(R, U, d, Cb)
    bound = np.abs(R) + (np.abs(U) * np.abs(d.astype(np.float64))) @ np.abs(Cb)
    # From w = 16 on the deflation runs on the tensor cores with d split into two fp16 parts (each term exact to
    # 2^-22 relative) and fp32 accumulation over 2 ceil(w / 16) MMA steps plus the final subtraction (2^-24
    # each); narrower blocks use float32 FMAs (w + 1 roundings of 2^-24).
    steps = 2 * -(-w // 16) + 1 if w >= 16 else w + 1
    tol = (2.0 ** -22 if w >= 16 else 0.0) + steps * 2.0 ** -24
    assert np.all(np.abs(Rg.cpu().numpy() - ref) <= tol * bound + 1e-30)
    assert abs(norm2 - O.weighted_norm2(ref, h)) <= 1e-5 * O.weighted_norm2(ref, h)


def test_energy_of_given_factors(X):
    A = W.gaussian(200, 300, 0.02, 21)
    res = O.block_als(A, 1.0, 0.7, 16, 2)
    h = W.importance(300, 21)
    for weights in (None, h):
        e = X.energy(cuda(A), cuda(res.B), cuda(res.D.astype(np.float32)), cuda(res.C),
                     None if weights is None else cuda(weights))
        ref = O.energy(A, res.B, res.D.astype(np.float32), res.C, weights)
        assert abs(e - ref) <= 1e-6


# ------------------------------------------------------------------------------------------------ full sizes
@pytest.mark.parametrize("wl", [W.OUTLIER_2048, W.MLP_UP_2560x9728, W.ATTN_4096_WEIGHTED], ids=lambda w: w.name)
def test_full_size_products_sampled(X, wl):
    """The products at the workloads' full sizes and block widths, checked on sampled outputs."""
    A = wl.matrix()
    h = wl.weights()
    b = O.block_width(wl.m, wl.n, wl.block)
    U = W.ternary(wl.m, b, 0.58, 1)
    Cb = W.ternary(b, wl.n, 0.58, 2)
    PV = X.vstep_product(cuda(A), cuda(U)).cpu().numpy()
    PU = X.ustep_product(cuda(A), cuda(Cb), None if h is None else cuda(h)).cpu().numpy()
    rng = np.random.default_rng(3)
    A64 = A.astype(np.float64)
    hh = np.ones(wl.n) if h is None else h.astype(np.float64)
    for _ in range(300):
        a, c, r = rng.integers(b), rng.integers(wl.n), rng.integers(wl.m)
        ref_v = float(U[:, a].astype(np.float64) @ A64[:, c])
        bnd_v = float(np.abs(U[:, a]) @ np.abs(A64[:, c]))
        assert abs(PV[a, c] - ref_v) <= 1e-5 * bnd_v
        ref_u = float(A64[r] @ (hh * Cb[a]))
        bnd_u = float(np.abs(A64[r]) @ (hh * np.abs(Cb[a])))
        assert abs(PU[r, a] - ref_u) <= 1e-5 * bnd_u
