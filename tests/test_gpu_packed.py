"""Packed inference (§2.6, Eq. 5) through the C ABI against the oracle.

* Packing is bit-exact: decoding the words by the layout include/externd.h states gives the matrix back, padding
  codes are zero, no code has a sign without a nonzero, the row-major mask and sign streams equal the oracle's
  sparse packing, and the nonzero count matches.
* y = B diag(D) (C x): the vector is split exactly into three bf16 parts (3 x 8 significant bits hold a float32
  above 2^-110), the products are exact, and the tensor core accumulates one k-step of 16 products at a time in
  fp32, so each of the ceil(c/16) steps of a product over c columns, the slice sums and the final additions
  contribute at most 2^-22 of the magnitude sum:
  |dy_i| <= (ceil(n/16) + ceil(k/16) + 16) 2^-22 (|B| |D| |C| |x|)_i.
"""
import numpy as np
import pytest

from oracle import externd_oracle as O
from oracle import externd_next as N
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


def random_ternary(rows, cols, density, seed):
    rng = np.random.default_rng(seed)
    t = rng.choice(np.array([-1, 1], np.int8), size=(rows, cols))
    return np.where(rng.random((rows, cols)) < density, t, 0).astype(np.int8)


def decode_words(words, rows, cols):
    """The matrix from the packed words, following the documented layout; also the raw codes' sanity."""
    w = words.view(np.uint32)
    RT, G = w.shape[:2]
    T = np.full((RT * 16, G * 128), 9, np.int8)
    lane = np.arange(32)
    g, t = lane >> 2, lane & 3
    bad = 0
    for q in range(4):
        for p in range(8):
            ks, r = 2 * q + p // 4, p & 3
            ri = 16 * np.arange(RT)[:, None, None] + (g + 8 * (r & 1))[None, None, :]
            for half, shift in ((0, 14 - 2 * p), (1, 30 - 2 * p)):
                code = (w[:, :, :, q] >> np.uint32(shift)) & np.uint32(3)
                bad += int(np.count_nonzero(code == 2))
                ci = 128 * np.arange(G)[None, :, None] + (16 * ks + 8 * (r >> 1) + 2 * t + half)[None, None, :]
                T[np.broadcast_to(ri, code.shape), np.broadcast_to(ci, code.shape)] = \
                    np.where(code == 1, 1, np.where(code == 3, -1, 0))
    assert not (T == 9).any()                      # every position written exactly by the layout
    assert bad == 0
    return T


@pytest.mark.parametrize("rows,cols", [(1, 1), (3, 31), (5, 32), (17, 129), (64, 1000), (130, 4099), (2, 51200)])
@pytest.mark.parametrize("density", [0.0, 0.3, 1.0])
def test_pack_is_bit_exact(X, rows, cols, density):
    T = random_ternary(rows, cols, density, rows * 7919 + cols)
    pk = X.pack_ternary(cuda(T))
    assert pk.nnz == int(np.count_nonzero(T))
    full = decode_words(pk.words.cpu().numpy(), rows, cols)
    np.testing.assert_array_equal(full[:rows, :cols], T)
    assert not full[rows:].any() and not full[:, cols:].any()
    om, os_ = N.pack_mask_sign(T)
    np.testing.assert_array_equal((full[:rows, :cols] != 0).reshape(-1), om)
    nz = full[:rows, :cols].reshape(-1)
    np.testing.assert_array_equal((nz[nz != 0] < 0).astype(np.uint8), os_)


def apply_bound(B, D, C, x):
    k, n = C.shape
    mag = np.abs(B).astype(np.float64) @ (np.abs(np.asarray(D, np.float64)) * (np.abs(C).astype(np.float64) @
                                                                               np.abs(x).astype(np.float64)))
    return (-(-n // 16) + -(-k // 16) + 16) * 2.0 ** -22 * mag


@pytest.mark.parametrize("m,k,n,density", [
    (1, 1, 1, 1.0),
    (33, 47, 70, 0.5),
    (300, 517, 1000, 0.4),
    (4096, 3072, 4096, 0.45),
    (64, 200, 51200, 0.5),
    (512, 51200, 96, 0.5),
])
def test_ternary_apply_matches_oracle(X, m, k, n, density):
    B = random_ternary(m, k, density, m + 3)
    C = random_ternary(k, n, density, n + 5)
    rng = np.random.default_rng(k)
    D = (0.01 + rng.random(k)).astype(np.float32)
    x = W.student_t(1, n, 5.0, 1.0, n + k)[0].astype(np.float32)
    y = X.ternary_apply(X.pack_ternary(cuda(B)), cuda(D), X.pack_ternary(cuda(C)), cuda(x)).cpu().numpy()
    ref = N.ternary_apply(B, D.astype(np.float64), C, x.astype(np.float64))
    err = np.abs(y.astype(np.float64) - ref)
    assert np.all(err <= apply_bound(B, D, C, x) + 1e-30)


def test_apply_of_a_gpu_decomposition_and_eq5(X):
    """The packed product of factors the GPU path produced, and Eq. 5's storage from the packer's counts."""
    m, n, mu = 256, 384, 1.5
    A = W.student_t(m, n, 5.0, 0.02, 77)
    dec = X.decompose(cuda(A.astype(np.float32)), mu, 0.7, 8, 3)
    torch.cuda.synchronize()
    B, D, C = dec.B.cpu().numpy(), dec.D.cpu().numpy(), dec.C.cpu().numpy()
    pb, pc = X.pack_ternary(dec.B), X.pack_ternary(dec.C)
    x = W.gaussian(1, n, 1.0, 3)[0].astype(np.float32)
    y = X.ternary_apply(pb, dec.D, pc, cuda(x)).cpu().numpy()
    ref = N.ternary_apply(B, D.astype(np.float64), C, x.astype(np.float64))
    assert np.all(np.abs(y - ref) <= apply_bound(B, D, C, x) + 1e-30)
    k = O.inner_rank(m, n, mu)
    assert k == mu * min(m, n)                       # Eq. 5 holds exactly when mu min(m, n) is an integer
    sparsity = 1.0 - (pb.nnz + pc.nnz) / (m * k + k * n)
    bits = m * k + pb.nnz + k * n + pc.nnz           # one mask bit per entry, one sign bit per nonzero
    assert bits / (m * n) == pytest.approx(N.bpw_eff(mu, m, n, sparsity), rel=1e-12)


def test_apply_with_zero_and_tiny_vectors(X):
    """An all-zero slice and a vector far below 1 (the bf16 parts keep the float32 exponent range)."""
    m, k, n = 200, 300, 700
    B, C = random_ternary(m, k, 0.5, 1), random_ternary(k, n, 0.5, 2)
    D = np.linspace(0.5, 1.5, k).astype(np.float32)
    pb, pc = X.pack_ternary(cuda(B)), X.pack_ternary(cuda(C))
    for x in (np.zeros(n, np.float32), (1e-30 * W.gaussian(1, n, 1.0, 4)[0]).astype(np.float32)):
        x[:128] = 0.0
        y = X.ternary_apply(pb, cuda(D), pc, cuda(x)).cpu().numpy()
        ref = N.ternary_apply(B, D.astype(np.float64), C, x.astype(np.float64))
        assert np.all(np.abs(y - ref) <= apply_bound(B, D, C, x) + 1e-45)
