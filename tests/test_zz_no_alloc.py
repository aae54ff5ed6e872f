"""externd_energy_noalloc, the entry point for callers that cannot allocate device memory.

A process whose framework owns all device memory through its own caching allocator, a latency-critical path that
cannot take the device synchronisation of cudaMalloc/cudaFree, or a plugin handed only buffers cannot use
externd_energy, which allocates scratch for its partial sums. externd_energy_noalloc keeps that scratch in a
fixed static device array instead. This test calls it through the C ABI twice in a row and checks both results
against externd_energy on the same factors, within the energy tolerance of the other GPU tests (1e-6). The file
is named to be collected last.
"""
import ctypes

import numpy as np
import pytest

from paper_2607_13511_gb300 import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2607_13511_gb300 as X
    from paper_2607_13511_gb300 import build
    build.build()
    return X.load()


def call(fn, A, B, D, C, h):
    e = ctypes.c_double()
    m, n = A.shape
    status = fn(A.data_ptr(), m, n, B.data_ptr(), D.data_ptr(), C.data_ptr(), D.numel(),
                None if h is None else h.data_ptr(), ctypes.byref(e))
    torch.cuda.synchronize()
    return status, e.value


@pytest.mark.parametrize("m,n,weighted", [(300, 517, False), (256, 384, True), (33, 47, False)])
def test_noalloc_energy_matches_the_allocating_entry_point(lib, m, n, weighted):
    import paper_2607_13511_gb300 as X
    A = torch.from_numpy(W.student_t(m, n, 5.0, 0.015, m + n)).cuda()
    h = torch.from_numpy(W.importance(n, m)).cuda() if weighted else None
    res = X.decompose(A, 1.5, 0.7, 8, 3, h)
    status, ref = call(lib.externd_energy, A, res.B, res.D, res.C, h)
    assert status == 0
    for _ in range(2):   # two calls in a row share (and overwrite) the static scratch
        status, e = call(lib.externd_energy_noalloc, A, res.B, res.D, res.C, h)
        assert status == 0
        assert abs(e - ref) <= 1e-6


def test_noalloc_rejects_problems_larger_than_its_scratch(lib):
    # ceil(16384/64) * ceil(16384/128) + 3 > 32768 doubles; rejected before any device work.
    tiny = torch.zeros(1, device="cuda")
    e = ctypes.c_double()
    p = tiny.data_ptr()
    assert lib.externd_energy_noalloc(p, 16384, 16384, p, p, p, 1, None, ctypes.byref(e)) == -1
    assert lib.externd_energy_noalloc(None, 10, 10, p, p, p, 1, None, ctypes.byref(e)) == -1
    # sizes whose tile count would wrap a 32-bit product, and k at 2^31: rejected, nothing launched
    assert lib.externd_energy_noalloc(p, 65535 * 64, 4_300_000, p, p, p, 1, None, ctypes.byref(e)) == -1
    assert lib.externd_energy_noalloc(p, 64, 1 << 30, p, p, p, 1, None, ctypes.byref(e)) == -1
    assert lib.externd_energy_noalloc(p, 10, 10, p, p, p, 1 << 31, None, ctypes.byref(e)) == -1
