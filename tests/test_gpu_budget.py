"""The greedy-prefix property behind the rank budgets, on the GPU path: a decomposition at a smaller rank (a block
boundary) is the prefix of one at a larger rank, so one run's trace gives the energy of every smaller run."""
import numpy as np
import pytest

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


@pytest.mark.parametrize("m,n,block", [(256, 384, 8), (200, 300, 1), (512, 640, 64)])
def test_gpu_prefix_and_rank_for_energy(X, m, n, block):
    A = torch.from_numpy(W.student_t(m, n, 5.0, 0.015, m + n).astype(np.float32)).cuda()
    mu = 1.5
    big = X.decompose_traced(A, mu, 1.0, block, 3)
    ranks = X.block_boundaries(m, n, mu, block)
    assert len(big.trace) == len(ranks)
    k1 = ranks[len(ranks) // 2 - 1]
    small = X.decompose_traced(A, k1 / min(m, n), 1.0, block, 3)
    torch.cuda.synchronize()
    assert small.B.shape[1] == k1
    assert torch.equal(small.B, big.B[:, :k1]) and torch.equal(small.C, big.C[:k1])
    assert torch.equal(small.D, big.D[:k1])
    assert small.trace == big.trace[:len(small.trace)]
    target = big.trace[len(ranks) // 2 - 1]
    assert X.rank_for_energy(big.trace, m, n, mu, block, target) == N.rank_for_energy(big.trace, ranks, target)
    assert X.rank_for_energy(big.trace, m, n, mu, block, target) <= k1
