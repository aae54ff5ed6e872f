"""Parity of the opt-in tensor-core Gram inverse (EXTERND_TCINV=1) with the oracle, on the GPU.

The switch is read once per process, so the runs take place in a child process. The tensor-core inverse serves
blocks of 65 to 128 components: Eq. 3's (G + eps I)^-1 for both half-steps and the Eq. 4 solve. Its rank-16
updates carry ~22-bit products, so the bar is the end-to-end one of the default path: |E_gpu - E_oracle| <= 1e-4,
and the first block's trits, which no near-tie flips, bit for bit.
"""
import json
import os
import subprocess
import sys

import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = r"""
import json, sys
import numpy as np
import torch
sys.path.insert(0, sys.argv[1])
import paper_2607_13511_gb300 as X
from oracle import externd_oracle as O
from paper_2607_13511_gb300 import workloads as W

out = []
# whole method, (m, n, mu, tau, block, iters, weighted, seed): blocks of 80 and 128 components, the last
# weighted case with a ragged tail block
for m, n, mu, tau, b, it, weighted, seed in [(640, 768, 0.25, 0.7, 80, 2, False, 3),
                                              (1024, 1100, 0.25, 0.7, 128, 2, False, 4),
                                              (1024, 1100, 0.2, 1.0, 128, 2, True, 5)]:
    A = W.gaussian(m, n, 0.02, seed)
    h = W.importance(n, seed) if weighted else None
    ref = O.decompose(A, mu, tau, b, it, h)
    res = X.decompose(torch.from_numpy(A).cuda(), mu, tau, b, it, None if h is None else torch.from_numpy(h).cuda())
    torch.cuda.synchronize()
    out.append(["decompose", m, n, b, weighted, res.energy, ref.energy])
# one block of 80 components on Student-t entries (the first-block case of the default path's tests)
A = W.student_t(640, 768, 5.0, 0.015, 6)
ref = O.block_als(A, 80 / 640, 0.7, 80, 2)
res = X.decompose(torch.from_numpy(A).cuda(), 80 / 640, 0.7, 80, 2)
torch.cuda.synchronize()
out.append(["first_block", bool((res.B.cpu().numpy() == ref.B).all() and (res.C.cpu().numpy() == ref.C).all()),
            bool(np.allclose(res.D.cpu().numpy(), ref.D, rtol=1e-4))])
print(json.dumps(out))
"""


def test_tensor_core_inverse_matches_oracle():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_13511_gb300 import build
    build.build()
    env = dict(os.environ, EXTERND_TCINV="1")
    p = subprocess.run([sys.executable, "-c", CHILD, ROOT], env=env, cwd=ROOT, capture_output=True, text=True,
                       timeout=900)
    assert p.returncode == 0, p.stderr[-4000:]
    rows = json.loads(p.stdout.strip().splitlines()[-1])
    assert len(rows) == 4
    for kind, m, n, b, weighted, e_gpu, e_ref in rows[:3]:
        assert abs(e_gpu - e_ref) <= 1e-4, (m, n, b, weighted, e_gpu, e_ref)
    assert rows[3] == ["first_block", True, True]
