"""nmd_gram_noalloc: the Gram matrix of a device matrix without any device
allocation (its scratch is a static device array), for callers that cannot
call cudaMalloc.  Checked against the Gram matrix the solver computes for a
stochastic column step (nmd_block_terms), on two calls in a row.  This file
is collected last on purpose."""
import numpy as np
import pytest

import oracle as O
from paper_2608_21607_gb300 import nmd as N
from paper_2608_21607_gb300 import workloads as WL

from gpu_common import rel, require_gpu

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("r", [3, 64, 100])
def test_gram_noalloc_matches_solver_gram(r):
    torch = require_gpu()
    n, b = 2000, 700
    S = WL.connectome(n, seed=r)
    W, H = WL.init_factors(n, n, r, r)
    sol = N.Solver(S, r, block_rows=b, block_cols=b, precision=N.NMD_BF16)
    sol.set_factors(W, H)
    K = O.num_blocks(n, b)
    stream = torch.cuda.current_stream()
    for block in (K - 1, 0):
        _, G_ref = sol.block_terms(N.NMD_COL, block, N.NMD_STOCH)     # G = B_J^T B_J
        j0, j1 = O.block_range(block, b, n)
        Q = torch.from_numpy(np.ascontiguousarray(H.T[j0:j1])).cuda()
        for call in range(2):
            G = torch.full((r, r), float("nan"), device="cuda")
            st = N.nmd_gram_noalloc(Q, j1 - j0, r, r, G, stream.cuda_stream)
            assert st == N.NMD_OK
            torch.cuda.synchronize()
            Gh = G.cpu().numpy()
            assert np.all(np.isfinite(Gh))
            assert rel(Gh, G_ref) <= 2e-6, (block, call, rel(Gh, G_ref))


def test_gram_noalloc_strided_and_limits():
    torch = require_gpu()
    rng = np.random.default_rng(5)
    Qf = rng.standard_normal((5000, 40)).astype(np.float32)
    Q = torch.from_numpy(Qf).cuda()
    G = torch.zeros((24, 24), device="cuda")
    s = torch.cuda.current_stream().cuda_stream
    # the first 24 columns of a 40-wide matrix: row stride 40
    assert N.nmd_gram_noalloc(Q, 5000, 24, 40, G, s) == N.NMD_OK
    torch.cuda.synchronize()
    want = Qf[:, :24].astype(np.float64).T @ Qf[:, :24]
    assert rel(G.cpu().numpy(), want) <= 2e-6
    # beyond the static scratch: rejected, nothing written
    big = torch.zeros((200, 200), device="cuda")
    Qb = torch.zeros((10, 200), device="cuda")
    assert N.nmd_gram_noalloc(Qb, 10, 200, 200, big, s) == N.NMD_ERR_WORKSPACE
    assert N.nmd_gram_noalloc(Q, 5000, 24, 10, G, s) == N.NMD_ERR_INVALID      # ld < r
