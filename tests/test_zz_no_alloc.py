"""nmd_gram_noalloc: the Gram matrix of a device matrix without any device
allocation (its scratch is a static device array), for callers that cannot
call cudaMalloc.  Each result is checked against the fp64 product Q^T Q of
the same fp32 rows and against the Gram matrix that the solver's own entry
point computes for the same block (nmd_block_terms), on two calls in a row.
This file is collected last on purpose.

Tolerance: both sides accumulate in fp32.  The no-allocation kernel sums at
most ceil(K / parts) <= 700 products per partial sum before the partials are
added, so its relative error is at most about 700 u = 4e-5 (u = 2^-24) and
typically sqrt(700) u = 1.6e-6; 1e-5 in relative Frobenius norm."""
import numpy as np
import pytest

import oracle as O
from paper_2608_21607_gb300 import nmd as N
from paper_2608_21607_gb300 import workloads as WL

from gpu_common import rel, require_gpu

pytestmark = pytest.mark.gpu

TOL = 1e-5


def _gram_twice(torch, Q, K, r, ld):
    """Two calls in a row into buffers pre-filled with NaN; both results."""
    stream = torch.cuda.current_stream()
    out = []
    for _ in range(2):
        G = torch.full((r, r), float("nan"), device="cuda")
        assert N.nmd_gram_noalloc(Q, K, r, ld, G, stream.cuda_stream) == N.NMD_OK
        torch.cuda.synchronize()
        out.append(G.cpu().numpy())
    return out


@pytest.mark.parametrize("r", [3, 64, 100, 128])
def test_gram_noalloc_matches_fp64_and_solver_gram(r):
    torch = require_gpu()
    n, b = 2000, 700
    S = WL.connectome(n, seed=r)
    W, H = WL.init_factors(n, n, r, r)
    sol = N.Solver(S, r, block_rows=b, block_cols=b, precision=N.NMD_BF16)
    sol.set_factors(W, H)
    K = O.num_blocks(n, b)
    for block in (K - 1, 0):                                           # ragged last block first
        _, G_sol = sol.block_terms(N.NMD_COL, block, N.NMD_STOCH)     # G = B_J^T B_J
        j0, j1 = O.block_range(block, b, n)
        Qh = np.ascontiguousarray(H.T[j0:j1])
        want = Qh.astype(np.float64).T @ Qh.astype(np.float64)
        Q = torch.from_numpy(Qh).cuda()
        for call, Gh in enumerate(_gram_twice(torch, Q, j1 - j0, r, r)):
            assert np.all(np.isfinite(Gh))
            assert rel(Gh, want) <= TOL, (block, call, rel(Gh, want))
            assert rel(Gh, G_sol) <= TOL, (block, call, rel(Gh, G_sol))


def test_gram_noalloc_part_count_capped_by_the_static_array():
    """r = 128 with K = 20,001 rows: the static array holds only 32 partial
    128 x 128 matrices, fewer than the 79 parts of 256 rows the kernel would
    otherwise use, so each part sums 626 rows; the last part is ragged
    (20,001 is not a multiple of the 32-row staging tile)."""
    torch = require_gpu()
    rng = np.random.default_rng(11)
    K, r = 20001, 128
    Qh = (rng.standard_normal((K, r)) * rng.uniform(0.5, 2.0, r)).astype(np.float32)
    want = Qh.astype(np.float64).T @ Qh.astype(np.float64)
    Q = torch.from_numpy(Qh).cuda()
    for call, Gh in enumerate(_gram_twice(torch, Q, K, r, r)):
        assert np.all(np.isfinite(Gh))
        assert rel(Gh, want) <= TOL, (call, rel(Gh, want))


def test_gram_noalloc_strided_and_limits():
    torch = require_gpu()
    rng = np.random.default_rng(5)
    Qf = rng.standard_normal((5000, 40)).astype(np.float32)
    Q = torch.from_numpy(Qf).cuda()
    # the first 24 columns of a 40-wide matrix: row stride 40
    want = Qf[:, :24].astype(np.float64).T @ Qf[:, :24]
    for Gh in _gram_twice(torch, Q, 5000, 24, 40):
        assert rel(Gh, want) <= TOL
    s = torch.cuda.current_stream().cuda_stream
    G = torch.zeros((24, 24), device="cuda")
    # beyond the static scratch: rejected, nothing written
    big = torch.zeros((200, 200), device="cuda")
    Qb = torch.zeros((10, 200), device="cuda")
    assert N.nmd_gram_noalloc(Qb, 10, 200, 200, big, s) == N.NMD_ERR_WORKSPACE
    assert N.nmd_gram_noalloc(Q, 5000, 24, 10, G, s) == N.NMD_ERR_INVALID      # ld < r
