"""Delta-form tile skipping (Sec. 4.3): a Q chunk whose rectified tile
max(0, L) is zero on all 128 rows of an M tile contributes nothing to
R = Delta Q, so the tensor-core kernel skips its second product.  The
results must equal the oracle's, and the skip count must show that chunks
were skipped exactly when the rectified tile vanished.

Inputs follow the paper's sign-structured start (Sec. 4.3: A > 0, B < 0,
so that L = A B^T < 0 and the rectified matrix is empty), optionally with
one chunk of Q-side rows of flipped sign so that only some chunks vanish."""
import numpy as np
import pytest

import oracle as O
from gpu_common import TOL, make_pair, rel, require_gpu
from paper_2608_21607_gb300 import nmd as N
from paper_2608_21607_gb300 import workloads as WL

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def gpu():
    return require_gpu()


def _signed_factors(n, r, seed, flip=None):
    rng = np.random.default_rng(seed)
    W = np.abs(0.1 * rng.standard_normal((n, r))).astype(np.float32)    # A > 0
    H = -np.abs(0.1 * rng.standard_normal((r, n))).astype(np.float32)   # B < 0
    if flip is not None:
        H[:, flip] *= -1.0
    return W, H


def _step_terms(sol, orc, side, block, kind):
    Rg, Gg = sol.block_terms(side, block, kind)
    Ro, Go = orc.block_terms(side, block, kind)
    M, _, (m0, m1), _, _, _ = orc._roles(side, block, kind)
    return Rg, Ro - M[m0:m1] @ Go        # Delta Q = Z Q - L Q


CASES = [(3, 1500, 192), (32, 1500, 320), (64, 2000, 640), (100, 1500, 1000)]


@pytest.mark.parametrize("prec", [N.NMD_BF16, N.NMD_FP32], ids=["bf16", "fp32"])
@pytest.mark.parametrize("r,n,b", CASES, ids=[str(c[0]) for c in CASES])
def test_skipped_chunks_keep_the_result(r, n, b, prec):
    S = WL.connectome(n, seed=r)
    block = 1
    q0 = block * b
    # all-negative L: every chunk but the first of each tile is skipped
    W, H = _signed_factors(n, r, seed=r)
    sol, orc = make_pair(S, r, W, H, block_rows=b, block_cols=b, precision=prec, epilogue=N.NMD_EPI_DELTA,
                         eta=1.0, gamma=0.0, skip_zero_chunks=True)
    sol.skip_count(reset=True)
    Rg, Ro = _step_terms(sol, orc, N.NMD_COL, block, N.NMD_STOCH)
    all_neg = sol.skip_count(reset=True)
    assert rel(Rg, Ro) <= TOL[prec], rel(Rg, Ro)
    tiles = -(-n // 128)
    assert all_neg > 0 and all_neg % tiles == 0, all_neg       # the same chunks in every tile

    # Q-side rows 128-191 of the block flipped positive: the chunk holding
    # them (never the first of a tile, for chunks of 64 or 128 rows) must be
    # computed, the others are still skipped
    W2, H2 = _signed_factors(n, r, seed=r, flip=np.arange(q0 + 128, min(q0 + 192, n)))
    sol2, orc2 = make_pair(S, r, W2, H2, block_rows=b, block_cols=b, precision=prec,
                           epilogue=N.NMD_EPI_DELTA, eta=1.0, gamma=0.0, skip_zero_chunks=True)
    sol2.skip_count(reset=True)
    Rg2, Ro2 = _step_terms(sol2, orc2, N.NMD_COL, block, N.NMD_STOCH)
    mixed = sol2.skip_count(reset=True)
    assert rel(Rg2, Ro2) <= TOL[prec], rel(Rg2, Ro2)
    assert 0 <= mixed < all_neg, (mixed, all_neg)

    # the update from the skipped products equals the oracle's
    sol2.block_update(N.NMD_COL, block, N.NMD_STOCH)
    orc2.block_update(N.NMD_COL, block, N.NMD_STOCH)
    Wg, _ = sol2.get_factors()
    assert rel(Wg, orc2.A) <= TOL[prec]


def test_skipping_is_off_by_default():
    S = WL.connectome(1500, seed=6)
    W, H = _signed_factors(1500, 32, seed=6)
    sol, _ = make_pair(S, 32, W, H, block_rows=320, block_cols=320, precision=N.NMD_BF16,
                       epilogue=N.NMD_EPI_DELTA, eta=1.0, gamma=0.0)
    sol.skip_count(reset=True)
    sol.block_update(N.NMD_COL, 1, N.NMD_STOCH)
    assert sol.skip_count() == 0


def test_z_form_never_skips():
    S = WL.connectome(1500, seed=5)
    W, H = _signed_factors(1500, 32, seed=5)
    sol, _ = make_pair(S, 32, W, H, block_rows=320, block_cols=320, precision=N.NMD_BF16,
                       epilogue=N.NMD_EPI_Z, eta=1.0, gamma=0.0, skip_zero_chunks=True)
    sol.skip_count(reset=True)
    sol.block_update(N.NMD_COL, 1, N.NMD_STOCH)
    assert sol.skip_count() == 0
