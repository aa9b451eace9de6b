"""Combined row and column sub-sampling (Sec. 4.1, the remark after eq.
lsqA_sto): nmd_block_update_combined against the oracle's combined step,
each from the GPU's current state (teacher forcing), on row and column block
pairs including the ragged last blocks, both sides, every precision.  The
panel of S[I, J] is a row range of the stochastic panel of J (or I): short
rows, whole long rows and the slices of split rows are all cut to it (the
dense case has rows of up to ~240 entries per block)."""
import numpy as np
import pytest

import oracle as O
from paper_2608_21607_gb300 import nmd as N
from paper_2608_21607_gb300 import workloads as WL

from gpu_common import PREC_NAMES, TOL, make_pair, rel, require_gpu, sync_oracle_to
from test_gpu_support import _dense_rows

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def gpu():
    return require_gpu()


CASES = [
    # name, make S, r, block_rows, block_cols
    ("connectome4000_r64", lambda: WL.connectome(4000, seed=3), 64, 1024, 1024),
    ("planted1500x1300_r32", lambda: WL.planted(1500, 1300, 32, tau=None, density=0.05, noise=0.01, seed=2)[0],
     32, 500, 480),
    ("dense900x800_r32", lambda: _dense_rows(900, 800, 0.5, 12), 32, 400, 350),
    ("connectome6000_r256", lambda: WL.connectome(6000, seed=5), 256, 2560, 2560),
]


@pytest.mark.parametrize("prec", [N.NMD_BF16, N.NMD_FP32, N.NMD_SIMT], ids=lambda p: PREC_NAMES[p])
@pytest.mark.parametrize("name,make,r,br,bc", CASES, ids=[c[0] for c in CASES])
def test_combined_step_parity(name, make, r, br, bc, prec):
    S = make()
    W, H = WL.init_factors(S.m, S.n, r, 4)
    sol, orc = make_pair(S, r, W, H, block_rows=br, block_cols=bc, precision=prec, eta=0.7, gamma=0.5)
    Kr, Kc = O.num_blocks(S.m, br), O.num_blocks(S.n, bc)
    pairs = [(N.NMD_ROW, Kr - 1, 0), (N.NMD_COL, 0, Kc - 1), (N.NMD_ROW, 0, Kc - 1), (N.NMD_COL, Kr - 1, 0),
             (N.NMD_ROW, Kr // 2, Kc // 2)]
    for side, I, J in pairs:
        sync_oracle_to(sol, orc)
        sol.block_update_combined(side, I, J)
        orc.block_update_combined(side, I, J)
        Wg, Hg, EW, EH, _ = sol.get_state()
        if side == N.NMD_ROW:
            i0, i1 = O.block_range(I, br, S.m)
            got, want = Wg[i0:i1], orc.A[i0:i1]
            gotE, wantE = EW[i0:i1], orc.EA[i0:i1]
            # the other rows of W and all of H are untouched
            assert np.array_equal(np.delete(Wg, np.s_[i0:i1], axis=0), np.delete(orc.A, np.s_[i0:i1], axis=0).astype(np.float32))
        else:
            j0, j1 = O.block_range(J, bc, S.n)
            got, want = Hg.T[j0:j1], orc.B[j0:j1]
            gotE, wantE = EH.T[j0:j1], orc.EB[j0:j1]
        assert rel(got, want) <= TOL[prec], (name, side, I, J, rel(got, want))
        assert rel(gotE, wantE) <= 10 * TOL[prec], (name, side, I, J)
