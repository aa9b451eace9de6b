"""The support term of a block step (nmd_support_term) against a CPU
restatement of its definition (eqs. updateZ/updateD, Sec. 3.2): for every
M-side row with support in the block's panel,
    Rs_i = sum over the panel's entries (i, k) of (S_ik - min(0, L_ik)) q_k,
L_ik = m_i . q_k, on the step's own operands (the bf16 pieces in the bf16
mode, the fp32 masters otherwise), and Rs_i = 0 on the other rows.  Covers
short rows (one warp per row), whole long rows (lanes over the entries) and
rows split into 128-entry slices with their fixed-order reduction, the
shared-memory kernel (whole Q-side block staged, bf16 at r_pad 16 and 32),
every padded rank, ragged blocks, all four step kinds.  Tolerance 1e-5 relative
(fp32 accumulation against fp64)."""
import numpy as np
import pytest

import oracle as O
from paper_2608_21607_gb300 import nmd as N
from paper_2608_21607_gb300 import workloads as WL

from gpu_common import rel, require_gpu
from test_gpu_tc import pieces

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def gpu():
    return require_gpu()


def _dense_rows(m, n, density, seed):
    """A sparse matrix whose rows hold up to several hundred entries of one
    block (long rows and split rows of the support kernels)."""
    rng = np.random.default_rng(seed)
    D = np.where(rng.random((m, n)) < density, np.ceil(np.exp(1 + rng.standard_normal((m, n)))), 0.0)
    return WL.csr_from_dense(D)


CASES = [
    # name, S, r, block
    ("connectome2000_r64", lambda: WL.connectome(2000, seed=7), 64, 512),
    ("connectome1500_r3", lambda: WL.connectome(1500, seed=8), 3, 400),
    ("dense600x700_r32", lambda: _dense_rows(600, 700, 0.6, 9), 32, 400),   # rows of ~240 entries per panel
    ("dense500_r100", lambda: _dense_rows(500, 500, 0.35, 10), 100, 300),
    ("dense700_r256", lambda: _dense_rows(700, 700, 0.3, 11), 256, 600),
    # whole Q-side blocks in shared memory (bf16, r_pad 32 and 16) at sizes
    # near the limit: 2048 rows of 64 B, 4800 rows of 32 B
    ("dense3000x2400_r32", lambda: _dense_rows(3000, 2400, 0.05, 12), 32, 2048),
    ("dense2000x5000_r12", lambda: _dense_rows(2000, 5000, 0.02, 13), 12, 4800),
]


@pytest.mark.parametrize("prec", [N.NMD_BF16, N.NMD_FP32], ids=["bf16", "fp32"])
@pytest.mark.parametrize("name,make,r,b", CASES, ids=[c[0] for c in CASES])
def test_support_term(name, make, r, b, prec):
    S = make()
    W, H = WL.init_factors(S.m, S.n, r, 3)
    sol = N.Solver(S, r, block_rows=b, block_cols=b, precision=prec)
    sol.set_factors(W, H)
    st = O.State(S, W, H, O.Options(block_rows=b, block_cols=b))
    Kr, Kc = O.num_blocks(S.m, b), O.num_blocks(S.n, b)
    for side, kind, block in [(N.NMD_COL, N.NMD_STOCH, Kc - 1), (N.NMD_ROW, N.NMD_STOCH, 0),
                              (N.NMD_ROW, N.NMD_EXACT, Kr - 1), (N.NMD_COL, N.NMD_EXACT, 0)]:
        M, _, (m0, m1), Q, src, (c0, c1) = st._roles(side, block, kind)
        Mf, Qf = M[m0:m1].astype(np.float32), Q.astype(np.float32)
        if prec == N.NMD_BF16:
            Mo, Qo = pieces(Mf)[0], pieces(Qf)[0]
        else:
            Mo, Qo = Mf.astype(np.float64), Qf.astype(np.float64)
        Sd = src.dense_panel(m0, m1, c0, c1)
        sup = Sd > 0
        L = Mo @ Qo.T
        want = np.where(sup, Sd - np.minimum(0, L), 0.0) @ Qo
        got = sol.support_term(side, block, kind)
        sol.sync()
        got = got.cpu().numpy()[:, :r]
        assert got.shape == want.shape
        assert np.all(got[~sup.any(axis=1)] == 0)          # rows without support stay zero
        assert rel(got, want) <= 1e-5, (name, side, kind, block, rel(got, want))
