"""Range-search chunk skipping (Sec. 4.3, eqs. nonzeros and range-search).

Before the dense kernel of a Delta-form step, balls around the normalised
rows of every 128-row M tile and every Q chunk clear the (tile, chunk)
pairs on which every L_ij <= 0; the kernel then skips both products there.
Checked here:

* soundness: on every cleared pair, no entry of L is positive (the oracle's
  Omega of eq. nonzeros on the same rows is empty there) and every pair of
  normalised rows is at squared distance >= 2 + 2^-6 (eq. range-search with
  the margin the test guarantees);
* exactness: a cleared chunk adds exactly zero, so the factors and momentum
  after steps and sweeps equal, bit for bit, those of the same steps without
  skipping; and the oracle's step within the usual tolerance;
* coverage: stochastic, exact (split K) and combined steps, both
  tensor-core precisions, r_pad 32, 64 and 128.

Inputs: factors whose rows cluster by community (block-diagonal rectified
product, the case of Sec. 4.3 in which it is sparse), S = max(0, W H) on
them (a zero-loss fixed point) or a block-structured graph; and random
factors, on which nothing is cleared."""
import numpy as np
import pytest

import oracle as O
from gpu_common import TOL, make_pair, rel, require_gpu, sync_oracle_to
from paper_2608_21607_gb300 import nmd as N
from paper_2608_21607_gb300 import workloads as WL

pytestmark = pytest.mark.gpu

GAMMA = 2.0 ** -7


@pytest.fixture(scope="module", autouse=True)
def gpu():
    return require_gpu()


def _clustered(m, n, r, clusters, seed, planted=True, run=None):
    W, H, _, _ = WL.community_factors(m, n, r, clusters, seed=seed, run=run)
    if planted:
        S = WL.csr_from_dense(np.maximum(0.0, W.astype(np.float64) @ H.astype(np.float64)))
    else:
        S = WL.communities(m, n, clusters, 12.0, seed=seed, run=run)
    return S, W, H


def _cdiv(a, b):
    return -(-a // b)


def _rows(orc, side, block, kind):
    """(M-side rows, Q-side rows) of a step in the oracle's fp64 state."""
    M, _, (m0, m1), Q, _, _ = orc._roles(side, block, kind)
    return M[m0:m1], Q


def _check_sound(mask, bn, Mr, Qr):
    """Every cleared (tile, chunk) pair: no positive L and every pair of
    normalised rows at squared distance >= 2 + 2 gamma."""
    cleared = 0
    pos = O.positive_set(Mr, Qr)
    nm = np.linalg.norm(Mr, axis=1)
    nq = np.linalg.norm(Qr, axis=1)
    for t in range(mask.shape[0]):
        for w in range(mask.shape[1]):
            bits = int(mask[t, w])
            while bits:
                b = (bits & -bits).bit_length() - 1
                bits &= bits - 1
                c = 32 * w + b
                r0, r1 = 128 * t, min(128 * t + 128, Mr.shape[0])
                q0, q1 = bn * c, min(bn * c + bn, Qr.shape[0])
                assert q0 < Qr.shape[0] and r0 < Mr.shape[0], (t, c)
                assert not pos[r0:r1, q0:q1].any(), (t, c)
                cos = (Mr[r0:r1] @ Qr[q0:q1].T) / np.maximum(np.outer(nm[r0:r1], nq[q0:q1]), 1e-300)
                assert cos.max() <= -GAMMA, (t, c, cos.max())
                cleared += 1
    return cleared


def _state(sol):
    W, H, EW, EH, _ = sol.get_state()
    return W, H, EW, EH


def _same(a, b):
    for x, y in zip(a, b):
        assert np.array_equal(x, y)


PRECS = [N.NMD_BF16, N.NMD_FP32]
# contiguous communities: tiles and chunks mostly inside one community, but a
# block of rows holds only a few communities, so its Gram matrix is close to
# rank-deficient (fine for the exactness and soundness checks, not for a
# comparison with the oracle)
CASES = [  # m, n, r, clusters, block_rows, block_cols
    (1500, 1300, 32, 8, 500, 480),
    (2100, 1900, 64, 12, 700, 640),
    (1300, 1200, 100, 6, 650, 600),
]
# communities in runs of 128 taken in turn, r = number of communities: every
# tile and chunk in one community and every block holding all of them
ORACLE_CASES = [  # m, n, r, clusters, run, block_rows, block_cols
    (4796, 4500, 16, 16, 128, 2048, 2048),
    (8300, 8250, 32, 32, 128, 4096, 4096),
]


@pytest.mark.parametrize("prec", PRECS, ids=["bf16", "fp32"])
@pytest.mark.parametrize("case", CASES, ids=["r32", "r64", "r100"])
def test_range_mask_is_sound_and_clears_chunks(case, prec):
    m, n, r, C, br, bc = case
    S, W, H = _clustered(m, n, r, C, seed=r)
    sol, orc = make_pair(S, r, W, H, block_rows=br, block_cols=bc, precision=prec, epilogue=N.NMD_EPI_DELTA)
    total = 0
    for side, block, kind in [(N.NMD_COL, 1, N.NMD_STOCH), (N.NMD_ROW, 0, N.NMD_STOCH),
                              (N.NMD_ROW, _cdiv(m, br) - 1, N.NMD_EXACT), (N.NMD_COL, 0, N.NMD_EXACT)]:
        mask, bn = sol.range_mask(side, block, kind)
        Mr, Qr = _rows(orc, side, block, kind)
        assert mask.shape == (_cdiv(Mr.shape[0], 128), _cdiv(_cdiv(Qr.shape[0], bn), 32))
        cleared = _check_sound(mask, bn, Mr, Qr)
        total += cleared
    assert total > 0


@pytest.mark.parametrize("prec", PRECS, ids=["bf16", "fp32"])
def test_range_mask_random_factors_clear_nothing_wrong(prec):
    S = WL.connectome(3000, seed=5)
    W, H = WL.init_factors(3000, 3000, 64, 5)
    sol, orc = make_pair(S, 64, W, H, block_rows=1000, block_cols=1000, precision=prec,
                         epilogue=N.NMD_EPI_DELTA)
    for side, block, kind in [(N.NMD_COL, 0, N.NMD_STOCH), (N.NMD_ROW, 2, N.NMD_EXACT)]:
        mask, bn = sol.range_mask(side, block, kind)
        Mr, Qr = _rows(orc, side, block, kind)
        _check_sound(mask, bn, Mr, Qr)


def _pair(S, r, W, H, br, bc, prec, skip, schedule=N.NMD_STOCH):
    return make_pair(S, r, W, H, block_rows=br, block_cols=bc, precision=prec, epilogue=N.NMD_EPI_DELTA,
                     schedule=schedule, skip_zero_chunks=skip)


def _steps(m, n, br, bc, ragged_stoch=True):
    """Stochastic steps on full blocks, exact steps on the ragged last row
    block and the first column block, and (optionally) a stochastic step on
    the ragged last column block."""
    steps = [(N.NMD_COL, 1, N.NMD_STOCH), (N.NMD_ROW, 0, N.NMD_STOCH), (N.NMD_ROW, _cdiv(m, br) - 1, N.NMD_EXACT),
             (N.NMD_COL, 0, N.NMD_EXACT)]
    return steps + [(N.NMD_COL, _cdiv(n, bc) - 1 if ragged_stoch else 0, N.NMD_STOCH)]


@pytest.mark.parametrize("prec", PRECS, ids=["bf16", "fp32"])
@pytest.mark.parametrize("case", CASES, ids=["r32", "r64", "r100"])
def test_range_skipping_gives_the_same_steps(case, prec):
    """Every step kind with and without range skipping: identical factors and
    momentum, and chunks were skipped."""
    m, n, r, C, br, bc = case
    S, W, H = _clustered(m, n, r, C, seed=r + 1, planted=False)
    on, _ = _pair(S, r, W, H, br, bc, prec, N.NMD_SKIP_RANGE)
    off, _ = _pair(S, r, W, H, br, bc, prec, N.NMD_SKIP_NONE)
    on.skip_count(reset=True)
    for side, block, kind in _steps(m, n, br, bc):
        on.block_update(side, block, kind)
        off.block_update(side, block, kind)
        _same(_state(on), _state(off))
    assert on.skip_count() > 0
    # combined row and column sub-sampling
    for side in (N.NMD_ROW, N.NMD_COL):
        on.block_update_combined(side, 1, 0)
        off.block_update_combined(side, 1, 0)
        _same(_state(on), _state(off))


@pytest.mark.parametrize("prec", PRECS, ids=["bf16", "fp32"])
@pytest.mark.parametrize("case", ORACLE_CASES, ids=["r16", "r32"])
def test_range_skipping_matches_the_oracle(case, prec):
    """Steps of every kind with range skipping against the oracle's steps
    (teacher forcing), on communities whose blocks have well-conditioned Gram
    matrices; the masks are sound, and from the clustered start they clear
    most chunks (a tile meets its own community in one chunk in `clusters`)."""
    m, n, r, C, run, br, bc = case
    S, W, H = _clustered(m, n, r, C, seed=r + 2, planted=False, run=run)
    on, orc = _pair(S, r, W, H, br, bc, prec, N.NMD_SKIP_RANGE)
    on.skip_count(reset=True)
    for i, (side, block, kind) in enumerate(_steps(m, n, br, bc, ragged_stoch=False)):
        sync_oracle_to(on, orc)
        mask, bn = on.range_mask(side, block, kind)
        Mr, Qr = _rows(orc, side, block, kind)
        cleared = _check_sound(mask, bn, Mr, Qr)
        chunks = _cdiv(Mr.shape[0], 128) * _cdiv(Qr.shape[0], bn)
        # from the clustered start at least half the chunks are cleared (a tile
        # meets its own community in one chunk in `clusters`); the steps then
        # spread the rows, and later masks clear fewer (possibly none)
        if i == 0:
            assert cleared >= chunks // 2, (side, block, kind, cleared, chunks)
        on.block_update(side, block, kind)
        orc.block_update(side, block, kind)
        M, E, (m0, m1), _, _, _ = orc._roles(side, block, kind)
        W1, H1, EW, EH = _state(on)
        got = (W1 if M is orc.A else H1.T)[m0:m1]
        assert rel(got, M[m0:m1]) <= TOL[prec], (side, block, kind, rel(got, M[m0:m1]))
    assert on.skip_count() > 0


@pytest.mark.parametrize("prec", PRECS, ids=["bf16", "fp32"])
def test_range_skipping_sweeps_bit_identical(prec):
    m, n, r, C, br, bc = 2100, 1900, 64, 12, 700, 640
    S, W, H = _clustered(m, n, r, C, seed=9, planted=False)
    for schedule in (N.NMD_STOCH, N.NMD_EXACT):
        on, _ = _pair(S, r, W, H, br, bc, prec, N.NMD_SKIP_RANGE, schedule)
        off, _ = _pair(S, r, W, H, br, bc, prec, N.NMD_SKIP_NONE, schedule)
        on.skip_count(reset=True)
        for _ in range(2):
            on.sweep()
            off.sweep()
        _same(_state(on), _state(off))
        assert on.skip_count() > 0
        lo, lf = on.loss(), off.loss()
        assert lo["obj"] == lf["obj"]


def test_range_mode_needs_a_known_value():
    S, W, H = _clustered(300, 200, 16, 4, seed=1)
    with pytest.raises(N.NmdError):
        N.Solver(S, 16, block_rows=100, block_cols=100, skip_zero_chunks=3)
