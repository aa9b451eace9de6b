"""Parity at the full size of every benchmark workload, with its own step
sizes: the connectome-shaped graphs (139,255 x 139,255, 2,785,100 nonzeros;
r = 64 with blocks of 4096, r = 256 with blocks of 8192), the planted
20,000 x 20,000 matrix (r = 32, blocks of 2048, 1.99e7 nonzeros) and the
identity I_4096 (r = 3, blocks of 512).  Each checked step starts from the
GPU's current state (teacher forcing) and is compared with the oracle's full
step: every updated row, element by element (relative Frobenius error), and
the momentum.  The benchmark times these steps inside sweeps; a sweep gives
bit for bit the factors of the same steps run one by one (test_gpu_parity.py),
so the serial block updates here check the same arithmetic.  The losses are
checked on a seeded sample of 2,048 rows of the connectome against all of its
139,255 columns.  Each test takes seconds on the GPU and up to tens of seconds
on the host cores for the oracle's full steps."""
import gc

import numpy as np
import pytest

import oracle as O
from gpu_common import TOL, make_pair, rel, require_gpu, sync_oracle_to
from paper_2608_21607_gb300 import nmd as N
from paper_2608_21607_gb300 import workloads as WL

pytestmark = [pytest.mark.gpu, pytest.mark.slow]   # collected after every other test file (file name)


@pytest.fixture(scope="module", autouse=True)
def gpu():
    return require_gpu()


@pytest.fixture(scope="module")
def wl64():
    return WL.workload("connectome_r64")


@pytest.fixture(scope="module")
def wl256():
    return WL.workload("connectome_r256")


@pytest.fixture(scope="module")
def wlpm():
    return WL.workload("planted_medium")


def _check_steps(wl, precision, epilogue, pick):
    """pick(orc) -> the (side, block, kind) steps to check, in order."""
    sol, orc = make_pair(wl.S, wl.r, wl.W0, wl.H0, block_rows=wl.block_rows, block_cols=wl.block_cols,
                         precision=precision, epilogue=epilogue, eta=wl.eta, gamma=wl.gamma)
    try:
        for side, block, kind in pick(orc):
            sync_oracle_to(sol, orc)
            sol.block_update(side, block, kind)
            orc.block_update(side, block, kind)
            W, H, EW, EH, _ = sol.get_state()
            M, E, (m0, m1), _, _, _ = orc._roles(side, block, kind)
            got = (W if M is orc.A else H.T)[m0:m1]
            gotE = (EW if M is orc.A else EH.T)[m0:m1]
            err = rel(got, M[m0:m1])
            assert err <= TOL[precision], (wl.name, side, block, err)
            assert rel(gotE, E[m0:m1]) <= 10 * TOL[precision], (wl.name, side, block)
            assert np.isfinite(got).all()
    finally:
        del sol
        gc.collect()


def test_connectome_r64_bf16_z_full_size(wl64):
    """The benchmark's configuration: the first two steps of sweep 0 (one of
    each side) and the ragged last column block (4087 rows)."""
    last = -(-wl64.n // wl64.block_cols) - 1
    _check_steps(wl64, N.NMD_BF16, N.NMD_EPI_Z,
                 lambda orc: orc.sweep_steps(0)[:2] + [(N.NMD_COL, last, N.NMD_STOCH)])


def test_connectome_r64_fp32_full_size(wl64):
    _check_steps(wl64, N.NMD_FP32, N.NMD_EPI_Z, lambda orc: orc.sweep_steps(0)[:1])


def test_connectome_r64_bf16_delta_full_size(wl64):
    _check_steps(wl64, N.NMD_BF16, N.NMD_EPI_DELTA, lambda orc: orc.sweep_steps(0)[:1])


def test_connectome_r256_bf16_full_size(wl256):
    _check_steps(wl256, N.NMD_BF16, N.NMD_EPI_Z, lambda orc: orc.sweep_steps(0)[:1])


def test_connectome_r256_fp32_full_size(wl256):
    """The fp32-accurate mode at r = 256: W's hi and lo pieces take half of
    TMEM, so each CTA accumulates one 128-column half of R."""
    _check_steps(wl256, N.NMD_FP32, N.NMD_EPI_Z, lambda orc: orc.sweep_steps(0)[:1])


def _last_blocks(orc):
    Kc = -(-orc.n // orc.opts.block_cols)
    Kr = -(-orc.m // orc.opts.block_rows)
    return [(N.NMD_COL, Kc - 1, N.NMD_STOCH), (N.NMD_ROW, Kr - 1, N.NMD_STOCH)]


@pytest.mark.parametrize("prec", [N.NMD_BF16, N.NMD_FP32], ids=["bf16", "fp32"])
def test_planted_medium_full_size(wlpm, prec):
    """20,000 x 20,000 with about 2e6 support entries per step: rows of about
    100 entries per panel go through the long-row support kernel, rows above
    128 through its slices and the fixed-order slice reduction.  The first
    column and row steps of sweep 0 and the ragged last blocks (1,568 rows)."""
    _check_steps(wlpm, prec, N.NMD_EPI_Z, lambda orc: orc.sweep_steps(0)[:2] + _last_blocks(orc))


def test_identity_full_size_sweep():
    """I_4096 at r = 3 (padded to 16): every step of the first sweep."""
    wl = WL.workload("identity")
    _check_steps(wl, N.NMD_BF16, N.NMD_EPI_Z, lambda orc: orc.sweep_steps(0))


@pytest.mark.parametrize("prec", [N.NMD_BF16, N.NMD_FP32], ids=["bf16", "fp32"])
def test_connectome_loss_full_width_sample(wl64, prec):
    """nmd_loss (eqs. auxCost/SLloss, RMSE, WJD) on a seeded sample of 2,048
    rows of the connectome against all 139,255 columns, after one sweep from
    the benchmark's start: the sub-matrix S[rows, :] with W[rows] and the
    whole H, against the oracle's sums over the same rows.  The dense pass
    covers 2.85e8 entries, the support pass the rows' 41k nonzeros."""
    rng = np.random.default_rng(2048)
    rows = np.sort(rng.choice(wl64.m, 2048, replace=False))
    sol = N.Solver(wl64.S, wl64.r, block_rows=wl64.block_rows, block_cols=wl64.block_cols,
                   precision=prec, eta=wl64.eta, gamma=wl64.gamma)
    sol.set_factors(wl64.W0, wl64.H0)
    sol.sweep()
    W, H = sol.get_factors()
    del sol
    gc.collect()
    # the sampled rows as a problem of their own
    rp = wl64.S.row_ptr
    sub_ptr = np.zeros(len(rows) + 1, np.int64)
    sub_ptr[1:] = np.cumsum(rp[rows + 1] - rp[rows])
    sub_col = np.concatenate([wl64.S.col_idx[rp[i]:rp[i + 1]] for i in rows])
    sub_val = np.concatenate([wl64.S.vals[rp[i]:rp[i + 1]] for i in rows])
    Ssub = WL.CSR(len(rows), wl64.n, sub_ptr, sub_col.astype(np.int32), sub_val)
    sub = N.Solver(Ssub, wl64.r, block_rows=512, block_cols=4096, precision=prec)
    sub.set_factors(np.ascontiguousarray(W[rows]), H)
    got = sub.loss()
    want = O.loss(O.Sparse.from_csr(wl64.S), W.astype(np.float64), H.T.astype(np.float64), rows=rows)
    s_sub = float(np.sqrt(np.sum(np.asarray(sub_val, np.float64) ** 2)))
    tol = 5e-3 if prec == N.NMD_BF16 else 1e-4
    assert abs(got["obj"] - np.sqrt(want["zl2"]) / s_sub) <= tol * np.sqrt(want["zl2"]) / s_sub
    assert abs(got["rmse"] - np.sqrt(want["err2"]) / s_sub) <= tol * np.sqrt(want["err2"]) / s_sub
    wjd = 1.0 - want["sum_min"] / want["sum_max"]
    assert abs(got["wjd"] - wjd) <= tol * wjd


@pytest.mark.parametrize("prec", [N.NMD_BF16, N.NMD_FP32], ids=["bf16", "fp32"])
def test_connectome_combined_full_size(wl64, prec):
    """Combined row and column sub-sampling on the full connectome: W_I from
    H_:J and H_:J from W_I for the ragged last blocks and a middle pair
    (4,096 x 4,096 panels holding the hub rows)."""
    sol, orc = make_pair(wl64.S, wl64.r, wl64.W0, wl64.H0, block_rows=wl64.block_rows,
                         block_cols=wl64.block_cols, precision=prec, eta=wl64.eta, gamma=wl64.gamma)
    K = -(-wl64.n // wl64.block_cols)
    try:
        for side, I, J in [(N.NMD_ROW, K - 1, 17), (N.NMD_COL, 5, K - 1), (N.NMD_ROW, 11, 11)]:
            sync_oracle_to(sol, orc)
            sol.block_update_combined(side, I, J)
            orc.block_update_combined(side, I, J)
            W, H, EW, EH, _ = sol.get_state()
            if side == N.NMD_ROW:
                a, b = I * wl64.block_rows, min(wl64.m, (I + 1) * wl64.block_rows)
                got, want = W[a:b], orc.A[a:b]
            else:
                a, b = J * wl64.block_cols, min(wl64.n, (J + 1) * wl64.block_cols)
                got, want = H.T[a:b], orc.B[a:b]
            assert rel(got, want) <= TOL[prec], (side, I, J, rel(got, want))
    finally:
        del sol
        gc.collect()
