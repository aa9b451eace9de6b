"""Parity of the CUDA path (through the C ABI) with the fp64 oracle.

Per block step from an identical state (teacher forcing), on the seeded
stand-ins of the five workloads at sizes the oracle finishes in seconds,
each spanning several tiles and a ragged last block: right-hand sides and
Gram matrices, updated factors and momentum, losses; bit-exact block order
and sparse traversal; fixed points; determinism, checkpoint/resume and the
error paths.  Tolerances: relative Frobenius error 1e-4 for the fp32-accurate
paths, 5e-3 with bf16 operands.
"""
import numpy as np
import pytest

import oracle as O
from paper_2608_21607_gb300 import nmd as N
from paper_2608_21607_gb300 import workloads as WL

from gpu_common import TOL, PREC_NAMES, make_pair, rel, require_gpu, small_cases, sync_oracle_to

pytestmark = pytest.mark.gpu

PRECISIONS = [N.NMD_SIMT, N.NMD_BF16, N.NMD_FP32]
EPILOGUES = [N.NMD_EPI_Z, N.NMD_EPI_DELTA]
KINDS = [(O.ROW, O.EXACT), (O.COL, O.EXACT), (O.COL, O.STOCH), (O.ROW, O.STOCH)]

_CASES = None


def cases():
    global _CASES
    if _CASES is None:
        _CASES = {c[0]: c for c in small_cases()}
    return _CASES


CASE_NAMES = ["planted600x400_r4_exact", "identity1000_r3", "planted1500x1300_r32",
              "connectome4000_r64", "connectome3400_r100", "connectome6000_r256"]


@pytest.fixture(scope="module", autouse=True)
def gpu():
    return require_gpu()


def _pair(name, precision, epilogue=N.NMD_EPI_Z, momentum=False, **kw):
    _, S, r, W, H, br, bc, sched = cases()[name]
    EW = EH = None
    if momentum:
        rng = np.random.default_rng(11)
        EW = (0.01 * rng.standard_normal(W.shape)).astype(np.float32)
        EH = (0.01 * rng.standard_normal(H.shape)).astype(np.float32)
    kw.setdefault("schedule", sched)
    return make_pair(S, r, W, H, block_rows=br, block_cols=bc, precision=precision,
                     epilogue=epilogue, EW=EW, EH=EH, **kw)


def _nblocks(orc, side):
    return O.num_blocks(orc.m if side == O.ROW else orc.n,
                        orc.opts.block_rows if side == O.ROW else orc.opts.block_cols)


@pytest.mark.parametrize("name", CASE_NAMES)
def test_block_order_bit_exact(name):
    sol, orc = _pair(name, N.NMD_SIMT, seed=0)
    for seed in (0, 12345):
        sol2, _ = _pair(name, N.NMD_SIMT, seed=seed)
        for sweep in (0, 1, 7, 199):
            for side in (O.ROW, O.COL):
                K = _nblocks(orc, side)
                assert sol2.block_order(sweep, side) == O.block_permutation(seed, sweep, side, K)


@pytest.mark.parametrize("name", CASE_NAMES)
def test_sparse_traversal_bit_exact(name):
    sol, orc = _pair(name, N.NMD_SIMT)
    for side, kind in KINDS:
        K = _nblocks(orc, side)
        for block in sorted({0, K // 2, K - 1}):
            rows, q = sol.panel_traversal(side, block, kind)
            er, eq = orc.traversal(side, block, kind)
            assert np.array_equal(rows, er) and np.array_equal(q, eq), (side, kind, block)


@pytest.mark.parametrize("prec", PRECISIONS, ids=lambda p: PREC_NAMES[p])
@pytest.mark.parametrize("epi", EPILOGUES, ids=["zform", "delta"])
@pytest.mark.parametrize("name", CASE_NAMES)
def test_block_terms_parity(name, epi, prec):
    """R = Z Q (or Delta Q) and G = Q^T Q of single block steps."""
    sol, orc = _pair(name, prec, epi)
    for side, kind in KINDS:
        K = _nblocks(orc, side)
        for block in sorted({0, K - 1}):
            Rg, Gg = sol.block_terms(side, block, kind)
            Ro, Go = orc.block_terms(side, block, kind)
            if epi == N.NMD_EPI_DELTA:
                M, _, (m0, m1), _, _, _ = orc._roles(side, block, kind)
                Ro = Ro - M[m0:m1] @ Go               # eq. Delta: Delta Q = Z Q - L Q
            assert rel(Gg, Go) <= 2e-6, (side, kind, block)
            assert rel(Rg, Ro) <= TOL[prec], (side, kind, block, rel(Rg, Ro))


@pytest.mark.parametrize("prec", PRECISIONS, ids=lambda p: PREC_NAMES[p])
@pytest.mark.parametrize("epi", EPILOGUES, ids=["zform", "delta"])
@pytest.mark.parametrize("name", CASE_NAMES)
def test_trajectory_parity(name, epi, prec):
    """Every block step of the first two sweeps of the workload's own schedule,
    each from the GPU's current state (teacher forcing): updated factors,
    momentum and, after each sweep, the losses."""
    sol, orc = _pair(name, prec, epi)
    worst = 0.0
    for sweep in range(2):
        for side, block, kind in orc.sweep_steps(sweep):
            sync_oracle_to(sol, orc)
            M, E, (m0, m1), Q, _, _ = orc._roles(side, block, kind)
            G = Q.T @ Q
            ev = np.linalg.eigvalsh(G)
            sol.block_update(side, block, kind)
            orc.block_update(side, block, kind)
            W, H, EW, EH, _ = sol.get_state()
            got = (W if M is orc.A else H.T)[m0:m1]
            err = rel(got, M[m0:m1])
            worst = max(worst, err)
            assert err <= TOL[prec], (sweep, side, kind, block, err, "kappa(G) = %.1f" % (ev[-1] / ev[0]))
            if kind == O.STOCH:
                gotE = (EW if M is orc.A else EH.T)[m0:m1]
                assert rel(gotE, E[m0:m1]) <= 10 * TOL[prec]
        sync_oracle_to(sol, orc)
        g, o = sol.loss(), orc.loss()
        for k in ("obj", "rmse", "wjd"):
            assert abs(g[k] - o[k]) <= TOL[prec] * max(abs(o[k]), 1e-3), (sweep, k, g[k], o[k])


@pytest.mark.parametrize("prec", PRECISIONS, ids=lambda p: PREC_NAMES[p])
@pytest.mark.parametrize("epi", EPILOGUES, ids=["zform", "delta"])
@pytest.mark.parametrize("name", CASE_NAMES)
def test_block_update_parity(name, epi, prec):
    """Updated factors and momentum after one step from an identical state,
    for all four kinds of step in turn.  The sequence (exact steps on a
    stochastic workload) drives the block Gram matrices to condition numbers
    in the thousands, a stress test of the accuracy of the second product."""
    sol, orc = _pair(name, prec, epi, momentum=True, eta=0.9, gamma=0.8)
    for side, kind in KINDS:
        K = _nblocks(orc, side)
        for block in sorted({K - 1, 0}):
            sync_oracle_to(sol, orc)
            sol.block_update(side, block, kind)
            orc.block_update(side, block, kind)
            W, H, EW, EH, _ = sol.get_state()
            M, E, (m0, m1), _, _, _ = orc._roles(side, block, kind)
            got = (W if M is orc.A else H.T)[m0:m1]
            gotE = (EW if M is orc.A else EH.T)[m0:m1]
            assert rel(got, M[m0:m1]) <= TOL[prec], (side, kind, block, rel(got, M[m0:m1]))
            if kind == O.STOCH:
                assert rel(gotE, E[m0:m1]) <= 10 * TOL[prec], (side, kind, block)


@pytest.mark.parametrize("prec", PRECISIONS, ids=lambda p: PREC_NAMES[p])
@pytest.mark.parametrize("name", CASE_NAMES)
def test_loss_parity(name, prec):
    sol, orc = _pair(name, prec)
    for trial in range(2):
        g = sol.loss()
        o = orc.loss()
        assert g["s_fro"] == pytest.approx(o["s_fro"], rel=1e-6)
        for k in ("obj", "rmse", "wjd"):
            assert abs(g[k] - o[k]) <= TOL[prec] * max(abs(o[k]), 1e-3), (k, g[k], o[k])
        assert g["obj"] >= g["rmse"] * (1 - 1e-6)          # Prop. 'Lipschitz'
        if trial == 0:   # move to a point with many positive entries of L
            side, kind = (O.COL, O.STOCH) if orc.opts.block_rows < orc.m else (O.ROW, O.EXACT)
            sol.block_update(side, 0, kind)
            sync_oracle_to(sol, orc)


@pytest.mark.parametrize("prec", PRECISIONS, ids=lambda p: PREC_NAMES[p])
def test_exact_sweeps_monotone_and_track_oracle(prec):
    """Config-1 shape: 600x400 planted, r=4, blocks of 128, exact sweeps."""
    sol, orc = _pair("planted600x400_r4_exact", prec, schedule=N.NMD_EXACT, gamma=0.0)
    prev = sol.loss()["obj"]
    for s in range(3):
        for side, block, kind in orc.sweep_steps(s):
            sol.block_update(side, block, kind)
            cur = sol.loss()["obj"]
            assert cur <= prev * (1 + 10 * TOL[prec])
            prev = cur
        orc.sweep()
    W, H = sol.get_factors()
    assert rel(W @ H, orc.A @ orc.B.T) <= 50 * TOL[prec]


@pytest.mark.parametrize("prec", PRECISIONS, ids=lambda p: PREC_NAMES[p])
def test_planted_zero_loss_point_is_fixed(prec):
    """Prop. 1: the rank-(d+1) completion [U, 1][V, -tau]^T of a planted S."""
    S, U, V, tau = WL.planted(700, 500, 4, tau=0.5, seed=7)
    W0 = np.hstack([U, np.ones((700, 1))]).astype(np.float32)
    H0 = np.hstack([V, -tau * np.ones((500, 1))]).T.astype(np.float32)
    sol = N.Solver(S, 5, block_rows=128, block_cols=128, precision=prec, gamma=0.9)
    sol.set_factors(W0, H0)
    l0 = sol.loss()
    assert l0["obj"] < 20 * TOL[prec] and l0["rmse"] < 20 * TOL[prec]
    sol.sweep()
    W, H = sol.get_factors()
    assert rel(W @ H, W0 @ H0) <= 20 * TOL[prec]


@pytest.mark.parametrize("prec", [N.NMD_SIMT, N.NMD_FP32], ids=lambda p: PREC_NAMES[p])
def test_identity_omega_point_is_fixed(prec):
    """Corollary 'ident': I_n = max(0, Omega) with rank-3 factors (eq. Omega).

    Omega_ij is a difference of products of size 1/(1 - cos(2 pi/n)), and its
    entries next to the diagonal are exactly 0: bf16 operands (8 significant
    bits) cannot resolve them, so only the fp32-accurate paths are checked."""
    n = 64
    th = 2 * np.pi * np.arange(n) / n
    c = np.cos(2 * np.pi / n)
    W0 = (np.stack([np.cos(th), np.sin(th), -c * np.ones(n)], 1) / (1 - c)).astype(np.float32)
    H0 = np.stack([np.cos(th), np.sin(th), np.ones(n)], 0).astype(np.float32)
    sol = N.Solver(WL.identity(n), 3, block_rows=16, block_cols=16, precision=prec, gamma=0.9)
    sol.set_factors(W0, H0)
    # factor entries of size 200 whose products cancel to 0 or 1: fp32
    # rounding alone moves L by ~1e-5 and a sweep by ~1e-4 relative
    assert sol.loss()["obj"] < (1e-4 if prec == N.NMD_SIMT else 2e-3)
    sol.sweep()
    W, H = sol.get_factors()
    assert rel(W @ H, W0.astype(np.float64) @ H0) < 1e-3


@pytest.mark.parametrize("prec", [N.NMD_SIMT, N.NMD_FP32], ids=lambda p: PREC_NAMES[p])
def test_ring_point_is_fixed(prec):
    """Prop. 'ring': the ring matrix (1 on the diagonal, delta = 1/2 between
    neighbours) is max(0, L) for the rank-3 L of points on a circle of
    radius r with threshold tau (eqs. tau, r2); support values other than 1
    on the GPU path.  Products of size r^2 ~ 40 cancel to 0, 1/2 or 1, so
    only the fp32-accurate paths are checked (as for eq. Omega)."""
    n, delta = 48, 0.5
    phi = 2 * np.pi / n
    tau = (np.cos(phi) - delta) / (1 - delta)
    r2 = (1 - delta) / (1 - np.cos(phi))
    th = phi * np.arange(n)
    r = np.sqrt(r2)
    W0 = np.stack([r * np.cos(th), r * np.sin(th), -tau * r2 * np.ones(n)], 1).astype(np.float32)
    H0 = np.stack([r * np.cos(th), r * np.sin(th), np.ones(n)], 0).astype(np.float32)
    i, j = np.meshgrid(np.arange(n), np.arange(n), indexing="ij")
    d = np.abs(i - j)
    D = np.where(d == 0, 1.0, np.where((d == 1) | (d == n - 1), delta, 0.0))
    sol = N.Solver(WL.csr_from_dense(D), 3, block_rows=16, block_cols=16, precision=prec, gamma=0.9)
    sol.set_factors(W0, H0)
    assert sol.loss()["obj"] < (1e-4 if prec == N.NMD_SIMT else 2e-3)
    sol.sweep()
    W, H = sol.get_factors()
    assert rel(W @ H, W0.astype(np.float64) @ H0) < 1e-3


@pytest.mark.parametrize("r, prec", [(4, N.NMD_SIMT), (200, N.NMD_BF16), (200, N.NMD_FP32)])
def test_not_spd_is_reported_and_update_skipped(r, prec):
    # 700 columns in blocks of 233: the last block has 1 column < r, so its
    # Gram matrix has rank 1 (r = 4: the register-resident factorisation;
    # r = 200, r_pad = 256: the shared-memory one)
    S, _, _, _ = WL.planted(300, 700, 4, tau=0.5, seed=0)
    W, H = WL.init_factors(300, 700, r, 0)
    sol = N.Solver(S, r, block_rows=100, block_cols=233, precision=prec)
    sol.set_factors(W, H)
    sol.block_update(N.NMD_COL, 3, N.NMD_STOCH)
    with pytest.raises(N.NmdError) as e:
        sol.sync()
    assert e.value.status == N.NMD_ERR_NOT_SPD
    W1, H1 = sol.get_factors()
    assert np.array_equal(W1, W) and np.array_equal(H1, H)   # update was skipped
    sol.block_update(N.NMD_COL, 0, N.NMD_STOCH)              # the handle stays usable
    sol.sync()
    assert not np.array_equal(sol.get_factors()[0], W)


def test_divergence_is_reported():
    S, _, _, _ = WL.planted(300, 200, 4, tau=0.5, seed=0)
    W, H = WL.init_factors(300, 200, 4, 0)
    sol = N.Solver(S, 4, block_rows=100, block_cols=100, precision=N.NMD_SIMT, eta=1e38)
    sol.set_factors(100 * W, 100 * H)
    sol.block_update(N.NMD_COL, 0, N.NMD_STOCH)
    with pytest.raises(N.NmdError) as e:
        sol.sync()
    assert e.value.status == N.NMD_ERR_DIVERGED


def test_bad_block_index_rejected():
    S, _, _, _ = WL.planted(300, 200, 4, tau=0.5, seed=0)
    sol = N.Solver(S, 4, block_rows=100, block_cols=100, precision=N.NMD_SIMT)
    with pytest.raises(N.NmdError) as e:
        sol.block_update(N.NMD_ROW, 3, N.NMD_EXACT)
    assert e.value.status == N.NMD_ERR_INVALID
    with pytest.raises(N.NmdError):
        sol.block_update(N.NMD_COL, -1, N.NMD_STOCH)


@pytest.mark.parametrize("order", [N.NMD_ALTERNATE, N.NMD_PHASED], ids=["alternate", "phased"])
@pytest.mark.parametrize("prec", [N.NMD_BF16, N.NMD_FP32], ids=lambda p: PREC_NAMES[p])
def test_sweep_schedule_equals_serial_steps(prec, order):
    """A sweep (four streams; the rows the next step does not read updated
    beside it) gives bit for bit the factors and momentum of the same block
    steps run one after another, in the oracle's order of the sweep."""
    _, S, r, W, H, br, bc, _ = cases()["planted1500x1300_r32"]
    a = N.Solver(S, r, block_rows=br, block_cols=bc, precision=prec, order=order)
    b = N.Solver(S, r, block_rows=br, block_cols=bc, precision=prec, order=order)
    a.set_factors(W, H)
    b.set_factors(W, H)
    orc = O.State(S, np.asarray(W, np.float64), np.asarray(H, np.float64),
                  O.Options(block_rows=br, block_cols=bc, order=order))
    a.sweep()
    for side, block, kind in orc.sweep_steps(0):
        b.block_update(side, block, kind)
    a.sync()
    b.sync()
    for x, y in zip(a.get_state()[:4], b.get_state()[:4]):
        assert np.array_equal(x, y)


@pytest.mark.parametrize("prec", PRECISIONS, ids=lambda p: PREC_NAMES[p])
def test_deterministic_and_resumable(prec):
    _, S, r, W, H, br, bc, _ = cases()["connectome4000_r64"]
    a = N.Solver(S, r, block_rows=br, block_cols=bc, precision=prec)
    b = N.Solver(S, r, block_rows=br, block_cols=bc, precision=prec)
    a.set_factors(W, H)
    b.set_factors(W, H)
    for _ in range(2):
        a.sweep()
        b.sweep()
    sa, sb = a.get_state(), b.get_state()
    for x, y in zip(sa[:4], sb[:4]):
        assert np.array_equal(x, y)                      # bit-identical reruns
    c = N.Solver(S, r, block_rows=br, block_cols=bc, precision=prec)
    c.set_state(*sa[:4], sa[4])                         # resume from a checkpoint
    a.sweep()
    c.sweep()
    for x, y in zip(a.get_state()[:4], c.get_state()[:4]):
        assert np.array_equal(x, y)
