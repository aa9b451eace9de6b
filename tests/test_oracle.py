"""Pins of the fp64 oracle against what the paper and mathematics fix.

Each test checks the oracle through a route other than its own code: a
published test vector, a textbook factorisation, a library least-squares
solve on a dense brute-force problem, a closed-form zero-loss point from the
paper, or an invariant the paper proves.
"""
import math
import os

import numpy as np
import pytest

import oracle as O
from paper_2608_21607_gb300 import workloads as WL

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _read_numbers(name):
    rows = []
    for line in open(os.path.join(GOLDEN, name)):
        line = line.strip()
        if line and not line.startswith("#"):
            rows.append([float(x) if "." in x or "e" in x else int(x) for x in line.split()])
    return rows


def _rand_sparse(m, n, density, seed):
    rng = np.random.default_rng(seed)
    D = np.where(rng.random((m, n)) < density, rng.random((m, n)) + 0.1, 0.0)
    return WL.csr_from_dense(D, dtype=np.float64), D


# --------------------------------------------------------------------------
# block order
# --------------------------------------------------------------------------

def test_splitmix64_reference_vector():
    expect = [row[0] for row in _read_numbers("splitmix64_seed1234567.txt")]
    g = O.SplitMix64(1234567)
    assert [g.next() for _ in range(5)] == expect


def test_block_permutation_is_a_seeded_permutation():
    for K in (1, 2, 8, 34, 157):
        p = O.block_permutation(0, 0, 0, K)
        assert sorted(p) == list(range(K))
        assert p == O.block_permutation(0, 0, 0, K)
    a = O.block_permutation(0, 0, O.ROW, 34)
    assert a != O.block_permutation(0, 1, O.ROW, 34)
    assert a != O.block_permutation(0, 0, O.COL, 34)
    assert a != O.block_permutation(1, 0, O.ROW, 34)


def test_block_permutation_golden():
    """Regression against permutations written by tests/golden/make_golden.py."""
    for row in _read_numbers("block_order.txt"):
        seed, sweep, side, K = row[:4]
        assert O.block_permutation(seed, sweep, side, K) == row[4:]


_SM64 = [row[0] for row in _read_numbers("splitmix64_seed1234567.txt")]
_GOLDEN_GAMMA = 0x9E3779B97F4A7C15


def test_fisher_yates_hand_derived_from_published_vector():
    """Shuffle of 6 blocks driven by SplitMix64 from state 1234567, derived by
    hand from the published outputs v1..v5 (tests/golden/splitmix64_seed1234567.txt):
      i=5: j = v1 mod 6 = 3 -> [0 1 2 5 4 3]
      i=4: j = v2 mod 5 = 3 -> [0 1 2 4 5 3]
      i=3: j = v3 mod 4 = 3 -> [0 1 2 4 5 3]
      i=2: j = v4 mod 3 = 1 -> [0 2 1 4 5 3]
      i=1: j = v5 mod 2 = 1 -> [0 2 1 4 5 3]"""
    assert [_SM64[0] % 6, _SM64[1] % 5, _SM64[2] % 4, _SM64[3] % 3, _SM64[4] % 2] == [3, 3, 3, 1, 1]
    assert O.fisher_yates(6, O.SplitMix64(1234567)) == [0, 2, 1, 4, 5, 3]


def test_block_order_state_derivation_from_published_vector():
    """state = mix(seed) xor mix((sweep << 1) | side), with both mixes taken
    from the published vector: mix(x) is the first output of a generator
    started at x - 0x9E3779B97F4A7C15, so mix(1234567 + g) = v1 and
    mix(1234567 + 2 g) = v2 (g = the golden gamma)."""
    mask = (1 << 64) - 1
    x1 = (1234567 + _GOLDEN_GAMMA) & mask
    x2 = (1234567 + 2 * _GOLDEN_GAMMA) & mask
    assert O.splitmix64_mix(x1) == _SM64[0] and O.splitmix64_mix(x2) == _SM64[1]
    seed, sweep, side = x1, x2 >> 1, x2 & 1
    state = _SM64[0] ^ _SM64[1]
    for K in (2, 5, 34):
        assert O.block_permutation(seed, sweep, side, K) == O.fisher_yates(K, O.SplitMix64(state))
    # swapping the roles of seed and (sweep, side) changes the order
    assert O.block_permutation(seed, sweep, 1 - side, 34) != O.block_permutation(seed, sweep, side, 34)


def _chi2_orders(perm_fn, K=4, samples=24000):
    counts = {}
    for s in range(samples):
        p = tuple(perm_fn(s))
        counts[p] = counts.get(p, 0) + 1
    cells = math.factorial(K)
    e = samples / cells
    return len(counts), sum((counts.get(p, 0) - e) ** 2 / e for p in counts) + (cells - len(counts)) * e


# chi-square with 23 degrees of freedom: mean 23, sd 6.8; P(chi2 > 60) ~ 4e-5
_CHI2_23_BOUND = 60.0


def test_fisher_yates_uniform_chi_square():
    """All 4! orders of 4 blocks are equally likely over 24,000 sweeps (chi-square
    with 23 degrees of freedom below 60)."""
    seen, chi2 = _chi2_orders(lambda s: O.block_permutation(7, s, 0, 4))
    assert seen == 24
    assert chi2 < _CHI2_23_BOUND, chi2


def test_chi_square_rejects_the_naive_shuffle():
    """The same statistic on the classic slip j = next() mod K (a swap with any
    position at every step: 4^4 = 256 equally likely paths over 24 orders) is
    far above the bound, so the uniformity test above can tell them apart."""
    def naive(s):
        g = O.SplitMix64(O.splitmix64_mix(7) ^ O.splitmix64_mix(s << 1))
        p = list(range(4))
        for i in range(3, -1, -1):
            j = g.next() % 4
            p[i], p[j] = p[j], p[i]
        return p
    _, chi2 = _chi2_orders(naive)
    assert chi2 > 10 * _CHI2_23_BOUND, chi2


# --------------------------------------------------------------------------
# Z update (eq. updateZ) and the Delta identity (eq. updateD)
# --------------------------------------------------------------------------

def test_update_z_constraints_and_delta_identity():
    rng = np.random.default_rng(1)
    S = np.where(rng.random((30, 20)) < 0.2, rng.random((30, 20)) + 0.05, 0.0)
    L = rng.standard_normal((30, 20))
    Z = O.update_z(S, L)
    sup = S > 0
    assert np.array_equal(Z[sup], S[sup])            # S = max(0, Z) on the support
    assert np.all(Z[~sup] <= 0)                        # and Z <= 0 off it
    assert np.array_equal(np.maximum(0, Z), S)
    Shat = np.maximum(0, L)
    delta = sup * (S + Shat - L) - Shat                # eq. updateD
    np.testing.assert_allclose(Z - L, delta, rtol=0, atol=1e-15)
    # Z minimises ||Z - L|| subject to max(0, Z) = S, entry by entry:
    for z, l, s in zip(Z.ravel(), L.ravel(), S.ravel()):
        cands = [s] if s > 0 else [min(0.0, l), 0.0, -abs(l) - 1.0]
        assert abs(z - l) <= min(abs(c - l) for c in cands) + 1e-15


# --------------------------------------------------------------------------
# dense linear algebra
# --------------------------------------------------------------------------

def test_cholesky_textbook_example():
    rows = _read_numbers("cholesky_textbook.txt")
    G = np.array(rows[:3], dtype=float)
    C = np.array(rows[3:], dtype=float)
    np.testing.assert_allclose(O.cholesky(G), C, atol=1e-14)


def test_cholesky_and_solve_against_library():
    rng = np.random.default_rng(2)
    for r in (1, 3, 16, 64):
        Q = rng.standard_normal((3 * r + 5, r))
        G = Q.T @ Q
        C = O.cholesky(G)
        np.testing.assert_allclose(C, np.linalg.cholesky(G), rtol=1e-10, atol=1e-12)
        R = rng.standard_normal((40, r))
        X = O.solve_normal(C, R)
        np.testing.assert_allclose(X, np.linalg.solve(G, R.T).T, rtol=1e-9, atol=1e-10)


def test_cholesky_rejects_non_spd():
    with pytest.raises(O.NotSPD):
        O.cholesky(np.array([[1.0, 2.0], [2.0, 1.0]]))
    with pytest.raises(O.NotSPD):
        O.cholesky(np.zeros((3, 3)))


# --------------------------------------------------------------------------
# block updates against dense brute force (lstsq on the explicit Z)
# --------------------------------------------------------------------------

def _bruteforce_update(D, A, B, side, block, kind, opts, EA, EB):
    """Dense restatement: pick the sub-problem, build Z, solve with lstsq."""
    m, n = D.shape
    A, B, EA, EB = A.copy(), B.copy(), EA.copy(), EB.copy()
    if side == O.ROW:
        i0, i1 = O.block_range(block, opts.block_rows, m)
        if kind == O.EXACT:
            Z = O.update_z(D[i0:i1], A[i0:i1] @ B.T)
            X = np.linalg.lstsq(B, Z.T, rcond=None)[0].T       # argmin ||Z - X B^T||
            A[i0:i1] += opts.eta * (X - A[i0:i1])
        else:
            Z = O.update_z(D[i0:i1].T, B @ A[i0:i1].T)         # n x |I|
            X = np.linalg.lstsq(A[i0:i1], Z.T, rcond=None)[0].T
            EB[:] = opts.eta * (X - B) + opts.gamma * EB
            B += EB
    else:
        j0, j1 = O.block_range(block, opts.block_cols, n)
        if kind == O.EXACT:
            Z = O.update_z(D[:, j0:j1].T, B[j0:j1] @ A.T)
            X = np.linalg.lstsq(A, Z.T, rcond=None)[0].T
            B[j0:j1] += opts.eta * (X - B[j0:j1])
        else:
            Z = O.update_z(D[:, j0:j1], A @ B[j0:j1].T)
            X = np.linalg.lstsq(B[j0:j1], Z.T, rcond=None)[0].T
            EA[:] = opts.eta * (X - A) + opts.gamma * EA
            A += EA
    return A, B, EA, EB


@pytest.mark.parametrize("side", [O.ROW, O.COL])
@pytest.mark.parametrize("kind", [O.EXACT, O.STOCH])
def test_block_update_matches_dense_bruteforce(side, kind):
    S, D = _rand_sparse(13, 11, 0.3, 3)
    rng = np.random.default_rng(4)
    r = 3
    W = rng.standard_normal((13, r))
    H = rng.standard_normal((r, 11))
    opts = O.Options(block_rows=5, block_cols=4, eta=0.7, gamma=0.5)
    st = O.State(S, W, H, opts)
    st.EA[:] = 0.01 * rng.standard_normal(st.EA.shape)
    st.EB[:] = 0.01 * rng.standard_normal(st.EB.shape)
    nb = O.num_blocks(13 if side == O.ROW else 11, 5 if side == O.ROW else 4)
    for block in range(nb):                            # includes the ragged last block
        A, B, EA, EB = _bruteforce_update(D, st.A, st.B, side, block, kind, opts, st.EA, st.EB)
        st.block_update(side, block, kind)
        np.testing.assert_allclose(st.A, A, rtol=1e-10, atol=1e-11)
        np.testing.assert_allclose(st.B, B, rtol=1e-10, atol=1e-11)
        np.testing.assert_allclose(st.EA, EA, rtol=1e-10, atol=1e-11)
        np.testing.assert_allclose(st.EB, EB, rtol=1e-10, atol=1e-11)


@pytest.mark.parametrize("side", [O.ROW, O.COL])
def test_combined_update_matches_dense_bruteforce(side):
    """Combined row and column sub-sampling (Sec. 4.1, after eq. lsqA_sto):
    side ROW takes A_I to argmin_X ||Z[I, J] - X B_J^T|| with step eta and
    momentum; side COL the same for B_J against A_I on S[I, J]^T."""
    S, D = _rand_sparse(13, 11, 0.35, 6)
    rng = np.random.default_rng(7)
    r = 3
    W = rng.standard_normal((13, r))
    H = rng.standard_normal((r, 11))
    opts = O.Options(block_rows=5, block_cols=4, eta=0.7, gamma=0.5)
    st = O.State(S, W, H, opts)
    st.EA[:] = 0.01 * rng.standard_normal(st.EA.shape)
    st.EB[:] = 0.01 * rng.standard_normal(st.EB.shape)
    for I in range(O.num_blocks(13, 5)):                   # ragged last blocks included
        for J in range(O.num_blocks(11, 4)):
            i0, i1 = O.block_range(I, 5, 13)
            j0, j1 = O.block_range(J, 4, 11)
            A, B, EA, EB = st.A.copy(), st.B.copy(), st.EA.copy(), st.EB.copy()
            if side == O.ROW:
                Z = O.update_z(D[i0:i1, j0:j1], A[i0:i1] @ B[j0:j1].T)
                X = np.linalg.lstsq(B[j0:j1], Z.T, rcond=None)[0].T
                EA[i0:i1] = opts.eta * (X - A[i0:i1]) + opts.gamma * EA[i0:i1]
                A[i0:i1] += EA[i0:i1]
            else:
                Z = O.update_z(D[i0:i1, j0:j1].T, B[j0:j1] @ A[i0:i1].T)
                X = np.linalg.lstsq(A[i0:i1], Z.T, rcond=None)[0].T
                EB[j0:j1] = opts.eta * (X - B[j0:j1]) + opts.gamma * EB[j0:j1]
                B[j0:j1] += EB[j0:j1]
            st.block_update_combined(side, I, J)
            np.testing.assert_allclose(st.A, A, rtol=1e-10, atol=1e-11)
            np.testing.assert_allclose(st.B, B, rtol=1e-10, atol=1e-11)
            np.testing.assert_allclose(st.EA, EA, rtol=1e-10, atol=1e-11)
            np.testing.assert_allclose(st.EB, EB, rtol=1e-10, atol=1e-11)


def test_combined_update_reduces_to_the_other_steps():
    """A combined step whose row block is every row is the stochastic column
    step (eq. lsqA_sto); one whose column block is every column, with eta = 1
    and no momentum, is the parallel row step (eq. lsqA_par)."""
    S, _ = _rand_sparse(20, 15, 0.25, 8)
    W, H = WL.init_factors(20, 15, 3, 1)
    for eta, gamma in ((0.8, 0.6), (1.0, 0.0)):
        a = O.State(S, W, H, O.Options(block_rows=20, block_cols=6, eta=eta, gamma=gamma))
        b = O.State(S, W, H, O.Options(block_rows=20, block_cols=6, eta=eta, gamma=gamma))
        a.block_update_combined(O.ROW, 0, 1)
        b.block_update(O.COL, 1, O.STOCH)
        np.testing.assert_allclose(a.A, b.A, rtol=1e-12, atol=1e-13)
        np.testing.assert_allclose(a.EA, b.EA, rtol=1e-12, atol=1e-13)
    a = O.State(S, W, H, O.Options(block_rows=7, block_cols=15, eta=1.0, gamma=0.0))
    b = O.State(S, W, H, O.Options(block_rows=7, block_cols=15, eta=1.0, gamma=0.0))
    a.block_update_combined(O.ROW, 2, 0)
    b.block_update(O.ROW, 2, O.EXACT)
    np.testing.assert_allclose(a.A, b.A, rtol=1e-12, atol=1e-13)


def test_stochastic_full_batch_equals_parallel():
    """A mini-batch covering every column with eta=1, gamma=0 is plain ALS (eq. lsqA)."""
    S, _ = _rand_sparse(20, 15, 0.25, 5)
    W, H = WL.init_factors(20, 15, 4, 0)
    a = O.State(S, W, H, O.Options(block_rows=20, block_cols=15, eta=1.0, gamma=0.0))
    b = O.State(S, W, H, O.Options(block_rows=20, block_cols=15, eta=1.0, gamma=0.0))
    a.block_update(O.COL, 0, O.STOCH)
    b.block_update(O.ROW, 0, O.EXACT)
    np.testing.assert_allclose(a.A, b.A, rtol=1e-12, atol=1e-13)


# --------------------------------------------------------------------------
# properties the paper proves
# --------------------------------------------------------------------------

def test_exact_halfsteps_never_increase_objective():
    """Sec. 3.2: each alternating minimisation step lowers ||Z - L||."""
    S, _, _, _ = WL.planted(60, 50, 4, tau=0.5, seed=1)
    W, H = WL.init_factors(60, 50, 4, 1)
    st = O.State(S, W, H, O.Options(block_rows=16, block_cols=16, schedule=O.EXACT))
    prev = st.loss()["obj"]
    for _ in range(3):
        for side, block, kind in st.sweep_steps():
            st.block_update(side, block, kind)
            cur = st.loss()["obj"]
            assert cur <= prev * (1 + 1e-12) + 1e-15
            prev = cur
        st.sweep_index += 1


def test_exact_row_blocks_are_order_independent():
    """Sec. 4.1: row blocks of A are independent given B."""
    S, _, _, _ = WL.planted(50, 40, 3, tau=0.3, seed=2)
    W, H = WL.init_factors(50, 40, 3, 2)
    a = O.State(S, W, H, O.Options(block_rows=8, block_cols=8, schedule=O.EXACT))
    b = O.State(S, W, H, O.Options(block_rows=8, block_cols=8, schedule=O.EXACT))
    K = O.num_blocks(50, 8)
    for blk in range(K):
        a.block_update(O.ROW, blk, O.EXACT)
    for blk in O.block_permutation(9, 3, 0, K):
        b.block_update(O.ROW, blk, O.EXACT)
    assert np.array_equal(a.A, b.A)


def _planted_exact(m, n, d, tau, seed):
    """S = max(0, U V^T - tau) in fp64 and its rank-(d+1) completion [U, 1][V, -tau]^T."""
    S, U, V, _ = WL.planted(m, n, d, tau=tau, seed=seed, dtype=np.float64)
    W0 = np.hstack([U, np.ones((m, 1))])
    H0 = np.hstack([V, -tau * np.ones((n, 1))]).T
    return S, W0, H0


@pytest.mark.parametrize("schedule", [O.EXACT, O.STOCH])
def test_planted_completion_is_zero_loss_fixed_point(schedule):
    """Prop. 1 (Sec. 2.1): a thresholded rank-d matrix has a rank-(d+1) completion."""
    S, W0, H0 = _planted_exact(70, 50, 4, 0.5, 3)
    # blocks of 16 rows and 10 columns: every block (the ragged last one too)
    # has at least r = 5 rows, so each block Gram matrix is nonsingular
    st = O.State(S, W0, H0, O.Options(block_rows=16, block_cols=10, schedule=schedule,
                                      eta=1.0, gamma=0.9))
    l0 = st.loss()
    assert l0["obj"] < 1e-14 and l0["rmse"] < 1e-14 and l0["wjd"] < 1e-14
    st.sweep()
    np.testing.assert_allclose(st.A, W0, atol=1e-11)
    np.testing.assert_allclose(st.B, H0.T, atol=1e-11)
    assert st.loss()["obj"] < 1e-12


def _omega_factors(n):
    th = 2 * np.pi * np.arange(n) / n
    c = np.cos(2 * np.pi / n)
    W = np.stack([np.cos(th), np.sin(th), -c * np.ones(n)], 1) / (1 - c)
    H = np.stack([np.cos(th), np.sin(th), np.ones(n)], 1).T
    return W, H


def test_identity_has_rank3_completion_omega():
    """Corollary 'ident' (eq. Omega): I_n = max(0, Omega), rank(Omega) <= 3."""
    n = 64
    W, H = _omega_factors(n)
    Om = W @ H
    i, j = np.meshgrid(np.arange(n), np.arange(n), indexing="ij")
    c = np.cos(2 * np.pi / n)
    np.testing.assert_allclose(Om, (np.cos(2 * np.pi * (i - j) / n) - c) / (1 - c), atol=1e-10)
    np.testing.assert_allclose(np.maximum(0, Om), np.eye(n), atol=1e-9)
    # Corollary 'nuclear': ||Omega||_* = n (1 + |cos phi|) / (1 - cos phi)
    nuc = np.linalg.svd(Om, compute_uv=False).sum()
    assert nuc == pytest.approx(n * (1 + abs(c)) / (1 - c), rel=1e-10)
    S = WL.identity(n, dtype=np.float64)
    st = O.State(S, W, H, O.Options(block_rows=16, block_cols=16, eta=1.0, gamma=0.9))
    assert st.loss()["obj"] < 1e-9
    st.sweep()
    assert st.loss()["obj"] < 1e-8
    np.testing.assert_allclose(st.A @ st.B.T, Om, atol=1e-7)


def _fixed_point_checks(D, W, H, block, stoch_block=None):
    """The oracle at a zero-loss point of S = D: zero objective, and an exact
    and a stochastic sweep (eta = 1) leave the model L = W H unchanged.  The
    stochastic blocks must span the factor's column space (their Gram
    matrices must be invertible)."""
    S = WL.csr_from_dense(D, dtype=np.float64)
    L0 = W @ H
    for sched in (O.EXACT, O.STOCH):
        b = block if sched == O.EXACT or stoch_block is None else stoch_block
        st = O.State(S, W, H, O.Options(block_rows=b, block_cols=b, schedule=sched, eta=1.0,
                                        gamma=0.9 if sched == O.STOCH else 0.0))
        assert st.loss()["obj"] < 1e-12
        st.sweep()
        assert st.loss()["obj"] < 1e-10
        np.testing.assert_allclose(st.A @ st.B.T, L0, atol=1e-9)


@pytest.mark.parametrize("delta", [0.25, 0.5])
def test_ring_graph_rank3_completion_is_fixed(delta):
    """Prop. 'ring' (eqs. ring, ringvecs, tau, r2): with unit-spaced points on a
    circle of radius r and the threshold tau, the thresholded similarities
    reproduce the ring matrix (1 on the diagonal, delta between neighbours,
    0 elsewhere) as max(0, L) with rank(L) = 3; the oracle must treat that
    point as an exact, fixed completion."""
    n = 40
    phi = 2 * np.pi / n
    tau = (np.cos(phi) - delta) / (1 - delta)
    r2 = (1 - delta) / (1 - np.cos(phi))
    th = phi * np.arange(n)
    r = np.sqrt(r2)
    W = np.stack([r * np.cos(th), r * np.sin(th), -tau * r2 * np.ones(n)], 1)
    H = np.stack([r * np.cos(th), r * np.sin(th), np.ones(n)], 1).T
    i, j = np.meshgrid(np.arange(n), np.arange(n), indexing="ij")
    d = np.abs(i - j)
    D = np.where(d == 0, 1.0, np.where((d == 1) | (d == n - 1), delta, 0.0))
    np.testing.assert_allclose(np.maximum(0, W @ H), D, atol=1e-12)
    assert np.linalg.matrix_rank(W @ H) == 3
    _fixed_point_checks(D, W, H, 8)


def test_hypercube_rank_d_plus_1_completion_is_fixed():
    """Prop. 'hypercube' (eq. hypercube): with alpha_i = r v_i on the vertices
    v_i of the d-cube, r^2 = (1 - delta) / 2 and tau = 1 - 2 / (d (1 - delta)),
    max(0, L) is 1 on the diagonal, delta between vertices at distance 2 and 0
    otherwise, with rank(L) <= d + 1."""
    dim, delta = 5, 0.1
    V = np.array([[1.0 if (k >> b) & 1 else -1.0 for b in range(dim)] for k in range(2 ** dim)])
    r2 = (1 - delta) / 2
    tau = 1 - 2 / (dim * (1 - delta))
    W = np.hstack([np.sqrt(r2) * V, -tau * r2 * dim * np.ones((2 ** dim, 1))])
    H = np.hstack([np.sqrt(r2) * V, np.ones((2 ** dim, 1))])
    dist2 = ((V[:, None, :] - V[None, :, :]) ** 2).sum(-1)
    D = np.where(dist2 == 0, 1.0, np.where(dist2 == 4, delta, 0.0))
    np.testing.assert_allclose(np.maximum(0, W @ H.T), D, atol=1e-12)
    assert np.linalg.matrix_rank(W @ H.T) == dim + 1
    # a block of 8 or 16 consecutive vertices fixes the top coordinates, so its
    # rows of [r v, 1] are rank deficient: stochastic blocks take the whole cube
    _fixed_point_checks(D, W, H.T, 8, stoch_block=2 ** dim)


def test_loss_of_all_zero_model_is_one():
    """Sec. 3.1: RMSE(S, 0) = WJD(S, 0) = 1; with L = 0, Z = S so the objective is 1 too."""
    S, _ = _rand_sparse(20, 30, 0.2, 6)
    l = O.loss(O.Sparse.from_csr(S), np.zeros((20, 3)), np.zeros((30, 3)))
    assert l["obj"] == pytest.approx(1.0) and l["rmse"] == pytest.approx(1.0)
    assert l["wjd"] == pytest.approx(1.0)


def test_loss_definitions_bruteforce_and_lipschitz():
    """eq. SLloss equals ||Z - L||^2; eq. RMSE / WJD written densely; obj >= RMSE (Prop. 'Lipschitz')."""
    S, D = _rand_sparse(17, 23, 0.3, 7)
    rng = np.random.default_rng(8)
    A = rng.standard_normal((17, 4))
    B = rng.standard_normal((23, 4))
    L = A @ B.T
    sl = np.sum(np.where(D == 0, np.maximum(0, L) ** 2, 0)) + np.sum(np.where(D > 0, (D - L) ** 2, 0))
    Shat = np.maximum(0, L)
    sf = np.sqrt(np.sum(D ** 2))
    l = O.loss(O.Sparse.from_csr(S), A, B)
    assert l["obj"] == pytest.approx(math.sqrt(sl) / sf, rel=1e-12)
    assert l["rmse"] == pytest.approx(np.sqrt(np.sum((D - Shat) ** 2)) / sf, rel=1e-12)
    assert l["wjd"] == pytest.approx(1 - np.minimum(D, Shat).sum() / np.maximum(D, Shat).sum(), rel=1e-12)
    assert l["obj"] >= l["rmse"]


def test_momentum_is_heavy_ball():
    """Momentum reading: M_{t+1} - M_t = U_t + gamma (M_t - M_{t-1})."""
    S, _ = _rand_sparse(30, 24, 0.2, 9)
    W, H = WL.init_factors(30, 24, 3, 3)
    opts = O.Options(block_rows=8, block_cols=8, eta=0.8, gamma=0.6)
    st = O.State(S, W, H, opts)
    prev = st.A.copy()
    for t, blk in enumerate([0, 2, 1]):
        M = st.A.copy()
        R, G = st.block_terms(O.COL, blk, O.STOCH)
        U = opts.eta * (np.linalg.solve(G, R.T).T - M)
        st.block_update(O.COL, blk, O.STOCH)
        np.testing.assert_allclose(st.A - M, U + opts.gamma * (M - prev), rtol=1e-9, atol=1e-12)
        prev = M


def test_stochastic_sweep_decreases_loss_on_planted():
    S, _, _, _ = WL.planted(200, 160, 4, tau=0.5, seed=4)
    W, H = WL.init_factors(200, 160, 5, 4)
    st = O.State(S, W, H, O.Options(block_rows=40, block_cols=40, eta=1.0, gamma=0.5))
    l0 = st.loss()["obj"]
    for _ in range(10):
        st.sweep()
    assert st.loss()["obj"] < 0.5 * l0


def test_range_search_set_hand_examples():
    """Eq. range-search on pairs worked out by hand: L > 0 exactly when the
    normalised rows are less than sqrt(2) apart; an orthogonal pair sits at
    squared distance exactly 2 (L = 0: not in Omega); a zero row is in no
    pair."""
    A = np.array([[3.0, 4.0, 0.0], [1.0, 0.0, 0.0], [2.0, 0.0, 0.0], [0.0, 0.0, 0.0]])
    B = np.array([[4.0, 3.0, 0.0], [0.0, 0.0, 5.0], [-1.0, -1.0, 0.0]])
    # (0,0): L = 24, |a^ - b^|^2 = 0.08; (1,1): L = 0, distance^2 = 2; (2,2): L = -2,
    # distance^2 = 2 + sqrt(2); row 3 is zero
    want = np.array([[1, 0, 0], [1, 0, 0], [1, 0, 0], [0, 0, 0]], dtype=bool)
    np.testing.assert_array_equal(O.range_search_set(A, B), want)
    np.testing.assert_array_equal(O.positive_set(A, B), want)


def test_range_search_set_equals_positive_set():
    """Eq. nonzeros and eq. range-search define the same set (Sec. 4.3), on
    random factors with zero rows and with rows of very different lengths."""
    rng = np.random.default_rng(4)
    A = rng.standard_normal((30, 5)) * rng.uniform(0.01, 100.0, (30, 1))
    B = rng.standard_normal((40, 5)) * rng.uniform(0.01, 100.0, (40, 1))
    A[[3, 17]] = 0.0
    B[[0, 25, 39]] = 0.0
    got = O.range_search_set(A, B)
    want = np.zeros((30, 40), dtype=bool)
    for i in range(30):
        for j in range(40):
            want[i, j] = sum(A[i, k] * B[j, k] for k in range(5)) > 0
    np.testing.assert_array_equal(got, want)
    np.testing.assert_array_equal(O.positive_set(A, B), want)
    assert 0 < want.sum() < want.size
