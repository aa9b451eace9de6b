"""Pins of the oracle's cell embedding (Sec. 5.3, eqs. Lsvd and embed) and
its one-nearest-neighbour search, against closed forms, an independent
route through matrix square roots, invariances and brute force."""
import numpy as np

import oracle as O


def _orthonormal(rng, n, r):
    Q, _ = np.linalg.qr(rng.standard_normal((n, r)))
    return Q


def test_embedding_closed_form():
    """A = P diag(a), B = Q diag(b) with orthonormal P, Q: L = P diag(ab) Q^T
    is its own SVD (after sorting), so xi_i ~ [p_i, q_i] diag(sqrt(ab))."""
    rng = np.random.default_rng(1)
    n, r = 40, 5
    P, Q = _orthonormal(rng, n, r), _orthonormal(rng, n, r)
    a = np.array([3.0, 1.0, 2.0, 0.5, 4.0])
    b = np.array([1.0, 2.0, 0.25, 3.0, 0.5])
    xi, s = O.embed.embedding(P * a, Q * b)
    order = np.argsort(-(a * b))
    np.testing.assert_allclose(s, (a * b)[order], rtol=1e-12)
    root = np.sqrt((a * b)[order])
    want = np.concatenate([P[:, order] * root, Q[:, order] * root], axis=1)
    want /= np.linalg.norm(want, axis=1, keepdims=True)
    # columns are defined up to a common sign per singular triple: compare Gram matrices
    np.testing.assert_allclose(xi @ xi.T, want @ want.T, atol=1e-12)
    np.testing.assert_allclose(np.linalg.norm(xi, axis=1), 1.0, rtol=1e-13)


def _psd_root(M):
    w, V = np.linalg.eigh((M + M.T) / 2)
    return (V * np.sqrt(np.maximum(w, 0.0))) @ V.T


def test_embedding_inner_products_through_matrix_roots():
    """xi_i . xi_j n_i n_j = ((L L^T)^{1/2} + (L^T L)^{1/2})_ij, since
    U Sigma U^T and V Sigma V^T are the square roots of L L^T and L^T L;
    computed here by eigendecompositions, not by the SVD.  A non-symmetric
    L tells the two halves (u and v) apart."""
    rng = np.random.default_rng(2)
    n, r = 30, 4
    A = rng.standard_normal((n, r))
    B = rng.standard_normal((n, r)) * np.array([3.0, 1.0, 0.3, 2.0])
    L = A @ B.T
    K = _psd_root(L @ L.T) + _psd_root(L.T @ L)
    d = np.sqrt(np.diag(K))
    xi, _ = O.embed.embedding(A, B)
    # (the square roots of the rank-r products carry ~1e-7 from their n - r
    # zero eigenvalues)
    np.testing.assert_allclose(xi @ xi.T, K / np.outer(d, d), atol=1e-6)
    # the first half alone is u_i Sigma^{1/2}: swapping u and v fails here
    half = xi[:, :r] * d[:, None]
    np.testing.assert_allclose(half @ half.T, _psd_root(L @ L.T), atol=1e-6)


def test_embedding_is_invariant_to_the_factor_basis():
    rng = np.random.default_rng(3)
    n, r = 25, 3
    A = rng.standard_normal((n, r))
    B = rng.standard_normal((n, r))
    M = rng.standard_normal((r, r)) + 3 * np.eye(r)
    xi1, s1 = O.embed.embedding(A, B)
    xi2, s2 = O.embed.embedding(A @ M, B @ np.linalg.inv(M).T)
    np.testing.assert_allclose(s1, s2, rtol=1e-10)
    np.testing.assert_allclose(xi1 @ xi1.T, xi2 @ xi2.T, atol=1e-10)


def test_nearest_neighbors_brute_force_and_ties():
    rng = np.random.default_rng(4)
    X = rng.standard_normal((60, 5))
    X[17] = X[3]                      # a duplicate: 3 and 17 are each other's nearest
    X[40] = X[3]                      # ... and 40 ties with them: the smaller index wins
    nn, best = O.embed.nearest_neighbors(X)
    for i in range(60):
        sims = [(X[i] @ X[j], -j) for j in range(60) if j != i]
        v, mj = max(sims)
        assert nn[i] == -mj and abs(best[i] - v) < 1e-12
    assert nn[3] == 17 and nn[17] == 3 and nn[40] == 3


def test_one_nn_errors_counts_label_disagreements():
    nn = np.array([1, 0, 3, 2, 0])
    labels = np.array([7, 7, 5, 6, 7])
    assert O.embed.one_nn_errors(nn, labels) == 2     # cells 2 and 3
