"""fp64 CPU oracle of the cell embedding and the held-out one-nearest-neighbour
error of Sec. 5.3 -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU legs may
import this module; the CUDA library shares no code with it.

* Eq. Lsvd: the rank-r model L = A B^T (A = W, B = H^T of a square S) has the
  singular value decomposition L = U Sigma V^T; here L is formed explicitly
  in fp64 and decomposed by the library SVD, keeping its r leading triples.
* Eq. embed: cell i is the unit vector xi_i proportional to
  [u_i, v_i] Sigma^{1/2} (u_i, v_i the i-th rows of U and V).
* 1-NN error: for every labelled cell, the nearest other cell in the
  embedding (the largest inner product xi_i . xi_j, j != i: for unit vectors
  that is the smallest Euclidean distance) and whether its label differs;
  the error rate is the fraction that differ.  Ties go to the smallest j.
"""
from __future__ import annotations

import numpy as np


def embedding(A: np.ndarray, B: np.ndarray) -> tuple[np.ndarray, np.ndarray]:
    """(xi, sigma): the n x 2r unit rows of eq. embed and the r leading
    singular values of L = A B^T (eq. Lsvd), descending."""
    A = np.asarray(A, np.float64)
    B = np.asarray(B, np.float64)
    if A.shape[0] != B.shape[0]:
        raise ValueError("the embedding of cells needs a square matrix (rows and columns are the same cells)")
    r = A.shape[1]
    L = A @ B.T
    U, s, Vt = np.linalg.svd(L)
    U, s, V = U[:, :r], s[:r], Vt[:r].T
    root = np.sqrt(s)
    xi = np.concatenate([U * root, V * root], axis=1)
    norms = np.sqrt((xi * xi).sum(axis=1, keepdims=True))
    xi = xi / np.where(norms > 0, norms, 1.0)
    return xi, s


def nearest_neighbors(X: np.ndarray) -> tuple[np.ndarray, np.ndarray]:
    """(nn, best): for every row i of X, the row j != i with the largest
    inner product X_i . X_j (ties: the smallest j) and that inner product."""
    X = np.asarray(X, np.float64)
    n = X.shape[0]
    nn = np.full(n, -1, dtype=np.int64)
    best = np.full(n, -np.inf)
    for i0 in range(0, n, 1024):
        P = X[i0:i0 + 1024] @ X.T
        for k in range(P.shape[0]):
            P[k, i0 + k] = -np.inf
        nn[i0:i0 + 1024] = np.argmax(P, axis=1)   # the first maximum: the smallest j
        best[i0:i0 + 1024] = P[np.arange(P.shape[0]), nn[i0:i0 + 1024]]
    return nn, best


def one_nn_errors(nn: np.ndarray, labels: np.ndarray) -> int:
    """Cells whose nearest neighbour carries a different label."""
    nn = np.asarray(nn)
    labels = np.asarray(labels)
    return int(np.sum(labels[nn] != labels))
