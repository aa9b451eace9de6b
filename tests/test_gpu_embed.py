"""Cell embedding and held-out 1-NN search (Sec. 5.3, eqs. Lsvd and embed).

* nmd_embed against the oracle's embedding (the library SVD of the explicit
  L = W H): the singular values, and the Gram matrix xi xi^T, which does not
  depend on the signs of the singular triples or on rotations within equal
  singular values ((L L^T)^{1/2} + (L^T L)^{1/2}, normalised);
* nmd_nearest_neighbors against brute force in fp64 on the same fp32 points:
  the neighbour is another point whose inner product is the largest within
  1e-5 (the accuracy of three bf16 pieces per coordinate), equal to the
  brute-force neighbour wherever that one leads the runner-up by more than
  1e-4; the returned inner product is that of the returned pair; the label
  disagreements are counted exactly;
* the whole path on a block-structured graph: embedding after a few sweeps,
  1-NN error of the community labels well below chance."""
import numpy as np
import pytest

import oracle as O
from gpu_common import require_gpu
from paper_2608_21607_gb300 import nmd as N
from paper_2608_21607_gb300 import workloads as WL

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def gpu():
    return require_gpu()


@pytest.mark.parametrize("r", [3, 8, 16, 64, 100, 128])
def test_embedding_matches_oracle(r):
    import torch
    n = 1500 if r <= 64 else 2000
    S = WL.connectome(n, seed=r)
    W, H = WL.init_factors(n, n, r, r)
    H = H * np.linspace(2.0, 0.2, r, dtype=np.float32)[:, None]   # spread the spectrum
    sol = N.Solver(S, r, block_rows=512, block_cols=512)
    sol.set_factors(W, H)
    xi, sigma = sol.embed()
    torch.cuda.synchronize()
    xi, sigma = xi.cpu().numpy().astype(np.float64), sigma.cpu().numpy()
    xo, so = O.embed.embedding(W, H.T)
    np.testing.assert_allclose(sigma, so, rtol=1e-4)
    np.testing.assert_allclose(np.linalg.norm(xi, axis=1), 1.0, atol=1e-5)
    rows = np.random.default_rng(r).choice(n, 400, replace=False)
    G, Go = xi[rows] @ xi[rows].T, xo[rows] @ xo[rows].T
    assert np.abs(G - Go).max() <= 2e-4, np.abs(G - Go).max()
    # each half separately: u_i Sigma^{1/2} u_j^T and v_i Sigma^{1/2} v_j^T
    for half in (slice(0, r), slice(r, 2 * r)):
        Gh, Goh = xi[rows][:, half] @ xi[rows][:, half].T, xo[rows][:, half] @ xo[rows][:, half].T
        assert np.abs(Gh - Goh).max() <= 2e-4


def test_embedding_rejects_unsupported_shapes():
    S, _, _, _ = WL.planted(300, 200, 4, tau=0.5, seed=0)
    sol = N.Solver(S, 4, block_rows=100, block_cols=100)
    W, H = WL.init_factors(300, 200, 4, 0)
    sol.set_factors(W, H)
    with pytest.raises(N.NmdError) as e:
        sol.embed()                                   # not square
    assert e.value.status == N.NMD_ERR_INVALID


def _check_nn(x, nn, best, tie_margin=1e-4, tol=1e-5):
    X = x.astype(np.float64)
    no, bo = O.embed.nearest_neighbors(X)
    n = X.shape[0]
    assert np.all(nn != np.arange(n)) and np.all((nn >= 0) & (nn < n))
    got = np.einsum("ij,ij->i", X, X[nn])
    scale = np.linalg.norm(X, axis=1) * np.linalg.norm(X[nn], axis=1)
    assert np.all(np.abs(best - got) <= tol * np.maximum(scale, 1e-30)), np.abs(best - got).max()
    assert np.all(got >= bo - 2 * tol * np.maximum(scale, 1e-30))
    # where the brute-force maximum leads the runner-up clearly, the same neighbour
    clear = []
    for i0 in range(0, n, 1024):
        P = X[i0:i0 + 1024] @ X.T
        for k in range(P.shape[0]):
            P[k, i0 + k] = -np.inf
        top2 = np.sort(P, axis=1)[:, -2:]
        clear.append(top2[:, 1] - top2[:, 0] > tie_margin)
    clear = np.concatenate(clear)
    assert np.array_equal(nn[clear], no[clear])
    return no


@pytest.mark.parametrize("n,d", [(2, 1), (300, 16), (3000, 40), (2177, 128), (1500, 200), (1000, 256)])
def test_nearest_neighbors_match_brute_force(n, d):
    import torch
    rng = np.random.default_rng(n + d)
    x = rng.standard_normal((n, d)).astype(np.float32)
    x /= np.linalg.norm(x, axis=1, keepdims=True)
    labels = rng.integers(0, 5, n).astype(np.int32)
    nn, best, errors = N.nearest_neighbors(torch.from_numpy(x).cuda(), labels)
    nn, best = nn.cpu().numpy().astype(np.int64), best.cpu().numpy().astype(np.float64)
    _check_nn(x, nn, best)
    assert errors == int(np.sum(labels[nn] != labels))


def test_nearest_neighbors_exact_duplicates_take_the_smaller_index():
    import torch
    rng = np.random.default_rng(7)
    x = rng.standard_normal((700, 32)).astype(np.float32)
    x[20] *= 3.0                         # long enough to dominate every other inner product
    x[500] = x[20]
    x[650] = x[20]
    x[300] = 3.0 * x[20]                 # the largest inner product with 20's copies
    nn, best, _ = N.nearest_neighbors(torch.from_numpy(x).cuda())
    nn = nn.cpu().numpy()
    assert nn[20] == 300 and nn[500] == 300 and nn[650] == 300
    assert nn[300] == 20                 # three equal candidates: the smallest index


def test_embedding_and_1nn_on_communities():
    """A block-structured graph of 8 communities fitted from a random start:
    after a few sweeps the 1-NN error of the community labels in the
    embedding is far below chance (7/8)."""
    import torch
    n, r, C = 4096, 16, 8
    S = WL.communities(n, n, C, 30.0, seed=3)
    labels = WL.community_of(n, C).astype(np.int32)
    W, H = WL.init_factors(n, n, r, 3)
    sol = N.Solver(S, r, block_rows=1024, block_cols=1024, eta=0.5, gamma=0.9)
    sol.set_factors(W, H)
    for _ in range(5):
        sol.sweep()
    xi, _ = sol.embed()
    nn, best, errors = N.nearest_neighbors(xi, labels)
    torch.cuda.synchronize()
    nn = nn.cpu().numpy().astype(np.int64)
    assert errors == int(np.sum(labels[nn] != labels))
    assert errors / n < 0.5, errors / n   # (the fp64 oracle's trajectory gives 0.19)
    _check_nn(xi.cpu().numpy(), nn, best.cpu().numpy().astype(np.float64))
