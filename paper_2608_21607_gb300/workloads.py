"""Seeded synthetic inputs for the SALSA block sweep.

This module only *generates* inputs: the sparse nonnegative matrix S (CSR) and
the initial factors W (m x r) and H (r x n).  It contains none of the solver's
arithmetic, so the fp64 oracle and the CUDA path can both consume it without
sharing any part of the method.

The paper's datasets (MNIST similarities, the FlyWire connectome, Wikipedia
bigrams; Sec. 2.5, Table 1) are not available, so every workload is a seeded
stand-in with the structure the paper describes:

* ``planted``     -- S = max(0, U V^T - tau), a thresholded low-rank matrix
                     (Def. 2 / Prop. 1 of Sec. 2.1: it admits an exact
                     completion of rank d+1).
* ``identity``    -- S = I_n (Corollary "ident", Sec. 2.2: rank-3 completion).
* ``connectome``  -- a directed graph with power-law out-degree (exponent 2.2,
                     mean 20) and integer log-normal synapse counts, shaped
                     like the connectome of Table 1 (139k x 139k, sparse).

All random draws come from numpy's PCG64 with explicit seeds, so both sides of
every parity test see bit-identical inputs.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Optional

import numpy as np

__all__ = [
    "CSR", "Workload", "csr_from_dense", "planted", "identity", "connectome",
    "init_factors", "workload", "WORKLOADS",
]


@dataclasses.dataclass
class CSR:
    """Compressed sparse rows: ``row_ptr`` (int64, m+1), ``col_idx`` (int32,
    strictly increasing within a row), ``vals`` (float32 or float64, > 0)."""
    m: int
    n: int
    row_ptr: np.ndarray
    col_idx: np.ndarray
    vals: np.ndarray

    @property
    def nnz(self) -> int:
        return int(self.row_ptr[-1])

    def todense(self, dtype=np.float64) -> np.ndarray:
        d = np.zeros((self.m, self.n), dtype=dtype)
        rows = np.repeat(np.arange(self.m), np.diff(self.row_ptr))
        d[rows, self.col_idx] = self.vals
        return d


@dataclasses.dataclass
class Workload:
    name: str
    S: CSR
    r: int
    W0: np.ndarray            # m x r, float32
    H0: np.ndarray            # r x n, float32
    block_rows: int
    block_cols: int
    schedule: str             # "exact" | "stoch"
    sweeps: int
    eta: float
    gamma: float
    seed: int
    info: dict

    @property
    def m(self) -> int:
        return self.S.m

    @property
    def n(self) -> int:
        return self.S.n


def csr_from_dense(D: np.ndarray, dtype=np.float32) -> CSR:
    """CSR of the strictly positive entries of a dense array."""
    m, n = D.shape
    mask = D > 0
    counts = mask.sum(axis=1)
    row_ptr = np.zeros(m + 1, dtype=np.int64)
    np.cumsum(counts, out=row_ptr[1:])
    rows, cols = np.nonzero(mask)
    return CSR(m, n, row_ptr, cols.astype(np.int32), D[rows, cols].astype(dtype))


def init_factors(m: int, n: int, r: int, seed: int, sigma: float = 0.1, signs: str = "normal"):
    """W (m x r) and H (r x n) iid N(0, sigma^2), float32.

    signs="paper": the sign-structured start of Sec. 4.3, W = |N(0, sigma^2)|
    and H = -|N(0, sigma^2)|, so that W H < 0 everywhere at the start (the
    rectified matrix is empty)."""
    rng = np.random.default_rng([seed, 0xF0C7])
    W = (sigma * rng.standard_normal((m, r))).astype(np.float32)
    H = (sigma * rng.standard_normal((r, n))).astype(np.float32)
    if signs == "paper":
        W, H = np.abs(W), -np.abs(H)
    elif signs != "normal":
        raise ValueError("signs must be 'normal' or 'paper'")
    return W, H


def _csr_from_rows(m, n, row_cols, row_vals, dtype) -> CSR:
    counts = np.fromiter((len(c) for c in row_cols), dtype=np.int64, count=m)
    row_ptr = np.zeros(m + 1, dtype=np.int64)
    np.cumsum(counts, out=row_ptr[1:])
    col_idx = np.concatenate(row_cols).astype(np.int32) if m else np.zeros(0, np.int32)
    vals = np.concatenate(row_vals).astype(dtype) if m else np.zeros(0, dtype)
    return CSR(m, n, row_ptr, col_idx, vals)


def planted(m: int = 600, n: int = 400, d: int = 4, tau: Optional[float] = 0.5,
            density: Optional[float] = None, noise: float = 0.0, seed: int = 0,
            dtype=np.float32, chunk: int = 2048):
    """S = max(0, U V^T - tau) with U (m x d), V (n x d) iid N(0,1).

    If ``density`` is given, tau is the empirical (1-density) quantile of
    U_i . V_j over 10^6 seeded (i, j) pairs.  If ``noise`` > 0 every positive
    entry is multiplied by (1 + noise * N(0,1)).  Returns (S, U, V, tau).
    The product is formed in fp64 so that the support does not depend on the
    host's BLAS.
    """
    rng = np.random.default_rng([seed, 0x5EED])
    U = rng.standard_normal((m, d))
    V = rng.standard_normal((n, d))
    if density is not None:
        k = 1_000_000
        ii = rng.integers(0, m, size=k)
        jj = rng.integers(0, n, size=k)
        samp = np.einsum("kd,kd->k", U[ii], V[jj])
        tau = float(np.quantile(samp, 1.0 - density))
    rows_cols, rows_vals = [], []
    for r0 in range(0, m, chunk):
        L = U[r0:r0 + chunk] @ V.T - tau
        for row in L:
            c = np.nonzero(row > 0)[0]
            rows_cols.append(c)
            rows_vals.append(row[c])
    S = _csr_from_rows(m, n, rows_cols, rows_vals, np.float64)
    if noise > 0:
        nrng = np.random.default_rng([seed, 0x0015E])
        S.vals = S.vals * (1.0 + noise * nrng.standard_normal(S.nnz))
        S.vals = np.maximum(S.vals, np.finfo(np.float32).tiny)
    S.vals = S.vals.astype(dtype)
    return S, U, V, tau


def community_of(N: int, clusters: int, run: Optional[int] = None) -> np.ndarray:
    """Community of each of N indices: contiguous ranges (run None), or runs
    of `run` consecutive indices taking the communities in turn."""
    if run is None:
        return (np.arange(N) * clusters) // N
    return (np.arange(N) // run) % clusters


def community_factors(m: int, n: int, r: int, clusters: int, noise: float = 0.01, neg: float = 0.6,
                      seed: int = 0, run: Optional[int] = None):
    """W (m x r) and H (r x n), float32, whose rows fall into `clusters` tight
    groups of directions (communities by community_of): row i of W points
    along e_c of its community c, column j of H along 2 e_d - neg (the
    all-ones vector on the first `clusters` coordinates) of its community d,
    each with iid N(0, noise^2) added and a length drawn from U(0.5, 2).
    W_i . H_j is about (2 - neg) times the lengths within a community and
    about -neg times them across: the rectified product max(0, W H) is block
    diagonal up to the ordering.  Needs r >= clusters.  Also returns the
    communities of the rows of W and of the columns of H."""
    if r < clusters:
        raise ValueError("r must be at least the number of communities")
    rng = np.random.default_rng([seed, 0xC0DE])
    cw = community_of(m, clusters, run)
    ch = community_of(n, clusters, run)
    W = np.zeros((m, r))
    W[np.arange(m), cw] = 1.0
    H = np.zeros((n, r))
    H[:, :clusters] = -neg
    H[np.arange(n), ch] += 2.0
    W += noise * rng.standard_normal((m, r))
    H += noise * rng.standard_normal((n, r))
    W *= rng.uniform(0.5, 2.0, (m, 1))
    H *= rng.uniform(0.5, 2.0, (n, 1))
    return W.astype(np.float32), np.ascontiguousarray(H.T).astype(np.float32), cw, ch


def communities(m: int, n: int, clusters: int, mean_degree: float, seed: int = 0, run: Optional[int] = None,
                dtype=np.float32) -> CSR:
    """A stochastic block model: row i has Poisson(mean_degree) entries (at
    most the size of its community), at columns drawn uniformly without
    replacement from the columns of its own community (community_of), with
    values ceil(exp(1 + N(0, 1))); no entry joins two communities."""
    rng = np.random.default_rng([seed, 0x5B3])
    cw = community_of(m, clusters, run)
    ch = community_of(n, clusters, run)
    members = [np.nonzero(ch == c)[0] for c in range(clusters)]
    rows_cols, rows_vals = [], []
    for i in range(m):
        cols = members[cw[i]]
        k = min(len(cols), rng.poisson(mean_degree))
        c = np.sort(rng.choice(cols, size=k, replace=False)) if k else np.zeros(0, np.int64)
        rows_cols.append(c)
        rows_vals.append(np.ceil(np.exp(1.0 + rng.standard_normal(k))))
    return _csr_from_rows(m, n, rows_cols, rows_vals, dtype)


def identity(n: int = 4096, dtype=np.float32) -> CSR:
    """S = I_n in CSR (n nonzeros of value 1)."""
    return CSR(n, n, np.arange(n + 1, dtype=np.int64), np.arange(n, dtype=np.int32),
               np.ones(n, dtype=dtype))


def connectome(n: int = 139255, mean_degree: float = 20.0, exponent: float = 2.2,
               seed: int = 0, dtype=np.float32) -> CSR:
    """Directed graph shaped like the fly connectome of Table 1.

    Out-degree d_i = min(n-1, floor(x_min * u^(-1/(exponent-1)))), u ~ U(0,1],
    a discrete power law with tail exponent ``exponent``; x_min is tuned by
    bisection on the realised degrees so that their mean is ``mean_degree``.
    Targets are uniform without replacement over the other n-1 nodes (no
    self-loops); values are synapse counts ceil(exp(1 + N(0,1))).
    """
    rng = np.random.default_rng([seed, 0xC0EC7])
    u = 1.0 - rng.random(n)                       # (0, 1]
    base = u ** (-1.0 / (exponent - 1.0))
    cap = n - 1

    def mean_for(xm):
        return np.minimum(cap, np.floor(xm * base)).mean()

    lo, hi = 0.0, 2.0 * mean_degree
    for _ in range(100):
        mid = 0.5 * (lo + hi)
        if mean_for(mid) >= mean_degree:
            hi = mid
        else:
            lo = mid
    x_min = hi
    deg = np.minimum(cap, np.floor(x_min * base)).astype(np.int64)

    rows_cols, rows_vals = [], []
    for i in range(n):
        d = int(deg[i])
        if d == 0:
            rows_cols.append(np.zeros(0, np.int64))
            rows_vals.append(np.zeros(0, np.float64))
            continue
        if 2 * d > cap:
            c = rng.permutation(cap)[:d]
        else:
            got = np.zeros(0, np.int64)
            while got.size < d:
                k = d - got.size
                cand = np.concatenate([got, rng.integers(0, cap, size=k + k // 8 + 8)])
                _, first = np.unique(cand, return_index=True)
                first.sort()
                got = cand[first[:d]]
            c = got
        c = np.where(c >= i, c + 1, c)
        v = np.ceil(np.exp(1.0 + rng.standard_normal(d)))
        o = np.argsort(c, kind="stable")
        rows_cols.append(c[o])
        rows_vals.append(v[o])
    S = _csr_from_rows(n, n, rows_cols, rows_vals, dtype)
    return S


# ---------------------------------------------------------------------------
# Named workloads.  ``scale`` shrinks the large ones (same generator and
# structure) for parity tests the oracle finishes in seconds.
# ---------------------------------------------------------------------------

def _planted_tiny(seed=0, r=4, **kw):
    S, U, V, tau = planted(600, 400, 4, tau=0.5, seed=seed)
    W, H = init_factors(S.m, S.n, r, seed)
    return Workload("planted-600x400-r%d" % r, S, r, W, H, 128, 128, "exact", 20, 1.0, 0.0,
                    seed, {"tau": tau, "d": 4})


# Step size and momentum per workload.  The paper's defaults are eta = 1 and
# gamma = 0.9 (Sec. 5.2), with smaller steps for under-parameterized models
# (Table "hyper").  On the synthetic stand-ins: the identity keeps the
# defaults; the planted 20000^2 matrix diverges with gamma = 0.9 (a block Gram
# matrix loses rank by sweep 9) and converges with eta = 1, gamma = 0; the
# connectome-shaped graph has no latent low-rank structure and diverges with
# eta = 1 (gamma 0 or 0.9) while eta = 0.5, gamma = 0.9 decreases the
# objective steadily.

def _identity(seed=0, n=4096, r=3, block=512, **kw):
    S = identity(n)
    W, H = init_factors(n, n, r, seed)
    return Workload("identity-%d-r%d" % (n, r), S, r, W, H, block, block, "stoch", 200,
                    1.0, 0.9, seed, {})


def _planted_medium(seed=0, n=20000, r=32, block=2048, **kw):
    S, U, V, tau = planted(n, n, 32, tau=None, density=0.05, noise=0.01, seed=seed)
    W, H = init_factors(n, n, r, seed)
    return Workload("planted-%dx%d-r%d" % (n, n, r), S, r, W, H, block, block, "stoch", 50,
                    1.0, 0.0, seed, {"tau": tau, "d": 32})


def _connectome(seed=0, n=139255, r=64, block=4096, sweeps=10, mean_degree=20.0, tag="", **kw):
    S = connectome(n, mean_degree=mean_degree, seed=seed)
    W, H = init_factors(n, n, r, seed)
    return Workload("connectome%s-%d-r%d" % (tag, n, r), S, r, W, H, block, block, "stoch", sweeps,
                    0.5, 0.9, seed, {"mean_degree": mean_degree})


def _communities(seed=0, n=139255, r=64, block=8192, clusters=64, run=128, **kw):
    # runs of 128 indices per community, taken in turn: every 128-row tile and
    # 128-row chunk lies in one community, and every block of 8192 holds all
    # 64 communities (so that its Gram matrix has full rank)
    S = communities(n, n, clusters, 20.0, seed=seed, run=run)
    W, H, _, _ = community_factors(n, n, r, clusters, seed=seed, run=run)
    return Workload("communities-%d-r%d-c%d" % (n, r, clusters), S, r, W, H, block, block, "stoch", 10,
                    0.5, 0.9, seed, {"clusters": clusters, "run": run, "mean_degree": 20.0})


def _communities_planted(seed=0, n=40960, r=64, block=8192, clusters=64, run=128, **kw):
    # S = max(0, W H) of clustered factors: a zero-loss fixed point whose
    # rectified product is block diagonal, so that the factors stay clustered.
    # With 64 communities in 64 dimensions the cosine across communities is
    # only about -1/8, so the groups must be tight (noise 0.002) for the
    # range search to separate them.
    W, H, _, _ = community_factors(n, n, r, clusters, noise=0.002, seed=seed, run=run)
    rows_cols, rows_vals = [], []
    Hd = H.astype(np.float64)
    for r0 in range(0, n, 2048):
        L = W[r0:r0 + 2048].astype(np.float64) @ Hd
        for row in L:
            c = np.nonzero(row > 0)[0]
            rows_cols.append(c)
            rows_vals.append(row[c])
    S = _csr_from_rows(n, n, rows_cols, rows_vals, np.float32)
    # no momentum: in the bf16 mode the rounding of the operands moves the
    # factors off the planted point a little every sweep (objective about
    # 2e-3), and momentum 0.9 keeps amplifying that drift until a block Gram
    # matrix loses rank after several sweeps; with gamma = 0 it settles
    return Workload("communities-planted-%d-r%d-c%d" % (n, r, clusters), S, r, W, H, block, block, "stoch", 10,
                    0.5, 0.0, seed, {"clusters": clusters, "run": run})


WORKLOADS = {
    "planted_tiny": _planted_tiny,
    "identity": _identity,
    "planted_medium": _planted_medium,
    "connectome_r64": lambda seed=0, **kw: _connectome(seed, r=64, block=4096, sweeps=10, **kw),
    "connectome_r256": lambda seed=0, **kw: _connectome(seed, r=256, block=8192, sweeps=5, **kw),
    # the same generator at the density of Table 1's connectome
    # (rho+ = 0.00102 of the n^2 entries: mean out-degree 142, ~19.8M nonzeros)
    "connectome_dense_r64": lambda seed=0, **kw: _connectome(seed, r=64, block=4096, sweeps=10,
                                                             mean_degree=0.00102 * 139254, tag="-dense", **kw),
    # a block-structured graph started from factors whose rows cluster by
    # community (the situation of Sec. 4.3 in which max(0, W H) is sparse)
    "communities_r64": _communities,
    "communities_planted_r64": _communities_planted,
}


def workload(name: str, seed: int = 0, **kw) -> Workload:
    return WORKLOADS[name](seed=seed, **kw)
