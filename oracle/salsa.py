"""fp64 CPU oracle for the SALSA block sweep -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this module.  The CUDA library never calls it and
shares no code with it (the only common module is the seeded input generator,
which holds none of the method's arithmetic).

What it computes (paper notation: L = A B^T, A = W is m x r, B = H^T is n x r):

* Z update, Sec. 3.2 eq. (updateZ): Z_ij = S_ij where S_ij > 0, else
  L_ij - max(0, L_ij) = min(0, L_ij).
* Least-squares factor updates, eqs. (lsqA)/(lsqB): A <- Z B (B^T B)^{-1},
  B <- Z^T A (A^T A)^{-1}; restricted to a contiguous row block I (parallel
  least squares, eqs. Shat_par/Delta_par/lsqA_par, Sec. 4.1), to a random
  column mini-batch J with step size eta (stochastic least squares,
  eqs. Shat_sto/Delta_sto/lsqA_sto, Sec. 4.1), or to both at once (the
  combined row and column sub-sampling remarked on after eq. lsqA_sto).
* Momentum: "a multiple of the previously executed update" (Sec. 4.1, after
  eq. lsqA_sto), read as heavy ball E_t = U_t + gamma E_{t-1}, M += E_t.
* Losses: objective ||Z - L||_F / ||S||_F (eq. auxCost, evaluated through
  eq. SLloss), RMSE (eq. RMSE) and weighted Jaccard distance (eq. WJD).
* The index set Omega of the positive entries of L (Sec. 4.3), both by its
  definition (eq. nonzeros) and as a range search over the normalised rows
  (eq. range-search).

Every Z panel is materialised explicitly in fp64, the right-hand side R = Z Q
and Gram matrix G = Q^T Q are formed with plain matrix products, G is factored
by a hand-written Cholesky and the normal equations are solved by forward and
back substitution.  Nothing is fused, blocked or reordered beyond splitting
the M-side rows into chunks (each row's result is independent of the others).

The block order comes from the SplitMix64 generator (S. Vigna's published
definition) driving a Fisher-Yates shuffle of the block indices, one
permutation per (seed, sweep, side).
"""
from __future__ import annotations

import dataclasses
import math
from typing import Optional

import numpy as np

ROW, COL = 0, 1
EXACT, STOCH = 0, 1
ALTERNATE, PHASED = 0, 1

_MASK = (1 << 64) - 1
_GOLDEN = 0x9E3779B97F4A7C15


class NotSPD(ArithmeticError):
    """The block Gram matrix has a non-positive pivot."""


# ---------------------------------------------------------------------------
# Block order: SplitMix64 + Fisher-Yates
# ---------------------------------------------------------------------------

def splitmix64_mix(z: int) -> int:
    """SplitMix64 output function (Vigna): two xor-shift-multiply rounds."""
    z &= _MASK
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & _MASK
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & _MASK
    return z ^ (z >> 31)


class SplitMix64:
    def __init__(self, state: int):
        self.state = state & _MASK

    def next(self) -> int:
        self.state = (self.state + _GOLDEN) & _MASK
        return splitmix64_mix(self.state)


def fisher_yates(K: int, g: SplitMix64) -> list:
    """Shuffle of [0, K) from the top: for i = K-1 .. 1, j = next() mod (i+1),
    swap(i, j) (the modulo bias, below 2^-57 for K < 2^7, is part of the order)."""
    perm = list(range(K))
    for i in range(K - 1, 0, -1):
        j = g.next() % (i + 1)
        perm[i], perm[j] = perm[j], perm[i]
    return perm


def block_permutation(seed: int, sweep: int, side: int, K: int) -> list:
    """Order in which the K blocks of one side are visited in sweep ``sweep``:
    Fisher-Yates driven by SplitMix64 with state mix(seed) xor mix((sweep << 1) | side)."""
    return fisher_yates(K, SplitMix64(splitmix64_mix(seed) ^ splitmix64_mix(((sweep << 1) | side) & _MASK)))


def num_blocks(N: int, b: int) -> int:
    return (N + b - 1) // b


def block_range(k: int, b: int, N: int):
    """Contiguous index range of block k (Sec. 4.1: contiguous row indices)."""
    return k * b, min((k + 1) * b, N)


# ---------------------------------------------------------------------------
# Sparse helpers (CSR of S and of S^T)
# ---------------------------------------------------------------------------

@dataclasses.dataclass
class Sparse:
    m: int
    n: int
    row_ptr: np.ndarray
    col_idx: np.ndarray
    vals: np.ndarray      # fp64

    @staticmethod
    def from_csr(S) -> "Sparse":
        """Copy of a CSR (only entries with value > 0 form the support)."""
        keep = np.asarray(S.vals) > 0
        rows = np.repeat(np.arange(S.m), np.diff(S.row_ptr))[keep]
        cols = np.asarray(S.col_idx)[keep].astype(np.int64)
        vals = np.asarray(S.vals)[keep].astype(np.float64)
        row_ptr = np.zeros(S.m + 1, np.int64)
        np.cumsum(np.bincount(rows, minlength=S.m), out=row_ptr[1:])
        return Sparse(S.m, S.n, row_ptr, cols, vals)

    def transpose(self) -> "Sparse":
        rows = np.repeat(np.arange(self.m), np.diff(self.row_ptr))
        order = np.lexsort((rows, self.col_idx))       # by column, then row
        cols_t = rows[order]
        row_ptr = np.zeros(self.n + 1, np.int64)
        np.cumsum(np.bincount(self.col_idx, minlength=self.n), out=row_ptr[1:])
        return Sparse(self.n, self.m, row_ptr, cols_t, self.vals[order])

    def dense_panel(self, r0: int, r1: int, c0: int, c1: int) -> np.ndarray:
        """Rows [r0, r1) and columns [c0, c1) of this matrix as a dense fp64 array."""
        out = np.zeros((r1 - r0, c1 - c0))
        a, b = self.row_ptr[r0], self.row_ptr[r1]
        rows = np.repeat(np.arange(r0, r1), np.diff(self.row_ptr[r0:r1 + 1])) - r0
        cols = self.col_idx[a:b]
        keep = (cols >= c0) & (cols < c1)
        out[rows[keep], cols[keep] - c0] = self.vals[a:b][keep]
        return out

    def fro(self) -> float:
        return float(np.sqrt(np.sum(self.vals ** 2)))


# ---------------------------------------------------------------------------
# Dense linear algebra written out
# ---------------------------------------------------------------------------

def cholesky(G: np.ndarray) -> np.ndarray:
    """Lower-triangular C with C C^T = G (column-by-column Cholesky)."""
    n = G.shape[0]
    C = np.zeros_like(G, dtype=np.float64)
    for j in range(n):
        d = G[j, j] - C[j, :j] @ C[j, :j]
        if not d > 0.0:
            raise NotSPD("non-positive pivot %r at column %d" % (d, j))
        C[j, j] = math.sqrt(d)
        C[j + 1:, j] = (G[j + 1:, j] - C[j + 1:, :j] @ C[j, :j]) / C[j, j]
    return C


def solve_normal(C: np.ndarray, R: np.ndarray) -> np.ndarray:
    """X = R G^{-1} for G = C C^T: forward then back substitution on X^T."""
    r = C.shape[0]
    Rt = np.asarray(R, dtype=np.float64).T
    Y = np.zeros_like(Rt)
    for i in range(r):
        Y[i] = (Rt[i] - C[i, :i] @ Y[:i]) / C[i, i]
    X = np.zeros_like(Rt)
    for i in range(r - 1, -1, -1):
        X[i] = (Y[i] - C[i + 1:, i] @ X[i + 1:]) / C[i, i]
    return X.T


# ---------------------------------------------------------------------------
# Z update and the losses
# ---------------------------------------------------------------------------

def update_z(S_panel: np.ndarray, L: np.ndarray) -> np.ndarray:
    """Eq. (updateZ): S where S > 0, otherwise L - max(0, L) = min(0, L)."""
    return np.where(S_panel > 0, S_panel, L - np.maximum(0.0, L))


def loss(Sp: Sparse, A: np.ndarray, B: np.ndarray, rows: Optional[np.ndarray] = None,
         chunk: int = 2048) -> dict:
    """Objective (eq. auxCost via eq. SLloss), RMSE (eq. RMSE), WJD (eq. WJD).

    L = A B^T is materialised row chunk by row chunk.  With ``rows`` given,
    the sums run over those rows of S only (the normalisation still uses the
    whole ||S||_F) -- used to check large problems on a sample.
    """
    A = np.asarray(A, np.float64)
    B = np.asarray(B, np.float64)
    idx = np.arange(Sp.m) if rows is None else np.asarray(rows)
    zl2 = err2 = smin = smax = 0.0
    for c0 in range(0, len(idx), chunk):
        rr = idx[c0:c0 + chunk]
        L = A[rr] @ B.T
        Sd = np.zeros_like(L)
        for k, i in enumerate(rr):
            a, b = Sp.row_ptr[i], Sp.row_ptr[i + 1]
            Sd[k, Sp.col_idx[a:b]] = Sp.vals[a:b]
        Z = update_z(Sd, L)
        Shat = np.maximum(0.0, L)
        zl2 += float(np.sum((Z - L) ** 2))
        err2 += float(np.sum((Sd - Shat) ** 2))
        smin += float(np.sum(np.minimum(Sd, Shat)))
        smax += float(np.sum(np.maximum(Sd, Shat)))
    s_fro = Sp.fro()
    return {"obj": math.sqrt(zl2) / s_fro, "rmse": math.sqrt(err2) / s_fro,
            "wjd": 1.0 - smin / smax if smax > 0 else 0.0, "s_fro": s_fro,
            "sum_min": smin, "sum_max": smax, "zl2": zl2, "err2": err2}


# ---------------------------------------------------------------------------
# The solver state and one block update
# ---------------------------------------------------------------------------

# ---------------------------------------------------------------------------
# The positive entries of L (Sec. 4.3, "Fast similarity search")
# ---------------------------------------------------------------------------

def positive_set(A: np.ndarray, B: np.ndarray) -> np.ndarray:
    """Omega of eq. nonzeros: the pairs (i, j) with (A B^T)_ij > 0, as an
    m x n boolean array (fp64 product)."""
    return (np.asarray(A, np.float64) @ np.asarray(B, np.float64).T) > 0


def range_search_set(A: np.ndarray, B: np.ndarray) -> np.ndarray:
    """Omega of eq. range-search: the pairs whose normalised rows a_i/|a_i|
    and b_j/|b_j| are less than two units of squared distance apart, found
    by comparing every pair (brute force).  A zero row has no direction and
    takes part in no pair (its entries of L are zero)."""
    A = np.asarray(A, np.float64)
    B = np.asarray(B, np.float64)
    na = np.sqrt((A * A).sum(axis=1))
    nb = np.sqrt((B * B).sum(axis=1))
    out = np.zeros((A.shape[0], B.shape[0]), dtype=bool)
    for i in range(A.shape[0]):
        if na[i] == 0:
            continue
        ahat = A[i] / na[i]
        for j in range(B.shape[0]):
            if nb[j] == 0:
                continue
            d = ahat - B[j] / nb[j]
            out[i, j] = float(d @ d) < 2.0
    return out


@dataclasses.dataclass
class Options:
    block_rows: int = 128
    block_cols: int = 128
    schedule: int = STOCH
    order: int = ALTERNATE
    eta: float = 1.0
    gamma: float = 0.0
    ridge: float = 0.0
    seed: int = 0


class State:
    """Factors A = W (m x r) and B = H^T (n x r) in fp64 plus momentum."""

    def __init__(self, S, W, H, opts: Options):
        self.S = Sparse.from_csr(S)
        self.St = self.S.transpose()
        self.A = np.array(W, dtype=np.float64)
        self.B = np.array(H, dtype=np.float64).T.copy()
        self.EA = np.zeros_like(self.A)
        self.EB = np.zeros_like(self.B)
        self.opts = opts
        self.sweep_index = 0
        self.m, self.n = self.S.m, self.S.n
        self.r = self.A.shape[1]

    @property
    def W(self):
        return self.A

    @property
    def H(self):
        return self.B.T

    def loss(self, **kw):
        return loss(self.S, self.A, self.B, **kw)

    def _roles(self, side: int, block: int, kind: int):
        """(M factor, E of M, M row range, Q rows, panel source, panel column range).

        ROW/EXACT: A_I from all of B on S[I, :]      (eq. lsqA_par)
        COL/EXACT: B_J from all of A on S[:, J]^T    (same, for B)
        COL/STOCH: all of A from B_J on S[:, J]      (eq. lsqA_sto)
        ROW/STOCH: all of B from A_I on S[I, :]^T    (eq. lsqA_sto for B)
        """
        o = self.opts
        if side == ROW:
            i0, i1 = block_range(block, o.block_rows, self.m)
            if kind == EXACT:
                return self.A, self.EA, (i0, i1), self.B, self.S, (0, self.n)
            return self.B, self.EB, (0, self.n), self.A[i0:i1], self.St, (i0, i1)
        j0, j1 = block_range(block, o.block_cols, self.n)
        if kind == EXACT:
            return self.B, self.EB, (j0, j1), self.A, self.St, (0, self.m)
        return self.A, self.EA, (0, self.m), self.B[j0:j1], self.S, (j0, j1)

    def _roles_combined(self, side: int, row_block: int, col_block: int):
        """Combined row and column sub-sampling (Sec. 4.1, the remark after eq.
        lsqA_sto: one update that subsamples rows and columns of Delta):

        ROW: A_I from B_J on S[I, J]      (eq. lsqA_sto restricted to the rows I)
        COL: B_J from A_I on S[I, J]^T    (the same for B)
        """
        o = self.opts
        i0, i1 = block_range(row_block, o.block_rows, self.m)
        j0, j1 = block_range(col_block, o.block_cols, self.n)
        if side == ROW:
            return self.A, self.EA, (i0, i1), self.B[j0:j1], self.S, (j0, j1)
        return self.B, self.EB, (j0, j1), self.A[i0:i1], self.St, (i0, i1)

    def block_terms(self, side: int, block: int, kind: int, chunk_elems: int = 1 << 24,
                    rows=None):
        """R = Z Q for the M-side rows and G = Q^T Q.

        With ``rows`` (indices relative to the first M-side row) only those
        rows of R are formed -- each row of R depends on its own row of Z only.
        """
        return self._terms(self._roles(side, block, kind), chunk_elems, rows)

    def block_terms_combined(self, side: int, row_block: int, col_block: int):
        """R = Z Q and G = Q^T Q of a combined row and column step."""
        return self._terms(self._roles_combined(side, row_block, col_block))

    def _terms(self, roles, chunk_elems: int = 1 << 24, rows=None):
        M, _, (m0, m1), Q, src, (c0, c1) = roles
        K = c1 - c0
        G = Q.T @ Q
        if rows is not None:
            R = np.zeros((len(rows), self.r))
            for t, i in enumerate(rows):
                a = m0 + int(i)
                L = M[a:a + 1] @ Q.T
                Z = update_z(src.dense_panel(a, a + 1, c0, c1), L)
                R[t] = (Z @ Q)[0]
            return R, G
        R = np.zeros((m1 - m0, self.r))
        step = max(1, chunk_elems // max(K, 1))
        for a in range(m0, m1, step):
            b = min(m1, a + step)
            L = M[a:b] @ Q.T
            Z = update_z(src.dense_panel(a, b, c0, c1), L)
            R[a - m0:b - m0] = Z @ Q
        return R, G

    def traversal(self, side: int, block: int, kind: int):
        """(M-side row, Q-side index) pairs of the block's support: rows
        ascending, Q-side index ascending within a row (both relative to the
        block's first M-side / Q-side row)."""
        _, _, (m0, m1), _, src, (c0, c1) = self._roles(side, block, kind)
        a, b = src.row_ptr[m0], src.row_ptr[m1]
        rows = np.repeat(np.arange(m0, m1), np.diff(src.row_ptr[m0:m1 + 1]))
        cols = src.col_idx[a:b]
        keep = (cols >= c0) & (cols < c1)
        return rows[keep] - m0, cols[keep] - c0

    def block_update(self, side: int, block: int, kind: int):
        self._update(self._roles(side, block, kind), momentum=kind == STOCH)

    def block_update_combined(self, side: int, row_block: int, col_block: int):
        """A stochastic step (step size eta, momentum) on the rows of one block
        of the updated factor against one block of the other, on S[I, J]."""
        self._update(self._roles_combined(side, row_block, col_block), momentum=True)

    def _update(self, roles, momentum: bool):
        o = self.opts
        M, E, (m0, m1), Q, _, _ = roles
        R, G = self._terms(roles)
        if o.ridge:
            G = G + o.ridge * np.eye(self.r)
        C = cholesky(G)
        M_ls = solve_normal(C, R)
        U = o.eta * (M_ls - M[m0:m1])
        if momentum:
            E[m0:m1] = U + o.gamma * E[m0:m1]
            M[m0:m1] += E[m0:m1]
        else:
            M[m0:m1] += U

    def sweep_steps(self, sweep: Optional[int] = None):
        """The (side, block, kind) sequence of one sweep."""
        o = self.opts
        s = self.sweep_index if sweep is None else sweep
        Kr, Kc = num_blocks(self.m, o.block_rows), num_blocks(self.n, o.block_cols)
        pr = block_permutation(o.seed, s, ROW, Kr)
        pc = block_permutation(o.seed, s, COL, Kc)
        if o.schedule == EXACT:
            return [(ROW, b, EXACT) for b in pr] + [(COL, b, EXACT) for b in pc]
        if o.order == PHASED:
            return [(COL, b, STOCH) for b in pc] + [(ROW, b, STOCH) for b in pr]
        steps = []
        for t in range(max(Kr, Kc)):
            if t < Kc:
                steps.append((COL, pc[t], STOCH))
            if t < Kr:
                steps.append((ROW, pr[t], STOCH))
        return steps

    def sweep(self):
        for side, block, kind in self.sweep_steps():
            self.block_update(side, block, kind)
        self.sweep_index += 1
