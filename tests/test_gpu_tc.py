"""The two tensor-core products of the fused panel kernel, checked separately.

MMA1 (L = M Q^T) through the nmd_dense_products hook against the same
product of the rounded operands in fp64; MMA2 (R = P(L) Q plus the sparse
correction) against a CPU restatement fed with the kernel's own L (in the
bf16 mode the whole step uses the bf16 rows q_hi: P q_hi plus the support
term on q_hi, paired with the Gram matrix of q_hi, reported by the hook as
the equivalent right-hand side under the exact G).  Covers
every padded rank (16, 32, 64, 128, 256), both epilogues, both tensor-core
precisions, ragged M and K tails.
"""
import numpy as np
import pytest

import oracle as O
from paper_2608_21607_gb300 import nmd as N
from paper_2608_21607_gb300 import workloads as WL

from gpu_common import rel, require_gpu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def gpu():
    return require_gpu()


def bf16_round(x):
    """Round fp32 values to bf16 (nearest even), returned as float64."""
    a = np.ascontiguousarray(x, np.float32).view(np.uint32).astype(np.uint64)
    rounded = (a + 0x7FFF + ((a >> 16) & 1)) & 0xFFFF0000
    return rounded.astype(np.uint32).view(np.float32).astype(np.float64)


def pieces(X):
    """bf16 pieces hi, lo, lo2 of fp32 values (each difference exact in fp32)."""
    X = np.asarray(X, np.float32).astype(np.float64)
    hi = bf16_round(X.astype(np.float32))
    lo = bf16_round((X - hi).astype(np.float32))
    lo2 = bf16_round((X - hi - lo).astype(np.float32))
    return hi, lo, lo2


def operands(X, precision):
    """The values the first product sees for factor rows X (fp32)."""
    hi, lo, _ = pieces(X)
    if precision == N.NMD_BF16:
        return hi
    return hi, lo


def products(A, B, precision):
    if precision == N.NMD_BF16:
        return operands(A, precision) @ operands(B, precision).T
    ah, al = operands(A, precision)
    bh, bl = operands(B, precision)
    return ah @ bh.T + ah @ bl.T + al @ bh.T


# (r, n, block): every block, the ragged last one too, has at least r rows
RANKS = [(3, 1000, 192), (32, 700, 160), (64, 900, 200), (100, 600, 224), (256, 900, 300)]


@pytest.mark.parametrize("precision", [N.NMD_BF16, N.NMD_FP32], ids=["bf16", "fp32"])
@pytest.mark.parametrize("r,n,b", RANKS, ids=[str(x[0]) for x in RANKS])
def test_first_product_L(r, n, b, precision):
    S = WL.connectome(n, seed=r)
    W, H = WL.init_factors(n, n, r, r)
    sol = N.Solver(S, r, block_rows=b, block_cols=b, precision=precision)
    sol.set_factors(W, H)
    B = H.T
    K = O.num_blocks(n, b)
    for side, kind, block in [(N.NMD_COL, N.NMD_STOCH, 0), (N.NMD_COL, N.NMD_STOCH, K - 1),
                              (N.NMD_ROW, N.NMD_EXACT, K - 1), (N.NMD_ROW, N.NMD_STOCH, 1)]:
        if side == N.NMD_COL and kind == N.NMD_STOCH:
            j0, j1 = O.block_range(block, b, n)
            want = products(W, B[j0:j1], precision)
        elif side == N.NMD_ROW and kind == N.NMD_EXACT:
            i0, i1 = O.block_range(block, b, n)
            want = products(W[i0:i1], B, precision)
        else:
            i0, i1 = O.block_range(block, b, n)
            want = products(B, W[i0:i1], precision)
        got = sol.dense_products(side, block, kind, *want.shape)
        assert got.shape == want.shape
        tol = 2e-6 if precision == N.NMD_BF16 else 1e-5
        assert rel(got, want) <= tol, (side, kind, block, rel(got, want))


@pytest.mark.parametrize("precision", [N.NMD_BF16, N.NMD_FP32], ids=["bf16", "fp32"])
@pytest.mark.parametrize("epi", [N.NMD_EPI_Z, N.NMD_EPI_DELTA], ids=["zform", "delta"])
@pytest.mark.parametrize("r,n,b", RANKS, ids=[str(x[0]) for x in RANKS])
def test_second_product_R(r, n, b, epi, precision):
    S = WL.connectome(n, seed=r + 1)
    W, H = WL.init_factors(n, n, r, r + 1)
    sol = N.Solver(S, r, block_rows=b, block_cols=b, precision=precision, epilogue=epi)
    sol.set_factors(W, H)
    st = O.State(S, W, H, O.Options(block_rows=b, block_cols=b))
    K = O.num_blocks(n, b)
    for side, kind, block in [(N.NMD_COL, N.NMD_STOCH, K - 1), (N.NMD_ROW, N.NMD_STOCH, 0)]:
        M, _, (m0, m1), Q, src, (c0, c1) = st._roles(side, block, kind)
        L = sol.dense_products(side, block, kind, m1 - m0, c1 - c0).astype(np.float64)
        P = np.minimum(0, L) if epi == N.NMD_EPI_Z else -np.maximum(0, L)
        Qf = Q.astype(np.float32)
        qh, ql, ql2 = pieces(Qf)
        Qd = Qf.astype(np.float64)
        Sd = src.dense_panel(m0, m1, c0, c1)
        sup = Sd > 0
        if precision == N.NMD_BF16:
            # the whole step on the bf16 rows: R' = P q_hi + c q_hi with
            # c = S - min(0, m_hi . q_hi) on the support, solved with
            # Gt = q_hi^T q_hi; the hook reports the right-hand side with the
            # same solution under the exact G: R' Gt^{-1} G
            Pb = bf16_round(P.astype(np.float32))
            mh = pieces(M[m0:m1].astype(np.float32))[0]
            Lb = (mh @ qh.T).astype(np.float32).astype(np.float64)
            corr = np.where(sup, Sd - np.minimum(0, Lb), 0.0)
            want = (Pb @ qh + corr @ qh) @ np.linalg.solve(qh.T @ qh, Qd.T @ Qd)
        else:                             # P_hi (q_hi + q_lo + q_lo2) + P_lo q_hi
            ph = bf16_round(P.astype(np.float32))
            pl = bf16_round((P - ph).astype(np.float32))
            want = ph @ (qh + ql + ql2) + pl @ qh
            # the support correction uses fp32 L and q: c = S - min(0, L) on the support
            Lf = (M[m0:m1].astype(np.float32) @ Qf.T).astype(np.float64)
            corr = np.where(sup, Sd - np.minimum(0, Lf), 0.0)
            want = want + corr @ Qd
        got, _ = sol.block_terms(side, block, kind)
        assert rel(got, want) <= 1e-5, (side, kind, block, rel(got, want))
