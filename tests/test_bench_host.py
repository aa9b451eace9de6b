"""Host-side arithmetic of bench.py that no GPU run checks: the algorithmic
bytes of the support term (8 B per support entry, one m row read and one Rs
row written per panel row, each factor's rows once; the q-row gathers
counted apart) and the step count of a sweep, on a matrix small enough to
count by hand."""
import numpy as np

import bench
from paper_2608_21607_gb300 import workloads as WL


class _WL:
    def __init__(self, S, r, br, bc):
        self.S, self.r, self.block_rows, self.block_cols = S, r, br, bc
        self.m, self.n = S.m, S.n


def test_support_bytes_by_hand():
    # 4 x 5, blocks of 2 rows and 2 columns (3 column blocks, the last ragged)
    D = np.array([[1, 0, 2, 0, 0],
                  [0, 0, 0, 0, 3],
                  [4, 5, 0, 0, 0],
                  [0, 0, 0, 6, 7]], dtype=np.float64)
    S = WL.csr_from_dense(D)
    r, e = 3, 2
    dram, gather = bench.support_bytes_per_sweep(_WL(S, r, 2, 2), e)
    nnz = 7
    # column steps: (row, column block) pairs with support
    col_pairs = len({(0, 0), (0, 1), (1, 2), (2, 0), (3, 1), (3, 2)})
    # row steps: (column, row block) pairs with support
    row_pairs = len({(0, 0), (2, 0), (4, 0), (0, 1), (1, 1), (3, 1), (4, 1)})
    want = 2 * nnz * 8 + (col_pairs + row_pairs) * (e * r + 4 * r) + (4 + 5) * e * r
    assert dram == want
    assert gather == 2 * nnz * e * r


def test_support_bytes_scale_with_operand_width():
    S = WL.connectome(300, seed=1)
    w = _WL(S, 16, 64, 64)
    d2, g2 = bench.support_bytes_per_sweep(w, 2)
    d4, g4 = bench.support_bytes_per_sweep(w, 4)
    assert g4 == 2 * g2
    assert d4 > d2
