"""The C ABI library builds, loads and exports every symbol include/nmd.h
declares; host-side validation rejects malformed input.  No GPU needed."""
import ctypes as C
import os
import re

import numpy as np
import pytest

from paper_2608_21607_gb300 import build as B
from paper_2608_21607_gb300 import nmd as N
from paper_2608_21607_gb300 import workloads as WL

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def L():
    B.build()
    return N.lib()


def declared_symbols():
    text = open(os.path.join(ROOT, "include", "nmd.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(nmd_[a-z_]+)\s*\(", text)))


def test_every_declared_symbol_is_exported(L):
    decl = declared_symbols()
    assert len(decl) >= 15
    for name in decl:
        assert hasattr(L, name), name
    assert sorted(N.EXPORTS) == decl


def test_version_and_defaults(L):
    assert "libnmd" in N.nmd_version()
    o = N.nmd_default_options()
    assert o.block_rows == 4096 and o.eta == 1.0 and o.gamma == 0.9
    assert o.precision == N.NMD_BF16 and o.epilogue == N.NMD_EPI_Z and o.schedule == N.NMD_STOCH


def _ws(S, r=4, **kw):
    o = N.nmd_default_options()
    for k, v in kw.items():
        setattr(o, k, v)
    return N.nmd_workspace_bytes(S, r, o)


def test_workspace_bytes_for_a_valid_matrix(L):
    S, _, _, _ = WL.planted(60, 50, 4, tau=0.5, seed=0)
    nb = _ws(S, r=4, block_rows=16, block_cols=16)
    assert nb > 0 and nb % 256 == 0
    # grows with the rank padding
    assert _ws(S, r=100, block_rows=16, block_cols=16) > nb


class _Csr:
    def __init__(self, m, n, row_ptr, col_idx, vals):
        self.m, self.n = m, n
        self.row_ptr, self.col_idx, self.vals = row_ptr, col_idx, vals


@pytest.mark.parametrize("case,status", [
    ("rowptr0", N.NMD_ERR_CSR),
    ("decreasing", N.NMD_ERR_CSR),
    ("col_range", N.NMD_ERR_CSR),
    ("col_order", N.NMD_ERR_CSR),
    ("duplicate", N.NMD_ERR_CSR),
    ("negative", N.NMD_ERR_CSR),
    ("nan", N.NMD_ERR_CSR),
    ("all_zero", N.NMD_ERR_CSR),
    ("rank0", N.NMD_ERR_INVALID),
    ("rank257", N.NMD_ERR_INVALID),
    ("block0", N.NMD_ERR_INVALID),
    ("gamma1", N.NMD_ERR_INVALID),
    ("eta0", N.NMD_ERR_INVALID),
    ("precision", N.NMD_ERR_INVALID),
    ("m0", N.NMD_ERR_INVALID),
])
def test_validation_rejects(L, case, status):
    rp = np.array([0, 2, 3], np.int64)
    ci = np.array([0, 2, 1], np.int32)
    v = np.array([1.0, 2.0, 3.0], np.float32)
    m, n, r, kw = 2, 3, 2, {}
    if case == "rowptr0":
        rp = np.array([1, 2, 3], np.int64)
    elif case == "decreasing":
        rp = np.array([0, 3, 2], np.int64)
    elif case == "col_range":
        ci = np.array([0, 3, 1], np.int32)
    elif case == "col_order":
        ci = np.array([2, 0, 1], np.int32)
    elif case == "duplicate":
        ci = np.array([1, 1, 1], np.int32)
    elif case == "negative":
        v = np.array([1.0, -2.0, 3.0], np.float32)
    elif case == "nan":
        v = np.array([1.0, np.nan, 3.0], np.float32)
    elif case == "all_zero":
        v = np.zeros(3, np.float32)
    elif case == "rank0":
        r = 0
    elif case == "rank257":
        r = 257
    elif case == "block0":
        kw["block_rows"] = 0
    elif case == "gamma1":
        kw["gamma"] = 1.0
    elif case == "eta0":
        kw["eta"] = 0.0
    elif case == "precision":
        kw["precision"] = 7
    elif case == "m0":
        m = 0
        rp = np.array([0], np.int64)
    with pytest.raises(N.NmdError) as e:
        _ws(_Csr(m, n, rp, ci, v), r=r, **kw)
    assert e.value.status == status


def test_stored_zeros_are_dropped(L):
    """Support = stored entries with S_ij > 0 (eq. updateZ): zeros shrink nnz."""
    S = _Csr(2, 3, np.array([0, 2, 3], np.int64), np.array([0, 2, 1], np.int32),
             np.array([1.0, 2.0, 3.0], np.float32))
    Z = _Csr(2, 3, np.array([0, 2, 3], np.int64), np.array([0, 2, 1], np.int32),
             np.array([1.0, 0.0, 3.0], np.float32))
    assert _ws(Z, block_rows=1, block_cols=1) <= _ws(S, block_rows=1, block_cols=1)


def test_status_strings(L):
    for s in range(9):
        assert L.nmd_status_string(s)
