"""ctypes binding of libnmd (include/nmd.h).

Argument marshalling only: every step of the solver runs in the CUDA library.
PyTorch supplies the device workspace and the CUDA stream.  Importing this
module never falls back to anything: if ``_build/libnmd.so`` is missing the
first call raises.
"""
from __future__ import annotations

import ctypes as C
import os
from typing import Optional

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "_build", "libnmd.so")

NMD_OK, NMD_ERR_INVALID, NMD_ERR_CSR, NMD_ERR_NOT_SPD, NMD_ERR_DIVERGED = 0, 1, 2, 3, 4
NMD_ERR_TIMEOUT, NMD_ERR_CUDA, NMD_ERR_WORKSPACE, NMD_ERR_UNSUPPORTED = 5, 6, 7, 8
NMD_ROW, NMD_COL = 0, 1
NMD_EXACT, NMD_STOCH = 0, 1
NMD_ALTERNATE, NMD_PHASED = 0, 1
NMD_BF16, NMD_FP32, NMD_SIMT = 0, 1, 2
NMD_EPI_Z, NMD_EPI_DELTA = 0, 1
NMD_K_DENSE, NMD_K_SPARSE, NMD_K_GRAM, NMD_K_UPDATE, NMD_K_LOSS = 0, 1, 2, 3, 4
NMD_SKIP_NONE, NMD_SKIP_VOTE, NMD_SKIP_RANGE = 0, 1, 2

# every symbol include/nmd.h declares
EXPORTS = [
    "nmd_version", "nmd_default_options", "nmd_workspace_bytes", "nmd_create", "nmd_set_factors",
    "nmd_get_factors", "nmd_block_update", "nmd_sweep", "nmd_block_order", "nmd_loss", "nmd_sync",
    "nmd_block_terms", "nmd_dense_products", "nmd_panel_traversal", "nmd_get_state", "nmd_set_state",
    "nmd_launch_count", "nmd_skip_count", "nmd_selftest_wait_timeout", "nmd_profile", "nmd_profile_read", "nmd_status_string", "nmd_last_error",
    "nmd_destroy", "nmd_gram_noalloc", "nmd_support_term", "nmd_block_update_combined", "nmd_range_mask",
    "nmd_embed", "nmd_nn_workspace_bytes", "nmd_nearest_neighbors",
]


class nmd_options(C.Structure):
    _fields_ = [("block_rows", C.c_int64), ("block_cols", C.c_int64), ("schedule", C.c_int32),
                ("order", C.c_int32), ("eta", C.c_double), ("gamma", C.c_double),
                ("ridge", C.c_double), ("precision", C.c_int32), ("epilogue", C.c_int32),
                ("seed", C.c_uint64), ("skip_zero_chunks", C.c_int32)]


class nmd_loss_out(C.Structure):
    _fields_ = [("obj", C.c_double), ("rmse", C.c_double), ("wjd", C.c_double),
                ("s_fro", C.c_double), ("sum_relu2", C.c_double), ("sum_relu", C.c_double)]


class NmdError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__("%s (status %d)" % (msg, status))
        self.status = status


_lib = None
_P = C.c_void_p
_i64p = C.POINTER(C.c_int64)


def lib() -> C.CDLL:
    """The loaded libnmd.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError("libnmd.so not found at %s: build it with "
                               "paper_2608_21607_gb300.build.build()" % LIB_PATH)
        L = C.CDLL(LIB_PATH)
        sig = {
            "nmd_version": (C.c_char_p, []),
            "nmd_default_options": (None, [C.POINTER(nmd_options)]),
            "nmd_workspace_bytes": (C.c_int, [C.c_int64, C.c_int64, C.c_int32, _P, _P, _P,
                                              C.POINTER(nmd_options), C.POINTER(C.c_size_t)]),
            "nmd_create": (C.c_int, [C.c_int64, C.c_int64, C.c_int32, _P, _P, _P,
                                     C.POINTER(nmd_options), _P, C.c_size_t, _P, C.POINTER(_P)]),
            "nmd_set_factors": (C.c_int, [_P, _P, _P, C.c_int]),
            "nmd_get_factors": (C.c_int, [_P, _P, _P, C.c_int]),
            "nmd_block_update": (C.c_int, [_P, C.c_int32, C.c_int64, C.c_int32]),
            "nmd_sweep": (C.c_int, [_P]),
            "nmd_block_order": (C.c_int, [_P, C.c_int64, C.c_int32, _P, C.c_int64]),
            "nmd_loss": (C.c_int, [_P, C.POINTER(nmd_loss_out)]),
            "nmd_sync": (C.c_int, [_P]),
            "nmd_block_terms": (C.c_int, [_P, C.c_int32, C.c_int64, C.c_int32, _P, _P, _i64p]),
            "nmd_dense_products": (C.c_int, [_P, C.c_int32, C.c_int64, C.c_int32, _P, _i64p, _i64p]),
            "nmd_panel_traversal": (C.c_int, [_P, C.c_int32, C.c_int64, C.c_int32, _P, _P,
                                              C.c_int64, _i64p]),
            "nmd_get_state": (C.c_int, [_P, _P, _P, _P, _P, _i64p]),
            "nmd_set_state": (C.c_int, [_P, _P, _P, _P, _P, C.c_int64]),
            "nmd_launch_count": (C.c_int64, [_P]),
            "nmd_skip_count": (C.c_int, [_P, C.POINTER(C.c_int64), C.c_int32]),
            "nmd_selftest_wait_timeout": (C.c_int, [_P, C.c_int64]),
            "nmd_profile": (C.c_int, [_P, C.c_int]),
            "nmd_profile_read": (C.c_int, [_P, C.c_int32, C.POINTER(C.c_double), _i64p]),
            "nmd_status_string": (C.c_char_p, [C.c_int]),
            "nmd_last_error": (C.c_char_p, [_P]),
            "nmd_destroy": (None, [_P]),
            "nmd_gram_noalloc": (C.c_int, [_P, C.c_int64, C.c_int32, C.c_int64, _P, _P]),
            "nmd_support_term": (C.c_int, [_P, C.c_int32, C.c_int64, C.c_int32, _P, _i64p]),
            "nmd_block_update_combined": (C.c_int, [_P, C.c_int32, C.c_int64, C.c_int64]),
            "nmd_range_mask": (C.c_int, [_P, C.c_int32, C.c_int64, C.c_int32, _P, C.c_int64, _i64p, _i64p,
                                         _i64p]),
            "nmd_embed": (C.c_int, [_P, _P, _P]),
            "nmd_nn_workspace_bytes": (C.c_int, [C.c_int64, C.c_int32, C.POINTER(C.c_size_t)]),
            "nmd_nearest_neighbors": (C.c_int, [_P, C.c_int64, C.c_int32, _P, _P, _P, _i64p, _P, C.c_size_t,
                                                _P]),
        }
        for name, (res, args) in sig.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def _ptr(a) -> Optional[int]:
    if a is None:
        return None
    if isinstance(a, np.ndarray):
        return a.ctypes.data
    return a.data_ptr()   # torch tensor


def _check(h, st: int, what: str):
    if st != NMD_OK:
        L = lib()
        msg = L.nmd_last_error(h).decode() if h else ""
        raise NmdError(st, "%s: %s%s" % (what, L.nmd_status_string(st).decode(),
                                          (" -- " + msg) if msg else ""))


# ---------------------------------------------------------------------------
# The C calls under their own names
# ---------------------------------------------------------------------------

def nmd_version() -> str:
    return lib().nmd_version().decode()


def nmd_default_options() -> nmd_options:
    o = nmd_options()
    lib().nmd_default_options(C.byref(o))
    return o


def _csr_arrays(S):
    rp = np.ascontiguousarray(S.row_ptr, dtype=np.int64)
    ci = np.ascontiguousarray(S.col_idx, dtype=np.int32)
    v = np.ascontiguousarray(S.vals, dtype=np.float32)
    return rp, ci, v


def nmd_workspace_bytes(S, r: int, opts: nmd_options) -> int:
    rp, ci, v = _csr_arrays(S)
    out = C.c_size_t(0)
    st = lib().nmd_workspace_bytes(S.m, S.n, r, rp.ctypes.data, ci.ctypes.data, v.ctypes.data,
                                   C.byref(opts), C.byref(out))
    _check(None, st, "nmd_workspace_bytes")
    return out.value


def nmd_create(S, r: int, opts: nmd_options, workspace, stream_ptr: int):
    rp, ci, v = _csr_arrays(S)
    h = _P()
    st = lib().nmd_create(S.m, S.n, r, rp.ctypes.data, ci.ctypes.data, v.ctypes.data, C.byref(opts),
                          _ptr(workspace), workspace.numel() * workspace.element_size(), stream_ptr,
                          C.byref(h))
    _check(None, st, "nmd_create")
    return h


def nmd_set_factors(h, W, H, on_device: bool):
    _check(h, lib().nmd_set_factors(h, _ptr(W), _ptr(H), int(on_device)), "nmd_set_factors")


def nmd_get_factors(h, W, H, on_device: bool):
    _check(h, lib().nmd_get_factors(h, _ptr(W), _ptr(H), int(on_device)), "nmd_get_factors")


def nmd_block_update(h, side: int, block: int, kind: int):
    _check(h, lib().nmd_block_update(h, side, block, kind), "nmd_block_update")


def nmd_sweep(h):
    _check(h, lib().nmd_sweep(h), "nmd_sweep")


def nmd_block_order(h, sweep: int, side: int, K: int) -> list:
    out = np.zeros(K, np.int64)
    _check(h, lib().nmd_block_order(h, sweep, side, out.ctypes.data, K), "nmd_block_order")
    return out.tolist()


def nmd_loss(h) -> dict:
    o = nmd_loss_out()
    _check(h, lib().nmd_loss(h, C.byref(o)), "nmd_loss")
    return {k: getattr(o, k) for k, _ in nmd_loss_out._fields_}


def nmd_sync(h):
    _check(h, lib().nmd_sync(h), "nmd_sync")


def nmd_block_terms(h, side, block, kind, rows_max: int, r: int):
    R = np.zeros((rows_max, r), np.float32)
    G = np.zeros((r, r), np.float32)
    rows = C.c_int64(0)
    _check(h, lib().nmd_block_terms(h, side, block, kind, R.ctypes.data, G.ctypes.data, C.byref(rows)),
           "nmd_block_terms")
    return R[:rows.value], G


def nmd_dense_products(h, side, block, kind, d_L):
    rows = C.c_int64(0)
    cols = C.c_int64(0)
    _check(h, lib().nmd_dense_products(h, side, block, kind, _ptr(d_L), C.byref(rows), C.byref(cols)),
           "nmd_dense_products")
    return rows.value, cols.value


def nmd_panel_traversal(h, side, block, kind):
    cnt = C.c_int64(0)
    L = lib()
    _check(h, L.nmd_panel_traversal(h, side, block, kind, None, None, 0, C.byref(cnt)), "traversal")
    rows = np.zeros(cnt.value, np.int64)
    q = np.zeros(cnt.value, np.int64)
    _check(h, L.nmd_panel_traversal(h, side, block, kind, rows.ctypes.data, q.ctypes.data, cnt.value,
                                    C.byref(cnt)), "traversal")
    return rows, q


def nmd_block_update_combined(h, side, row_block, col_block):
    _check(h, lib().nmd_block_update_combined(h, side, row_block, col_block), "nmd_block_update_combined")


def nmd_support_term(h, side, block, kind, d_R) -> int:
    rows = C.c_int64(0)
    _check(h, lib().nmd_support_term(h, side, block, kind, _ptr(d_R), C.byref(rows)), "nmd_support_term")
    return rows.value


def nmd_range_mask(h, side, block, kind):
    """(mask, chunk_rows): mask[t, w] = word w of 128-row M tile t, bit c set =
    Q chunk 32 w + c cleared by the range search."""
    nt, nw, cr = C.c_int64(0), C.c_int64(0), C.c_int64(0)
    L = lib()
    _check(h, L.nmd_range_mask(h, side, block, kind, None, 0, C.byref(nt), C.byref(nw), C.byref(cr)),
           "nmd_range_mask")
    mask = np.zeros((nt.value, nw.value), dtype=np.uint32)
    _check(h, L.nmd_range_mask(h, side, block, kind, mask.ctypes.data, mask.size, C.byref(nt), C.byref(nw),
                               C.byref(cr)), "nmd_range_mask")
    return mask, cr.value


def nmd_embed(h, d_xi, d_sigma=None):
    _check(h, lib().nmd_embed(h, _ptr(d_xi), _ptr(d_sigma)), "nmd_embed")


def nmd_nn_workspace_bytes(N: int, d: int) -> int:
    v = C.c_size_t(0)
    _check(None, lib().nmd_nn_workspace_bytes(N, d, C.byref(v)), "nmd_nn_workspace_bytes")
    return v.value


def nmd_nearest_neighbors(d_x, N: int, d: int, d_labels, d_nn, d_best, workspace, stream_ptr: int):
    """Runs the search; returns the 1-NN error count (None without labels)."""
    err = C.c_int64(-1)
    _check(None, lib().nmd_nearest_neighbors(_ptr(d_x), N, d, _ptr(d_labels), _ptr(d_nn), _ptr(d_best),
                                             C.byref(err) if d_labels is not None else None, _ptr(workspace),
                                             workspace.numel(), stream_ptr), "nmd_nearest_neighbors")
    return err.value if d_labels is not None else None


def nearest_neighbors(x, labels=None):
    """(nn, best, errors) for the rows of a CUDA tensor x (N x d): the other
    row with the largest inner product, that inner product, and the number of
    rows whose neighbour has another label (None without labels).  The
    workspace is a torch tensor on x's device."""
    import torch
    x = x.contiguous().float()
    N, d = x.shape
    with torch.cuda.device(x.device):
        ws = torch.empty(nmd_nn_workspace_bytes(N, d), dtype=torch.uint8, device=x.device)
        nn = torch.empty(N, dtype=torch.int32, device=x.device)
        best = torch.empty(N, dtype=torch.float32, device=x.device)
        lab = None if labels is None else torch.as_tensor(labels, dtype=torch.int32).to(x.device).contiguous()
        errors = nmd_nearest_neighbors(x, N, d, lab, nn, best, ws, torch.cuda.current_stream(x.device).cuda_stream)
    return nn, best, errors


def nmd_get_state(h, m, n, r):
    W = np.zeros((m, r), np.float32); H = np.zeros((r, n), np.float32)
    EW = np.zeros((m, r), np.float32); EH = np.zeros((r, n), np.float32)
    s = C.c_int64(0)
    _check(h, lib().nmd_get_state(h, W.ctypes.data, H.ctypes.data, EW.ctypes.data, EH.ctypes.data,
                                  C.byref(s)), "nmd_get_state")
    return W, H, EW, EH, s.value


def nmd_set_state(h, W, H, EW, EH, sweep_index: int):
    arrs = [np.ascontiguousarray(a, np.float32) for a in (W, H, EW, EH)]
    _check(h, lib().nmd_set_state(h, *[a.ctypes.data for a in arrs], sweep_index), "nmd_set_state")


def nmd_launch_count(h) -> int:
    return lib().nmd_launch_count(h)


def nmd_selftest_wait_timeout(h, limit_ns: int) -> int:
    """Status of the bounded-wait self-test (NMD_ERR_TIMEOUT when it works)."""
    return int(lib().nmd_selftest_wait_timeout(h, int(limit_ns)))


def nmd_skip_count(h, reset: bool = False) -> int:
    v = C.c_int64(0)
    _check(h, lib().nmd_skip_count(h, C.byref(v), 1 if reset else 0), "nmd_skip_count")
    return int(v.value)


def nmd_profile(h, on: bool):
    _check(h, lib().nmd_profile(h, int(on)), "nmd_profile")


def nmd_profile_read(h, kernel_class: int):
    ms = C.c_double(0)
    n = C.c_int64(0)
    _check(h, lib().nmd_profile_read(h, kernel_class, C.byref(ms), C.byref(n)), "nmd_profile_read")
    return ms.value, n.value


def nmd_gram_noalloc(d_Q, K: int, r: int, ld: int, d_G, stream_ptr: int) -> int:
    """G = Q^T Q of a device matrix with no device allocation (static scratch);
    returns the status code."""
    return lib().nmd_gram_noalloc(_ptr(d_Q), K, r, ld, _ptr(d_G), stream_ptr)


def nmd_destroy(h):
    lib().nmd_destroy(h)


# ---------------------------------------------------------------------------
# Convenience wrapper owning the torch workspace
# ---------------------------------------------------------------------------

class Solver:
    """SALSA solver for S ~ max(0, W H) on the current CUDA device.

    ``S`` is any object with m, n, row_ptr, col_idx, vals (CSR).  The device
    workspace is a torch uint8 tensor owned by this object; the stream is
    torch's current stream unless one is given.
    """

    def __init__(self, S, r: int, *, block_rows=4096, block_cols=4096, schedule=NMD_STOCH,
                 order=NMD_ALTERNATE, eta=1.0, gamma=0.9, ridge=0.0, precision=NMD_BF16,
                 epilogue=NMD_EPI_Z, seed=0, skip_zero_chunks=False, stream=None, device=None):
        import torch
        self.m, self.n, self.r = int(S.m), int(S.n), int(r)
        o = nmd_default_options()
        o.block_rows, o.block_cols = int(block_rows), int(block_cols)
        o.schedule, o.order = int(schedule), int(order)
        o.eta, o.gamma, o.ridge = float(eta), float(gamma), float(ridge)
        o.precision, o.epilogue, o.seed = int(precision), int(epilogue), int(seed)
        o.skip_zero_chunks = int(skip_zero_chunks)   # False/True or an NMD_SKIP_* mode
        self.opts = o
        self.device = torch.device(device) if device is not None else torch.device("cuda", torch.cuda.current_device())
        nbytes = nmd_workspace_bytes(S, self.r, o)
        with torch.cuda.device(self.device):
            self.workspace = torch.empty(nbytes, dtype=torch.uint8, device=self.device)
            self.stream = stream if stream is not None else torch.cuda.current_stream(self.device)
            self.h = nmd_create(S, self.r, o, self.workspace, self.stream.cuda_stream)

    def __del__(self):
        h = getattr(self, "h", None)
        if h:
            nmd_destroy(h)
            self.h = None

    def set_factors(self, W, H):
        import torch
        on_dev = isinstance(W, torch.Tensor) and W.is_cuda
        if on_dev:
            W = W.contiguous().float(); H = H.contiguous().float()
            self._keep = (W, H)
        else:
            W = np.ascontiguousarray(W, np.float32); H = np.ascontiguousarray(H, np.float32)
        nmd_set_factors(self.h, W, H, on_dev)

    def get_factors(self):
        W = np.zeros((self.m, self.r), np.float32)
        H = np.zeros((self.r, self.n), np.float32)
        nmd_get_factors(self.h, W, H, False)
        return W, H

    def get_factors_device(self, W, H):
        nmd_get_factors(self.h, W, H, True)

    def block_update(self, side, block, kind):
        nmd_block_update(self.h, side, block, kind)

    def block_update_combined(self, side, row_block, col_block):
        """Combined row and column sub-sampling: W_I from H_:J (NMD_ROW) or
        H_:J from W_I (NMD_COL), on S[I, J]."""
        nmd_block_update_combined(self.h, side, row_block, col_block)

    def sweep(self):
        nmd_sweep(self.h)

    def loss(self) -> dict:
        return nmd_loss(self.h)

    def sync(self):
        nmd_sync(self.h)

    def block_order(self, sweep, side):
        K = -(-self.m // self.opts.block_rows) if side == NMD_ROW else -(-self.n // self.opts.block_cols)
        return nmd_block_order(self.h, sweep, side, K)

    def block_terms(self, side, block, kind):
        return nmd_block_terms(self.h, side, block, kind, max(self.m, self.n), self.r)

    def dense_products(self, side, block, kind, M, K):
        """L = M Q^T of one block as the tensor-core kernel forms it (numpy)."""
        import torch
        d = torch.zeros(M * K, dtype=torch.float32, device=self.device)
        rows, cols = nmd_dense_products(self.h, side, block, kind, d)
        return d[:rows * cols].view(rows, cols).cpu().numpy()

    def panel_traversal(self, side, block, kind):
        return nmd_panel_traversal(self.h, side, block, kind)

    @property
    def r_pad(self) -> int:
        return next(p for p in (16, 32, 64, 128, 256) if self.r <= p)

    def support_term(self, side, block, kind, d_R=None):
        """The support term Rs of one block update (rows x r_pad, device
        tensor); asynchronous on the solver's stream."""
        import torch
        if d_R is None:
            d_R = torch.empty(max(self.m, self.n) * self.r_pad, dtype=torch.float32, device=self.device)
        rows = nmd_support_term(self.h, side, block, kind, d_R)
        return d_R[:rows * self.r_pad].view(rows, self.r_pad)

    def get_state(self):
        return nmd_get_state(self.h, self.m, self.n, self.r)

    def set_state(self, W, H, EW, EH, sweep_index):
        nmd_set_state(self.h, W, H, EW, EH, sweep_index)

    def profile(self, on: bool):
        nmd_profile(self.h, on)

    def profile_read(self, kernel_class: int):
        """(device ms, launches) of one kernel class since profile(True)."""
        return nmd_profile_read(self.h, kernel_class)

    @property
    def launches(self) -> int:
        return nmd_launch_count(self.h)

    def skip_count(self, reset: bool = False) -> int:
        """Delta form: chunks skipped (NMD_SKIP_VOTE: second product of an
        all-zero P; NMD_SKIP_RANGE: both products of a cleared chunk)."""
        return nmd_skip_count(self.h, reset)

    def embed(self):
        """(xi, sigma) as CUDA tensors: the n x 2r unit rows of the cell
        embedding (Sec. 5.3) and the r singular values of W H, descending."""
        import torch
        with torch.cuda.device(self.device):
            xi = torch.empty((self.n, 2 * self.r), dtype=torch.float32, device=self.device)
            sigma = torch.empty(self.r, dtype=torch.float32, device=self.device)
            nmd_embed(self.h, xi, sigma)
        return xi, sigma

    def range_mask(self, side, block, kind):
        """The range-search mask of one block update and its chunk size."""
        return nmd_range_mask(self.h, side, block, kind)
