"""Shared pieces of the GPU parity tests: building the library, creating a
solver and an oracle from the same seeded state, and the error measures."""
import numpy as np
import pytest

import oracle as O
from paper_2608_21607_gb300 import nmd as N
from paper_2608_21607_gb300 import workloads as WL

# per-step agreement (relative Frobenius error) by precision: fp32-accurate
# paths 1e-4, bf16 operands 5e-3
TOL = {N.NMD_SIMT: 1e-4, N.NMD_FP32: 1e-4, N.NMD_BF16: 5e-3}
PREC_NAMES = {N.NMD_SIMT: "simt", N.NMD_FP32: "fp32", N.NMD_BF16: "bf16"}


def require_gpu():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_21607_gb300 import build
    build.build()
    return torch


def rel(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    nb = np.linalg.norm(b)
    return float(np.linalg.norm(a - b) / (nb if nb > 0 else 1.0))


def make_pair(S, r, W, H, *, block_rows, block_cols, precision, epilogue=N.NMD_EPI_Z,
              schedule=N.NMD_STOCH, eta=0.5, gamma=0.9, seed=0, order=N.NMD_ALTERNATE, EW=None,
              EH=None, skip_zero_chunks=False):
    """A GPU solver and an oracle state holding the same factors and momentum."""
    sol = N.Solver(S, r, block_rows=block_rows, block_cols=block_cols, schedule=schedule,
                   order=order, eta=eta, gamma=gamma, precision=precision, epilogue=epilogue,
                   seed=seed, skip_zero_chunks=skip_zero_chunks)
    W = np.ascontiguousarray(W, np.float32)
    H = np.ascontiguousarray(H, np.float32)
    if EW is None:
        sol.set_factors(W, H)
    else:
        sol.set_state(W, H, EW, EH, 0)
    orc = O.State(S, W.astype(np.float64), H.astype(np.float64),
                  O.Options(block_rows=block_rows, block_cols=block_cols,
                            schedule=O.EXACT if schedule == N.NMD_EXACT else O.STOCH,
                            order=order, eta=eta, gamma=gamma, seed=seed))
    if EW is not None:
        orc.EA[:] = EW
        orc.EB[:] = np.asarray(EH, np.float64).T
    return sol, orc


def sync_oracle_to(sol, orc):
    """Teacher forcing: load the solver's current state into the oracle."""
    W, H, EW, EH, sweep = sol.get_state()
    orc.A[:] = W
    orc.B[:] = H.T
    orc.EA[:] = EW
    orc.EB[:] = EH.T
    orc.sweep_index = sweep


# scaled-down stand-ins of the five workloads: same generators, several tiles
# and a ragged last block on both sides, blocks of at least 10 r rows (the
# full workloads have 32 r to 170 r): with fewer, the block Gram matrices of
# the stochastic steps become near-singular
def small_cases():
    cases = []
    S, _, _, _ = WL.planted(600, 400, 4, tau=0.5, seed=0)
    W, H = WL.init_factors(600, 400, 4, 0)
    cases.append(("planted600x400_r4_exact", S, 4, W, H, 128, 128, N.NMD_EXACT))
    S = WL.identity(1000)
    W, H = WL.init_factors(1000, 1000, 3, 1)
    cases.append(("identity1000_r3", S, 3, W, H, 192, 192, N.NMD_STOCH))
    S, _, _, _ = WL.planted(1500, 1300, 32, tau=None, density=0.05, noise=0.01, seed=2)
    W, H = WL.init_factors(1500, 1300, 32, 2)
    cases.append(("planted1500x1300_r32", S, 32, W, H, 320, 288, N.NMD_STOCH))
    S = WL.connectome(4000, seed=3)
    W, H = WL.init_factors(4000, 4000, 64, 3)
    cases.append(("connectome4000_r64", S, 64, W, H, 1024, 1024, N.NMD_STOCH))
    S = WL.connectome(3400, seed=4)
    W, H = WL.init_factors(3400, 3400, 100, 4)
    cases.append(("connectome3400_r100", S, 100, W, H, 1000, 1000, N.NMD_STOCH))
    S = WL.connectome(6000, seed=5)
    W, H = WL.init_factors(6000, 6000, 256, 5)
    cases.append(("connectome6000_r256", S, 256, W, H, 2560, 2560, N.NMD_STOCH))
    return cases
