"""Parity at the full size of the connectome-shaped workloads (139,255 x
139,255, 2,785,100 nonzeros; r = 64 with blocks of 4096, r = 256 with blocks
of 8192), with the step sizes the benchmark uses.  Each checked step starts
from the GPU's current state (teacher forcing) and is compared with the
oracle's full step: every one of the 139,255 updated rows, element by
element (relative Frobenius error), and the momentum.  The benchmark times
these steps inside sweeps; a sweep gives bit for bit the factors of the
same steps run one by one (test_gpu_parity.py), so the serial block updates
here check the same arithmetic.  Each test takes seconds on the GPU and up
to about ten on the host cores for the oracle's full steps."""
import gc

import numpy as np
import pytest

from gpu_common import TOL, make_pair, rel, require_gpu, sync_oracle_to
from paper_2608_21607_gb300 import nmd as N
from paper_2608_21607_gb300 import workloads as WL

pytestmark = [pytest.mark.gpu, pytest.mark.slow]   # collected after every other test file (file name)


@pytest.fixture(scope="module", autouse=True)
def gpu():
    return require_gpu()


@pytest.fixture(scope="module")
def wl64():
    return WL.workload("connectome_r64")


@pytest.fixture(scope="module")
def wl256():
    return WL.workload("connectome_r256")


def _check_steps(wl, precision, epilogue, pick):
    """pick(orc) -> the (side, block, kind) steps to check, in order."""
    sol, orc = make_pair(wl.S, wl.r, wl.W0, wl.H0, block_rows=wl.block_rows, block_cols=wl.block_cols,
                         precision=precision, epilogue=epilogue, eta=wl.eta, gamma=wl.gamma)
    try:
        for side, block, kind in pick(orc):
            sync_oracle_to(sol, orc)
            sol.block_update(side, block, kind)
            orc.block_update(side, block, kind)
            W, H, EW, EH, _ = sol.get_state()
            M, E, (m0, m1), _, _, _ = orc._roles(side, block, kind)
            got = (W if M is orc.A else H.T)[m0:m1]
            gotE = (EW if M is orc.A else EH.T)[m0:m1]
            err = rel(got, M[m0:m1])
            assert err <= TOL[precision], (wl.name, side, block, err)
            assert rel(gotE, E[m0:m1]) <= 10 * TOL[precision], (wl.name, side, block)
            assert np.isfinite(got).all()
    finally:
        del sol
        gc.collect()


def test_connectome_r64_bf16_z_full_size(wl64):
    """The benchmark's configuration: the first two steps of sweep 0 (one of
    each side) and the ragged last column block (4087 rows)."""
    last = -(-wl64.n // wl64.block_cols) - 1
    _check_steps(wl64, N.NMD_BF16, N.NMD_EPI_Z,
                 lambda orc: orc.sweep_steps(0)[:2] + [(N.NMD_COL, last, N.NMD_STOCH)])


def test_connectome_r64_fp32_full_size(wl64):
    _check_steps(wl64, N.NMD_FP32, N.NMD_EPI_Z, lambda orc: orc.sweep_steps(0)[:1])


def test_connectome_r64_bf16_delta_full_size(wl64):
    _check_steps(wl64, N.NMD_BF16, N.NMD_EPI_DELTA, lambda orc: orc.sweep_steps(0)[:1])


def test_connectome_r256_bf16_full_size(wl256):
    _check_steps(wl256, N.NMD_BF16, N.NMD_EPI_Z, lambda orc: orc.sweep_steps(0)[:1])
