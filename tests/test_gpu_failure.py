"""Failure detection on the GPU without a fault: every pipeline wait of the
tensor-core kernels is an mbarrier poll bounded by a timer.  The self-test
runs that wait on a barrier nothing arrives at (the flag that nothing sets)
with a short limit; the kernel must give up, record NMD_ERR_TIMEOUT in the
sticky status and return, and the handle must stay usable afterwards."""
import numpy as np
import pytest

from gpu_common import make_pair, rel, require_gpu
from paper_2608_21607_gb300 import nmd as N
from paper_2608_21607_gb300 import workloads as WL

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def gpu():
    return require_gpu()


def _pair():
    S = WL.connectome(1500, seed=9)
    W, H = WL.init_factors(1500, 1500, 32, 9)
    return make_pair(S, 32, W, H, block_rows=320, block_cols=320, precision=N.NMD_BF16)


def test_bounded_wait_times_out_and_the_handle_recovers():
    sol, orc = _pair()
    assert N.nmd_selftest_wait_timeout(sol.h, 10_000_000) == N.NMD_ERR_TIMEOUT      # 10 ms
    assert N.nmd_selftest_wait_timeout(sol.h, 1_000_000) == N.NMD_ERR_TIMEOUT       # twice in a row
    # the status was read and cleared: a block step still agrees with the oracle
    sol.block_update(N.NMD_COL, 1, N.NMD_STOCH)
    orc.block_update(N.NMD_COL, 1, N.NMD_STOCH)
    W, _ = sol.get_factors()
    assert rel(W, orc.A) <= 5e-3
    assert np.isfinite(sol.loss()["obj"])


def test_selftest_rejects_limits_out_of_range():
    sol, _ = _pair()
    assert N.nmd_selftest_wait_timeout(sol.h, 0) == N.NMD_ERR_INVALID
    assert N.nmd_selftest_wait_timeout(sol.h, 5_000_000_000) == N.NMD_ERR_INVALID
    sol.sync()
