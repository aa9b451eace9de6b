"""fp64 CPU oracle of the SALSA block sweep -- test infrastructure only.

Imported by ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg
of ``bench.py``; the CUDA library and its Python binding never import it.
"""
from .salsa import *  # noqa: F401,F403
from .salsa import (ROW, COL, EXACT, STOCH, ALTERNATE, PHASED, NotSPD, Options, State,  # noqa: F401
                    Sparse, block_permutation, block_range, num_blocks, cholesky,
                    solve_normal, update_z, loss, splitmix64_mix, SplitMix64,
                    positive_set, range_search_set)
from . import embed  # noqa: F401,E402  (Sec. 5.3: cell embedding and 1-NN error)
