"""Writes the stored expected values under tests/golden/ that come from the oracle.

Calls only ``oracle`` (and the seeded input generators).  Run from the repo
root:  python tests/golden/make_golden.py
"""
import os
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))

import oracle as O  # noqa: E402


def block_order():
    # (seed, sweep, side, K): the block counts of the five workloads
    # (600/128 -> 5, 400/128 -> 4, 4096/512 -> 8, 20000/2048 -> 10,
    #  139255/4096 -> 34, 139255/8192 -> 17) and a few other seeds.
    cases = []
    for seed in (0, 1, 12345):
        for sweep in (0, 1, 2, 9, 199):
            for side in (0, 1):
                for K in (1, 2, 4, 5, 8, 10, 17, 34):
                    cases.append((seed, sweep, side, K))
    cases.append((2 ** 64 - 1, 2 ** 40, 1, 300))
    lines = ["# seed sweep side K  permutation...  (oracle.block_permutation)"]
    for c in cases:
        p = O.block_permutation(*c)
        lines.append(" ".join(str(x) for x in list(c) + p))
    with open(os.path.join(HERE, "block_order.txt"), "w") as f:
        f.write("\n".join(lines) + "\n")


if __name__ == "__main__":
    block_order()
