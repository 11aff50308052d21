"""Writes tests/golden/branch_alloc.txt from the oracle's Sec. IV-C allocator.

Each line: B_alloc gamma alpha beta F_0 ... F_{gamma-1}.  The first line is the
per-depth budget of the 128256-vocabulary workload (B_alloc = 64, gamma = 16,
alpha = 0.9, beta = 1).  Calls only the oracle package.
"""
import os
import sys

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__)))))
from oracle import oracle as O  # noqa: E402

CASES = [(64, 16, 0.9, 1.0), (40, 8, 0.6, 0.5), (20, 4, 0.8, 1.0), (80, 16, 0.7, 1.0)]

if __name__ == "__main__":
    out = os.path.join(os.path.dirname(os.path.abspath(__file__)), "branch_alloc.txt")
    with open(out, "w") as f:
        f.write("# B_alloc gamma alpha beta F_0..F_{gamma-1}; Eq. for F*_k in Sec. IV-C,\n")
        f.write("# floor + largest remainder (ties to the shallower depth)\n")
        for c in CASES:
            _, ints = O.branch_alloc(*c)
            f.write(" ".join([str(c[0]), str(c[1]), repr(c[2]), repr(c[3])] + [str(x) for x in ints]) + "\n")
