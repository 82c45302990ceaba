"""Writes partition_boundaries.txt from the oracle alone (oracle/partition.py).

Run from the repository root:  python tests/golden/make_golden.py
The cases are the five workloads' (seq_len, chunks) pairs plus ragged extras.
"""
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

from oracle import partition as P  # noqa: E402

CASES = [
    (1024, 4, 128, P.UNIFORM),
    (8192, 8, 128, P.UNIFORM),
    (32768, 16, 128, P.LBCP),
    (32768, 16, 128, P.UNIFORM),
    (131072, 32, 128, P.LBCP),
    (131072, 32, 128, P.UNIFORM),
    (2048, 1, 128, P.LBCP),
    (4096, 2, 128, P.LBCP),
    (10240, 5, 128, P.LBCP),
    (23936, 12, 128, P.LBCP),
    (1000, 3, 128, P.LBCP),
    (1000, 7, 128, P.LBCP),
    (640, 5, 128, P.LBCP),
    (100000, 9, 64, P.LBCP),
]


def main():
    out = os.path.join(os.path.dirname(os.path.abspath(__file__)), "partition_boundaries.txt")
    with open(out, "w") as f:
        f.write("# seq_len chunks granularity mode(0=uniform,1=lbcp): b_0 .. b_M\n")
        f.write("# written by tests/golden/make_golden.py from oracle/partition.py\n")
        for s, m, g, mode in CASES:
            b = P.boundaries(s, m, g, mode)
            f.write(f"{s} {m} {g} {mode}: " + " ".join(str(x) for x in b) + "\n")


if __name__ == "__main__":
    main()
