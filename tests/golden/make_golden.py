"""Writes the partition fixtures from the oracle alone (oracle/partition.py).

Run from the repository root:  python tests/golden/make_golden.py
  partition_boundaries.txt  the closed-form split of the five workloads'
                            (seq_len, chunks) pairs plus ragged extras
  dp_boundaries.txt         Algorithm 1's stage-1 DP on the 32768-token /
                            16-chunk and 131072-token / 32-chunk shapes
                            (N = 16 stages; causal cost, Eq. 1's cost, and
                            the causal cost with a GEMM weight of 90)
  dp_latency_boundaries.txt the same DP with the attention kernel's latency
                            model (N = 16, 152 SMs; 32/8 and 64/8 heads,
                            d = 128; windows of 6 and 8 units)
The DP rows of the 131072-token shape take several minutes of pure Python.
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

# (seq_len, chunks, granularity, stages, cost model, gemm weight)
DP_CASES = [
    (32768, 16, 128, 16, P.COST_CAUSAL, 0),
    (32768, 16, 128, 16, P.COST_EQ1, 0),
    (32768, 16, 128, 16, P.COST_CAUSAL, 90),
    (131072, 32, 128, 16, P.COST_CAUSAL, 0),
    (131072, 32, 128, 16, P.COST_EQ1, 0),
    (131072, 32, 128, 16, P.COST_CAUSAL, 90),
]


# (seq_len, chunks, stages, Hq, Hkv, d, SMs, window)
DP_LATENCY_CASES = [
    (32768, 16, 16, 32, 8, 128, 152, 6),
    (131072, 32, 16, 64, 8, 128, 152, 8),
]


def main():
    here = os.path.dirname(os.path.abspath(__file__))
    with open(os.path.join(here, "partition_boundaries.txt"), "w") as f:
        f.write("# seq_len chunks granularity mode(0=uniform,1=lbcp): b_0 .. b_M\n")
        f.write("# written by tests/golden/make_golden.py from oracle/partition.py\n")
        for s, m, g, mode in CASES:
            b = P.boundaries(s, m, g, mode)
            f.write(f"{s} {m} {g} {mode}: " + " ".join(str(x) for x in b) + "\n")
    with open(os.path.join(here, "dp_boundaries.txt"), "w") as f:
        f.write("# seq_len chunks granularity stages model(0=causal,1=eq1) gemm_weight: "
                "b_0 .. b_M\n")
        f.write("# written by tests/golden/make_golden.py from oracle/partition.py "
                "(dp_boundaries)\n")
        for s, m, g, n, model, gemm in DP_CASES:
            b = P.dp_boundaries(s, m, g, n, model, gemm)
            f.write(f"{s} {m} {g} {n} {model} {gemm}: " + " ".join(str(x) for x in b) + "\n")
            f.flush()
    with open(os.path.join(here, "dp_latency_boundaries.txt"), "w") as f:
        f.write("# seq_len chunks stages n_q_heads n_kv_heads head_dim sms window: b_0 .. b_M\n")
        f.write("# written by tests/golden/make_golden.py from oracle/partition.py "
                "(dp_latency_boundaries)\n")
        for case in DP_LATENCY_CASES:
            b = P.dp_latency_boundaries(*case)
            f.write(" ".join(str(x) for x in case) + ": " + " ".join(str(x) for x in b) + "\n")
            f.flush()


if __name__ == "__main__":
    main()
