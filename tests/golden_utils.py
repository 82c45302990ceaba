"""Readers of the committed fixtures under tests/golden/ (plain text)."""

import os

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def dp_tie_case():
    """The hand-worked Algorithm 1 stage-1 case: (case parameters, states
    {(m, s): (k, t_max, t_sum)}, terminal (m, s, t_max, t_sum), boundaries)."""
    case, states, terminal, bounds = {}, {}, None, None
    with open(os.path.join(GOLDEN, "dp_tie_case.txt")) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            key, val = line.split(":", 1)
            if key == "case":
                case = {k: int(v) for k, v in (x.split("=") for x in val.split())}
            elif key == "state":
                m, s, k, tmax, tsum = (int(x) for x in val.split())
                states[(m, s)] = (k, tmax, tsum)
            elif key == "terminal":
                terminal = tuple(int(x) for x in val.split())
            elif key == "boundaries":
                bounds = [int(x) for x in val.split()]
    return case, states, terminal, bounds


def dp_boundary_rows():
    """Rows of dp_boundaries.txt: (seq_len, chunks, granularity, stages,
    model, gemm_weight, boundaries)."""
    rows = []
    with open(os.path.join(GOLDEN, "dp_boundaries.txt")) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            head, tail = line.split(":", 1)
            s, m, g, n, model, gemm = (int(x) for x in head.split())
            rows.append((s, m, g, n, model, gemm, [int(x) for x in tail.split()]))
    return rows


def dp_latency_rows():
    """Rows of dp_latency_boundaries.txt: ((seq_len, chunks, stages, Hq, Hkv,
    d, sms, window), boundaries)."""
    rows = []
    with open(os.path.join(GOLDEN, "dp_latency_boundaries.txt")) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            head, tail = line.split(":", 1)
            rows.append((tuple(int(x) for x in head.split()), [int(x) for x in tail.split()]))
    return rows
