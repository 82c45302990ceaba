"""Shared helpers for the GPU parity tests: bf16 bits -> float64, row
sampling, oracle evaluation of sampled rows, and the tolerances."""

import numpy as np
import torch

from oracle import attention as A

# Output and LSE tolerances (bf16 output, fp32 statistics).
O_MAX_ABS = 2e-2
O_MEAN_ABS = 2e-3
LSE_MAX_ABS = 1e-3


def f64(t: torch.Tensor) -> np.ndarray:
    return A.bf16_bits_to_f64(t.detach().contiguous().cpu().view(torch.int16).numpy())


def sample_rows(length: int, every: int = 97, edge: int = 3, seed: int = 0) -> np.ndarray:
    """First/last rows, rows around each 128-row tile boundary, a stride, and a
    few random rows -- sorted and unique."""
    rows = set(range(min(edge, length))) | set(range(max(0, length - edge), length))
    for b in range(128, length, 128):
        rows |= {b - 1, b}
    rows |= set(range(0, length, every))
    rng = np.random.default_rng(seed)
    rows |= set(int(x) for x in rng.integers(0, length, size=min(8, length)))
    return np.array(sorted(r for r in rows if 0 <= r < length), dtype=np.int64)


def compare(o_gpu: np.ndarray, lse_gpu: np.ndarray, o_ref: np.ndarray, lse_ref: np.ndarray):
    err = np.abs(o_gpu.astype(np.float64) - o_ref)
    lerr = np.abs(lse_gpu.astype(np.float64) - lse_ref)
    return float(err.max()), float(err.mean()), float(lerr.max())


def assert_close(o_gpu, lse_gpu, o_ref, lse_ref, what=""):
    assert np.all(np.isfinite(o_gpu)) and np.all(np.isfinite(lse_gpu)), what
    mx, mean, lmx = compare(o_gpu, lse_gpu, o_ref, lse_ref)
    assert mx <= O_MAX_ABS, f"{what}: O max-abs {mx:.3e}"
    assert mean <= O_MEAN_ABS, f"{what}: O mean-abs {mean:.3e}"
    assert lmx <= LSE_MAX_ABS, f"{what}: LSE max-abs {lmx:.3e}"
    return mx, mean, lmx


def chunk_rows_oracle(q_rows, kf, vf, prefix, rows, scale, heads=None):
    """Oracle for chunk-local `rows` whose queries were gathered into q_rows
    (all heads, or the listed `heads` in that order)."""
    q_full = np.zeros((int(rows.max()) + 1,) + q_rows.shape[1:])
    q_full[rows] = q_rows
    return A.chunk_attention(q_full, kf, vf, prefix, scale, rows=rows, heads=heads)


def check_single_request(pf, q, k, v, rows_fn=None, chunks=None, heads_fn=None, out=None,
                         lse_of_chunk=None):
    """Oracle check of a single-request ChunkedPrefill on the rows
    ``rows_fn(len, chunk)`` of every chunk (all rows by default) and the heads
    ``heads_fn(chunk)`` (all by default).  ``out`` / ``lse_of_chunk`` replace
    the prefill's own output buffer and per-chunk LSE view."""
    b = pf.bounds[0]
    out = pf.out if out is None else out
    lse_of_chunk = pf.chunk_lse if lse_of_chunk is None else lse_of_chunk
    kf, vf = f64(k), f64(v)
    worst = (0.0, 0.0, 0.0)
    for i in (range(len(b) - 1) if chunks is None else chunks):
        b0, b1 = b[i], b[i + 1]
        rows = np.arange(b1 - b0) if rows_fn is None else rows_fn(b1 - b0, i)
        heads = None if heads_fn is None else list(heads_fn(i))
        idx = torch.as_tensor(rows, device=q.device)
        o_ref, lse_ref = chunk_rows_oracle(f64(q[b0:b1][idx]), kf[:b1], vf[:b1], b0, rows,
                                           pf.w.scale, heads)
        o_gpu = out[b0:b1][idx]
        lse_gpu = lse_of_chunk(i)[:, idx]
        if heads is not None:
            o_gpu, lse_gpu = o_gpu[:, heads], lse_gpu[heads]
        r = assert_close(o_gpu.float().cpu().numpy(), lse_gpu.cpu().numpy(), o_ref, lse_ref,
                         f"chunk {i} [{b0},{b1})")
        worst = tuple(max(a, c) for a, c in zip(worst, r))
    return worst


def rotating_heads(n_q_heads, count=4):
    """`count` query heads for chunk i, rotating with i so that the chunks of a
    prompt together cover every head, every KV group and every head slot."""
    def heads(i):
        return sorted({(9 * i + 21 * j) % n_q_heads for j in range(count)})
    return heads
