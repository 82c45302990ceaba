"""Float64 oracle for the fused QKV projection + rotary embedding + KV append
(TEST INFRASTRUCTURE; see ``oracle/__init__.py``).

Sec. 3.2 / Eq. 1 splits each chunk's cost into attention and GEMM work that
grows with the chunk length (QKV projection, output projection, FFN).  The
QKV projection of a chunk is ``[Q | K | V] = X W^T``.  The paper's models
(Llama3 family, Sec. 5.1) rotate Q and K by the rotary position embedding
before attention; the paper does not spell it out, so this is the reading:

* rotate-half convention: for a head vector x of dimension d and
  j in [0, d/2), with angle a = pos * theta^(-2 j / d),
  x'[j] = x[j] cos a - x[j + d/2] sin a,  x'[j + d/2] = x[j + d/2] cos a + x[j] sin a;
* positions are the tokens' global indices (chunk offset + row);
* V is not rotated.
"""

from __future__ import annotations

import numpy as np


def rope(x: np.ndarray, pos: np.ndarray, theta: float) -> np.ndarray:
    """Rotate head vectors x [n, H, d] (float64) at positions pos [n]."""
    d = x.shape[-1]
    half = d // 2
    inv = theta ** (-2.0 * np.arange(half, dtype=np.float64) / d)
    ang = np.asarray(pos, dtype=np.float64)[:, None] * inv[None, :]    # [n, d/2]
    c = np.cos(ang)[:, None, :]
    s = np.sin(ang)[:, None, :]
    x0, x1 = x[..., :half], x[..., half:]
    return np.concatenate([x0 * c - x1 * s, x1 * c + x0 * s], axis=-1)


def qkv_rope(x, w, n_q_heads, n_kv_heads, head_dim, pos0, theta):
    """x [len, hidden], w [(Hq + 2 Hkv) d, hidden] (float64).  Returns
    Q [len, Hq, d] and K [len, Hkv, d] rotated at positions pos0 + r, and V."""
    n = x.shape[0]
    y = x @ w.T
    qc = n_q_heads * head_dim
    kc = n_kv_heads * head_dim
    q = y[:, :qc].reshape(n, n_q_heads, head_dim)
    k = y[:, qc:qc + kc].reshape(n, n_kv_heads, head_dim)
    v = y[:, qc + kc:qc + 2 * kc].reshape(n, n_kv_heads, head_dim)
    pos = pos0 + np.arange(n)
    return rope(q, pos, theta), rope(k, pos, theta), v
