"""Float64 oracle for chunked causal GQA prefill attention (TEST INFRASTRUCTURE).

Test infrastructure only (see ``oracle/__init__.py``); the product path never
imports this module.

What the paper fixes (Sec. 2.2, Sec. 3.2 / Eq. 1): a long prompt is split into
chunks; chunk ``i`` covers global positions ``[b_i, b_{i+1})`` and its queries
attend to the keys/values of every earlier chunk plus a causal block over the
chunk itself.  The KV of earlier chunks stays live for later chunks (Sec. 2.2,
Sec. 3.1).  Chunking therefore never changes the result: chunk attention is
plain causal attention restricted to the chunk's rows.

Readings taken where the paper is silent:

* GQA: query head ``h`` reads KV head ``h // (Hq // Hkv)``.
* Row ``t`` (global position) sees keys ``0..t`` inclusive.
* ``s_j = scale * q_t . k_j``;  ``O_t = sum_j softmax(s)_j v_j``;
  ``LSE_t = ln sum_j exp(s_j)`` (natural log of the scaled scores).
* Layouts: Q/O ``[rows, Hq, d]``, K/V ``[rows, Hkv, d]``, LSE ``[Hq, rows]``.

All arithmetic is float64.  Inputs are expected to hold exactly the bf16
values the device consumed (see :func:`bf16_bits_to_f64`).  Rows are evaluated
independently, straight from the definition; iterating over rows in blocks
only bounds memory and changes no arithmetic.
"""

from __future__ import annotations

import numpy as np

_ROW_BLOCK = 256


def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact widening of raw bf16 bit patterns (uint16/int16) to float64."""
    u = np.ascontiguousarray(bits).view(np.uint16).astype(np.uint32) << 16
    return u.view(np.float32).astype(np.float64)


def kv_append(cache: np.ndarray, chunk: np.ndarray, offset: int) -> np.ndarray:
    """KV-cache append (Sec. 2.2, Sec. 3.1): rows ``[offset, offset+len)`` of
    the cache become the chunk's rows; every other row is unchanged.  Works on
    any dtype (bit patterns included) and returns a new array."""
    out = cache.copy()
    out[offset:offset + chunk.shape[0]] = chunk
    return out


def _rows_for_head(q_rows, pos, k, v, scale):
    """Causal softmax attention for the given query rows of one head.

    q_rows [n, d] float64, pos [n] global positions, k/v [T, d] with
    T > max(pos).  Returns (o [n, d], lse [n]).
    """
    t_max = int(pos.max()) + 1
    s = scale * (q_rows @ k[:t_max].T)                       # [n, T]
    visible = np.arange(t_max)[None, :] <= pos[:, None]       # key j <= t
    s = np.where(visible, s, -np.inf)
    m = s.max(axis=1, keepdims=True)
    e = np.exp(s - m)
    l = e.sum(axis=1, keepdims=True)
    o = (e @ v[:t_max]) / l
    lse = m[:, 0] + np.log(l[:, 0])
    return o, lse


def chunk_attention(q_chunk, k_cache, v_cache, prefix, scale, rows=None, heads=None):
    """Attention of one chunk against the KV prefix plus itself (Sec. 2.2).

    q_chunk  [len, Hq, d] float64 -- the chunk's queries, global rows
             ``prefix .. prefix+len-1``.
    k_cache, v_cache [>= prefix+len, Hkv, d] float64 -- KV of all rows so far.
    rows     optional 1-D array of chunk-local row indices to evaluate
             (sampling); default all rows.
    heads    optional list of query heads to evaluate (sampling); default
             all Hq heads.  Each head is computed exactly as in the full call.
    Returns (O [n, H, d], LSE [H, n]) for the n requested rows and the H
    requested heads, in the order given.
    """
    length, n_q, d = q_chunk.shape
    n_kv = k_cache.shape[1]
    if n_q % n_kv:
        raise ValueError("Hq must be a multiple of Hkv")
    group = n_q // n_kv
    if rows is None:
        rows = np.arange(length)
    rows = np.asarray(rows, dtype=np.int64)
    if k_cache.shape[0] < prefix + (int(rows.max()) + 1 if rows.size else 0):
        raise ValueError("cache shorter than prefix + rows")
    heads = list(range(n_q)) if heads is None else [int(h) for h in heads]
    if any(h < 0 or h >= n_q for h in heads):
        raise ValueError("head index out of range")
    out = np.zeros((rows.size, len(heads), d), dtype=np.float64)
    lse = np.zeros((len(heads), rows.size), dtype=np.float64)
    for j, h in enumerate(heads):
        g = h // group
        for a in range(0, rows.size, _ROW_BLOCK):
            r = rows[a:a + _ROW_BLOCK]
            o_b, l_b = _rows_for_head(q_chunk[r, h, :], prefix + r,
                                      k_cache[:, g, :], v_cache[:, g, :], scale)
            out[a:a + r.size, j, :] = o_b
            lse[j, a:a + r.size] = l_b
    return out, lse


def causal_attention(q, k, v, scale, rows=None):
    """Unchunked causal attention over a whole sequence (the chunk == 0..S case)."""
    return chunk_attention(q, k, v, 0, scale, rows)


def chunked_prefill(q, k, v, bounds, scale):
    """Walk the chunks in order as the pipelined prefill does (Sec. 2.2): append
    chunk ``i``'s KV to the cache, then attend chunk ``i``'s queries to the
    cache.  Returns (O [S, Hq, d], list of per-chunk LSE [Hq, c_i], cache_k,
    cache_v)."""
    seq, n_q, d = q.shape
    ck = np.zeros_like(k)
    cv = np.zeros_like(v)
    outs, lses = [], []
    for i in range(len(bounds) - 1):
        b0, b1 = bounds[i], bounds[i + 1]
        ck = kv_append(ck, k[b0:b1], b0)
        cv = kv_append(cv, v[b0:b1], b0)
        o, l = chunk_attention(q[b0:b1], ck[:b1], cv[:b1], b0, scale)
        outs.append(o)
        lses.append(l)
    return np.concatenate(outs, axis=0), lses, ck, cv


def combine_partials(o_parts, lse_parts):
    """Merge attention results computed over disjoint key sets.

    o_parts [P, n, H, d], lse_parts [P, H, n]: part p holds the normalised
    output and log-sum-exp of the same rows over its own key subset.  The
    softmax over the union weighs each part by ``exp(LSE_p - LSE)`` with
    ``LSE = ln sum_p exp(LSE_p)``.  Parts with LSE = -inf (no keys) get weight 0.
    """
    o_parts = np.asarray(o_parts, dtype=np.float64)
    lse_parts = np.asarray(lse_parts, dtype=np.float64)
    m = lse_parts.max(axis=0)                                 # [H, n]
    w = np.exp(lse_parts - m[None])                           # [P, H, n]
    total = w.sum(axis=0)
    lse = m + np.log(total)
    w = w / total[None]
    o = np.einsum("phn,pnhd->nhd", w, o_parts)
    return o, lse
