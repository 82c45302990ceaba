"""GB300-native (sm_103a) chunked causal prefill attention -- the hot path of
MOCAP's prefill-only method (arXiv 2606.22968), behind a C ABI.

The functions below carry the C entry points' names and only marshal
arguments (torch tensors -> device pointers, streams -> handles); all work
runs in ``libmocap.so``.  There is no CPU fallback: a missing or unbuildable
library raises.
"""

from __future__ import annotations

import ctypes
from typing import List, Sequence

from . import _lib
from ._lib import AppendItem, CopyItem, VarlenItem

MOCAP_OK, MOCAP_EINVAL, MOCAP_ECUDA, MOCAP_EUNSUPPORTED, MOCAP_ETIMEOUT = 0, 1, 2, 3, 4
MOCAP_PART_UNIFORM, MOCAP_PART_LBCP = 0, 1
MOCAP_VARLEN_MAX_ITEMS = 64
MOCAP_VARLEN_DEV_MAX_ITEMS = 65536
MOCAP_FUSED_APPEND_MAX = 64
MOCAP_COPY_MAX_ITEMS = 8


class MocapError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        msg = _lib.load().mocap_status_string(status)
        super().__init__(f"{where}: {msg.decode() if msg else status}")


def _check(status: int, where: str):
    if status != MOCAP_OK:
        raise MocapError(status, where)


def _ptr(t) -> int:
    if t is None:
        return 0
    if isinstance(t, int):
        return t
    if not t.is_cuda:
        raise ValueError("expected a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError("expected a contiguous tensor")
    return t.data_ptr()


def _stream(stream) -> int:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def mocap_lbcp_partition(seq_len: int, num_chunks: int, granularity: int = 128,
                         mode: int = MOCAP_PART_LBCP) -> List[int]:
    out = (ctypes.c_int64 * (num_chunks + 1))()
    _check(_lib.load().mocap_lbcp_partition(seq_len, num_chunks, granularity, mode, out),
           "mocap_lbcp_partition")
    return list(out)


MOCAP_COST_CAUSAL, MOCAP_COST_EQ1 = 0, 1


def mocap_lbcp_partition_dp(seq_len: int, num_chunks: int, granularity: int = 128,
                            num_stages: int = 16, model: int = MOCAP_COST_CAUSAL,
                            gemm_weight: int = 0) -> List[int]:
    """Boundaries from the stage-1 dynamic program of Algorithm 1."""
    out = (ctypes.c_int64 * (num_chunks + 1))()
    _check(_lib.load().mocap_lbcp_partition_dp(seq_len, num_chunks, granularity, num_stages,
                                               model, gemm_weight, out),
           "mocap_lbcp_partition_dp")
    return list(out)


def mocap_lbcp_partition_dp_latency(seq_len: int, num_chunks: int, n_q_heads: int,
                                    n_kv_heads: int, head_dim: int, num_sms: int,
                                    num_stages: int = 16, window: int = 8) -> List[int]:
    """Boundaries from Algorithm 1's stage-1 DP with the attention kernel's
    compute-latency model as EvaluateChunk (128-row units, each boundary
    within `window` units of the closed-form split)."""
    out = (ctypes.c_int64 * (num_chunks + 1))()
    _check(_lib.load().mocap_lbcp_partition_dp_latency(seq_len, num_chunks, num_stages,
                                                       n_q_heads, n_kv_heads, head_dim, num_sms,
                                                       window, out),
           "mocap_lbcp_partition_dp_latency")
    return list(out)


def mocap_lbcp_gemm_weight(attn_s_per_pair: float, gemm_s_per_row: float,
                           granularity: int = 128) -> int:
    """The stage-1 DP's GEMM weight for chunk stages that cost
    ``a * pairs + b * rows`` (a = attention seconds per causal pair, b =
    projection seconds per row)."""
    out = ctypes.c_int64(0)
    st = _lib.load().mocap_lbcp_gemm_weight(float(attn_s_per_pair), float(gemm_s_per_row),
                                            granularity, ctypes.byref(out))
    if st == MOCAP_EINVAL:
        raise ValueError("attn_s_per_pair > 0 and gemm_s_per_row >= 0 required")
    _check(st, "mocap_lbcp_gemm_weight")
    return out.value


def mocap_kv_append(k_chunk, v_chunk, k_cache, v_cache, offset: int, stream=None):
    """Copy chunk K/V ([len, Hkv, d] bf16) into cache rows [offset, offset+len)."""
    length, n_kv, d = k_chunk.shape
    _check(_lib.load().mocap_kv_append(_ptr(k_chunk), _ptr(v_chunk), _ptr(k_cache), _ptr(v_cache),
                                       k_cache.shape[0], offset, length, n_kv, d,
                                       _stream(stream)), "mocap_kv_append")


def mocap_kv_append_overlap(k_chunk, v_chunk, k_cache, v_cache, offset: int, stream=None):
    """mocap_kv_append with a kernel that runs beside a concurrent attention
    launch (for a second stream)."""
    length, n_kv, d = k_chunk.shape
    _check(_lib.load().mocap_kv_append_overlap(_ptr(k_chunk), _ptr(v_chunk), _ptr(k_cache),
                                               _ptr(v_cache), k_cache.shape[0], offset, length,
                                               n_kv, d, _stream(stream)),
           "mocap_kv_append_overlap")


def _copy_array(pairs, to_host):
    arr = (CopyItem * max(1, len(pairs)))()
    for i, (dst, src) in enumerate(pairs):
        nbytes = dst.numel() * dst.element_size()
        if src.numel() * src.element_size() != nbytes:
            raise ValueError("copy source and destination differ in size")
        if not dst.is_contiguous() or not src.is_contiguous():
            raise ValueError("copy tensors must be contiguous")
        if (dst.is_cuda, src.is_cuda) != ((False, True) if to_host else (True, False)):
            raise ValueError("copies go between host and device tensors in the named direction")
        arr[i] = CopyItem(dst.data_ptr() if nbytes else None, src.data_ptr() if nbytes else None,
                          nbytes)
    return arr


def mocap_copy_from_host(pairs, beside_kernels: bool = False, stream=None):
    """Host -> device copies by the SMs: ``pairs`` is a sequence of up to
    MOCAP_COPY_MAX_ITEMS (device_tensor, pinned_host_tensor) of equal byte
    size, each contiguous."""
    _check(_lib.load().mocap_copy_from_host(_copy_array(pairs, False), len(pairs),
                                            int(bool(beside_kernels)), _stream(stream)),
           "mocap_copy_from_host")


def mocap_copy_to_host(pairs, beside_kernels: bool = False, stream=None):
    """Device -> host copies by the SMs: ``pairs`` of (pinned_host_tensor,
    device_tensor)."""
    _check(_lib.load().mocap_copy_to_host(_copy_array(pairs, True), len(pairs),
                                          int(bool(beside_kernels)), _stream(stream)),
           "mocap_copy_to_host")


def mocap_qkv_rope_append(x, w_qkv, q_out, k_cache, v_cache, offset: int,
                          rope_theta: float = 500000.0, stream=None):
    """[Q|K|V] = x w_qkv^T, RoPE on Q/K at positions offset + r, Q -> q_out,
    K/V -> cache rows [offset, offset + len).  x [len, hidden], w_qkv
    [(Hq + 2 Hkv) d, hidden], q_out [len, Hq, d], caches [cap, Hkv, d] (bf16)."""
    length, hidden = x.shape
    _, n_q, d = q_out.shape
    n_kv = k_cache.shape[1]
    _check(_lib.load().mocap_qkv_rope_append(_ptr(x), _ptr(w_qkv), _ptr(q_out), _ptr(k_cache),
                                             _ptr(v_cache), k_cache.shape[0], offset, length,
                                             hidden, n_q, n_kv, d, rope_theta, _stream(stream)),
           "mocap_qkv_rope_append")


def mocap_chunk_attn_workspace_size(prefix: int, length: int, n_q_heads: int, n_kv_heads: int,
                                    head_dim: int) -> int:
    """Bytes of scratch that let mocap_chunk_attn split the key range (0 = no split)."""
    return int(_lib.load().mocap_chunk_attn_workspace_size(prefix, length, n_q_heads, n_kv_heads,
                                                           head_dim))


def mocap_chunk_attn(q, k_cache, v_cache, prefix: int, out, lse, scale: float,
                     workspace=None, stream=None):
    """One chunk's causal GQA attention over cache rows [0, prefix+len).

    q/out [len, Hq, d] bf16, caches [>= prefix+len, Hkv, d] bf16, lse [Hq, len] fp32.
    """
    length, n_q, d = q.shape
    n_kv = k_cache.shape[1]
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    if workspace is not None and not workspace.is_contiguous():
        raise ValueError("workspace must be contiguous")
    _check(_lib.load().mocap_chunk_attn(_ptr(q), _ptr(k_cache), _ptr(v_cache), prefix, length,
                                        n_q, n_kv, d, scale, _ptr(out), _ptr(lse),
                                        _ptr(workspace), ws_bytes, _stream(stream)),
           "mocap_chunk_attn")


def mocap_chunk_attn_noalloc(q, k_cache, v_cache, prefix: int, out, lse, scale: float,
                             stream=None):
    """mocap_chunk_attn without a caller workspace: split-KV partials go to
    the library's fixed device scratch (MOCAP_NOALLOC_SCRATCH_BYTES); calls
    whose work overlaps on the GPU must not share it."""
    length, n_q, d = q.shape
    n_kv = k_cache.shape[1]
    _check(_lib.load().mocap_chunk_attn_noalloc(_ptr(q), _ptr(k_cache), _ptr(v_cache), prefix,
                                                length, n_q, n_kv, d, scale, _ptr(out), _ptr(lse),
                                                _stream(stream)),
           "mocap_chunk_attn_noalloc")


def mocap_chunk_attn_varlen(q, k_cache, v_cache, items: Sequence[tuple], out, lse, scale: float,
                            workspace=None, stream=None):
    """Many (q_row, kv_row, prefix, len) items in one launch; lse is [Hq, q_rows_total].
    With one non-empty item, ``workspace`` (as for mocap_chunk_attn) lets it split."""
    q_rows, n_q, d = q.shape
    n_kv = k_cache.shape[1]
    arr = (VarlenItem * max(1, len(items)))()
    for i, (q_row, kv_row, prefix, length) in enumerate(items):
        arr[i] = VarlenItem(q_row, kv_row, prefix, length)
    if workspace is not None and not workspace.is_contiguous():
        raise ValueError("workspace must be contiguous")
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _check(_lib.load().mocap_chunk_attn_varlen(_ptr(q), _ptr(k_cache), _ptr(v_cache), arr,
                                               len(items), q_rows, k_cache.shape[0], n_q, n_kv,
                                               d, scale, _ptr(out), _ptr(lse), _ptr(workspace),
                                               ws_bytes, _stream(stream)),
           "mocap_chunk_attn_varlen")


def mocap_chunk_attn_varlen_dev_workspace_size(n_items: int, max_rows: int, n_q_heads: int,
                                               n_kv_heads: int, head_dim: int) -> int:
    """Bytes of scratch mocap_chunk_attn_varlen_dev needs for n_items items of
    at most max_rows rows in all (0: n_items == 0 or out of range)."""
    return int(_lib.load().mocap_chunk_attn_varlen_dev_workspace_size(
        n_items, max_rows, n_q_heads, n_kv_heads, head_dim))


def mocap_chunk_attn_varlen_dev(q, k_cache, v_cache, items, out, lse, scale: float,
                                max_rows=None, workspace=None, stream=None):
    """mocap_chunk_attn_varlen with the items in device memory: ``items`` is a
    contiguous int64 tensor [n, 4] of (q_row, kv_row, prefix, len) rows on the
    device; lse is [Hq, q_rows_total].  ``max_rows`` bounds the items' total
    length (default: all rows of q).  ``workspace``: a uint8 device tensor of
    at least mocap_chunk_attn_varlen_dev_workspace_size bytes (allocated here
    when None).  An invalid item is reported by mocap_last_device_status."""
    import torch
    q_rows, n_q, d = q.shape
    n_kv = k_cache.shape[1]
    if items.dtype != torch.int64 or items.dim() != 2 or items.shape[1] != 4 or \
            not items.is_contiguous():
        raise ValueError("items must be a contiguous int64 tensor [n, 4]")
    n = items.shape[0]
    max_rows = q_rows if max_rows is None else int(max_rows)
    need = mocap_chunk_attn_varlen_dev_workspace_size(n, max_rows, n_q, n_kv, d)
    if workspace is None:
        workspace = torch.empty((max(need, 128),), device=q.device, dtype=torch.uint8)
    if not workspace.is_contiguous():
        raise ValueError("workspace must be contiguous")
    ws_bytes = workspace.numel() * workspace.element_size()
    _check(_lib.load().mocap_chunk_attn_varlen_dev(_ptr(q), _ptr(k_cache), _ptr(v_cache),
                                                   _ptr(items), n, q_rows, k_cache.shape[0],
                                                   max_rows, n_q, n_kv, d, scale, _ptr(out),
                                                   _ptr(lse), _ptr(workspace), ws_bytes,
                                                   _stream(stream)),
           "mocap_chunk_attn_varlen_dev")


def _append_array(appends):
    """(k_src, v_src, dst_row) triples -> the C descriptor array; the sources
    are [rows, Hkv, d] tensors (contiguous, on the device)."""
    arr = (AppendItem * max(1, len(appends)))()
    for i, (k_src, v_src, dst_row) in enumerate(appends):
        if k_src.shape != v_src.shape:
            raise ValueError("K and V sources of an append must have the same shape")
        arr[i] = AppendItem(_ptr(k_src), _ptr(v_src), dst_row, k_src.shape[0])
    return arr


def mocap_chunk_attn_append(q, k_cache, v_cache, prefix: int, out, lse, scale: float,
                            appends: Sequence[tuple] = (), workspace=None, stream=None):
    """mocap_chunk_attn that also writes ``appends`` -- (k_src, v_src, dst_row)
    with sources [rows, Hkv, d] -- into cache rows [dst_row, dst_row + rows)
    in the same launch (rows outside [0, prefix + len))."""
    length, n_q, d = q.shape
    n_kv = k_cache.shape[1]
    if workspace is not None and not workspace.is_contiguous():
        raise ValueError("workspace must be contiguous")
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _check(_lib.load().mocap_chunk_attn_append(_ptr(q), _ptr(k_cache), _ptr(v_cache), prefix,
                                               length, n_q, n_kv, d, scale, _ptr(out), _ptr(lse),
                                               _ptr(workspace), ws_bytes, _append_array(appends),
                                               len(appends), k_cache.shape[0], _stream(stream)),
           "mocap_chunk_attn_append")


def mocap_chunk_attn_varlen_append(q, k_cache, v_cache, items: Sequence[tuple], out, lse,
                                   scale: float, appends: Sequence[tuple] = (), workspace=None,
                                   stream=None):
    """mocap_chunk_attn_varlen that also writes ``appends`` (as in
    mocap_chunk_attn_append, rows of the packed caches) in the same launch."""
    q_rows, n_q, d = q.shape
    n_kv = k_cache.shape[1]
    arr = (VarlenItem * max(1, len(items)))()
    for i, (q_row, kv_row, prefix, length) in enumerate(items):
        arr[i] = VarlenItem(q_row, kv_row, prefix, length)
    if workspace is not None and not workspace.is_contiguous():
        raise ValueError("workspace must be contiguous")
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _check(_lib.load().mocap_chunk_attn_varlen_append(
        _ptr(q), _ptr(k_cache), _ptr(v_cache), arr, len(items), q_rows, k_cache.shape[0], n_q,
        n_kv, d, scale, _ptr(out), _ptr(lse), _ptr(workspace), ws_bytes, _append_array(appends),
        len(appends), _stream(stream)), "mocap_chunk_attn_varlen_append")


def mocap_last_row_attn_workspace_size(kv_len, n_q_heads: int, n_kv_heads: int,
                                       head_dim: int) -> int:
    arr = (ctypes.c_int64 * len(kv_len))(*kv_len)
    return int(_lib.load().mocap_last_row_attn_workspace_size(arr, len(kv_len), n_q_heads,
                                                              n_kv_heads, head_dim))


def mocap_last_row_attn(q_last, k_cache, v_cache, kv_row, kv_len, out, lse, scale: float,
                        workspace=None, stream=None):
    """Each request's last row against all its keys.  q_last/out [n_req, Hq, d],
    caches [rows, Hkv, d], lse [Hq, n_req]; kv_row/kv_len: host sequences."""
    import torch
    n_req, n_q, d = q_last.shape
    n_kv = k_cache.shape[1]
    rows = (ctypes.c_int64 * n_req)(*kv_row)
    lens = (ctypes.c_int64 * n_req)(*kv_len)
    need = mocap_last_row_attn_workspace_size(kv_len, n_q, n_kv, d)
    if workspace is None:
        workspace = torch.empty((max(need, 16),), device=q_last.device, dtype=torch.uint8)
    ws_bytes = workspace.numel() * workspace.element_size()
    _check(_lib.load().mocap_last_row_attn(_ptr(q_last), _ptr(k_cache), _ptr(v_cache), rows, lens,
                                           n_req, k_cache.shape[0], n_q, n_kv, d, scale,
                                           _ptr(out), _ptr(lse), _ptr(workspace), ws_bytes,
                                           _stream(stream)),
           "mocap_last_row_attn")


def mocap_last_device_status(stream=None) -> int:
    return int(_lib.load().mocap_last_device_status(_stream(stream)))


def mocap_selftest_bounded_wait(limit_us: int, stream=None):
    """Launch a kernel whose bounded wait expires after limit_us (failure-path test)."""
    _check(_lib.load().mocap_selftest_bounded_wait(limit_us, _stream(stream)),
           "mocap_selftest_bounded_wait")


def mocap_status_string(status: int) -> str:
    return _lib.load().mocap_status_string(status).decode()
