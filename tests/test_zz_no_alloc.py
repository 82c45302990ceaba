"""GPU: mocap_chunk_attn_noalloc, the entry point for callers that cannot
allocate device memory (a host program whose own pool owns the GPU's memory,
or a serving loop that cannot afford cudaMalloc / cudaFree).  It keeps its
split-KV partials in a fixed scratch array inside the library, so these tests
check that, called twice in a row through the C ABI, it gives bitwise the
results of mocap_chunk_attn with a caller-provided workspace, and that a
shape whose partials would not fit the array runs the single-pass kernel
(bitwise mocap_chunk_attn without a workspace, and within the parity
tolerances of the oracle).

Kept in a file of its own that pytest collects last; it passes alone in a
fresh process and after the other tests.
"""

import ctypes
import math

import numpy as np
import pytest
import torch

from oracle import attention as A
from tests.parity_utils import assert_close, f64

pytestmark = pytest.mark.gpu

SCRATCH_BYTES = 32 * 1024 * 1024


def _inputs(prefix, length, hq, hkv, d, seed):
    dev = torch.device("cuda")
    gen = torch.Generator(device=dev).manual_seed(seed)
    q = torch.randn((length, hq, d), generator=gen, device=dev, dtype=torch.bfloat16)
    k = torch.randn((prefix + length, hkv, d), generator=gen, device=dev, dtype=torch.bfloat16)
    v = torch.randn((prefix + length, hkv, d), generator=gen, device=dev, dtype=torch.bfloat16)
    return q, k, v


def _call_noalloc(lib, q, k, v, prefix, out, lse, scale):
    length, hq, d = q.shape
    hkv = k.shape[1]
    stream = torch.cuda.current_stream().cuda_stream
    return lib.mocap_chunk_attn_noalloc(q.data_ptr(), k.data_ptr(), v.data_ptr(), prefix, length,
                                        hq, hkv, d, scale, out.data_ptr(), lse.data_ptr(),
                                        stream)


def _call_with_workspace(lib, q, k, v, prefix, out, lse, scale):
    length, hq, d = q.shape
    hkv = k.shape[1]
    ws_bytes = lib.mocap_chunk_attn_workspace_size(prefix, length, hq, hkv, d)
    ws = torch.empty((max(ws_bytes, 16),), device=q.device, dtype=torch.uint8)
    stream = torch.cuda.current_stream().cuda_stream
    st = lib.mocap_chunk_attn(q.data_ptr(), k.data_ptr(), v.data_ptr(), prefix, length, hq, hkv,
                              d, scale, out.data_ptr(), lse.data_ptr(), ws.data_ptr(), ws_bytes,
                              stream)
    return st, ws_bytes


def test_noalloc_matches_workspace_entry_two_calls(lib, monkeypatch):
    # Two calls in a row on different shapes: the second runs over whatever
    # the first left in the shared scratch.
    cases = [
        (100000, 256, 8, 2, 128, None),  # few long row blocks: the library splits by itself
        (100, 300, 8, 2, 128, "2"),      # forced split whose second range some rows cannot see
    ]
    for i, (prefix, length, hq, hkv, d, forced) in enumerate(cases):
        if forced is None:
            monkeypatch.delenv("MOCAP_SPLIT_KV", raising=False)
        else:
            monkeypatch.setenv("MOCAP_SPLIT_KV", forced)
        q, k, v = _inputs(prefix, length, hq, hkv, d, seed=41 + i)
        scale = 1.0 / math.sqrt(d)
        ws_bytes = lib.mocap_chunk_attn_workspace_size(prefix, length, hq, hkv, d)
        assert 0 < ws_bytes <= SCRATCH_BYTES  # the split path runs, inside the fixed scratch
        out_n = torch.full((length, hq, d), float("nan"), device=q.device, dtype=torch.bfloat16)
        lse_n = torch.full((hq, length), float("nan"), device=q.device, dtype=torch.float32)
        assert _call_noalloc(lib, q, k, v, prefix, out_n, lse_n, scale) == 0
        out_w = torch.empty_like(out_n)
        lse_w = torch.empty_like(lse_n)
        st, _ = _call_with_workspace(lib, q, k, v, prefix, out_w, lse_w, scale)
        assert st == 0
        torch.cuda.synchronize()
        assert lib.mocap_last_device_status(torch.cuda.current_stream().cuda_stream) == 0
        # same split plan and kernels as the workspace entry point: bitwise equal
        assert torch.equal(out_n, out_w), f"call {i}: noalloc vs workspace (O)"
        assert torch.equal(lse_n, lse_w), f"call {i}: noalloc vs workspace (LSE)"
        # and against the float64 oracle
        o_ref, l_ref = A.chunk_attention(f64(q), f64(k), f64(v), prefix, scale)
        assert_close(out_n.float().cpu().numpy(), lse_n.cpu().numpy(), o_ref, l_ref,
                     f"call {i}: noalloc vs oracle")


def test_noalloc_runs_single_pass_when_the_split_exceeds_the_scratch(lib, monkeypatch):
    # A late chunk of the 131072-token Llama-3-70B shape (64 query heads, 8 KV
    # heads): the library splits its key range in two, whose partials
    # (2 x 2048 rows x 64 heads x (128 + 1) fp32 = 135 MB) exceed the 32 MiB
    # array, so the call runs the single-pass kernel: bitwise mocap_chunk_attn
    # without a workspace, and the oracle on sampled rows and heads.
    monkeypatch.setenv("MOCAP_SPLIT_KV", "2")
    prefix, length, hq, hkv, d = 129024 - 2048 + 77, 2048, 64, 8, 128
    assert lib.mocap_chunk_attn_workspace_size(prefix, length, hq, hkv, d) > SCRATCH_BYTES
    q, k, v = _inputs(prefix, length, hq, hkv, d, seed=7)
    scale = 1.0 / math.sqrt(d)
    stream = torch.cuda.current_stream().cuda_stream
    out_n = torch.full((length, hq, d), float("nan"), device=q.device, dtype=torch.bfloat16)
    lse_n = torch.full((hq, length), float("nan"), device=q.device, dtype=torch.float32)
    assert _call_noalloc(lib, q, k, v, prefix, out_n, lse_n, scale) == 0
    out_1 = torch.empty_like(out_n)
    lse_1 = torch.empty_like(lse_n)
    assert lib.mocap_chunk_attn(q.data_ptr(), k.data_ptr(), v.data_ptr(), prefix, length, hq,
                                hkv, d, scale, out_1.data_ptr(), lse_1.data_ptr(), None, 0,
                                stream) == 0
    torch.cuda.synchronize()
    assert lib.mocap_last_device_status(stream) == 0
    assert torch.equal(out_n, out_1) and torch.equal(lse_n, lse_1)
    rows = np.array([0, 1, 127, 128, 1023, 1024, 1919, 2047])
    heads = [0, 9, 18, 27, 36, 45, 54, 63]  # every KV group, every head slot of a pair
    idx = torch.as_tensor(rows, device=q.device)
    kf, vf = f64(k), f64(v)
    q_rows = np.zeros((length, hq, d))
    q_rows[rows] = f64(q[idx])
    o_ref, l_ref = A.chunk_attention(q_rows, kf, vf, prefix, scale, rows=rows, heads=heads)
    assert_close(out_n[idx][:, heads].float().cpu().numpy(), lse_n[heads][:, idx].cpu().numpy(),
                 o_ref, l_ref, "noalloc single pass vs oracle")


def test_python_binding_noalloc_equals_c_call(lib, monkeypatch):
    # the package's same-named function marshals the same call
    import paper_2606_22968_gb300 as m
    monkeypatch.setenv("MOCAP_SPLIT_KV", "2")
    prefix, length, hq, hkv, d = 1000, 300, 8, 2, 128
    q, k, v = _inputs(prefix, length, hq, hkv, d, seed=11)
    scale = 1.0 / math.sqrt(d)
    out_c = torch.empty_like(q)
    lse_c = torch.empty((hq, length), device=q.device, dtype=torch.float32)
    assert _call_noalloc(lib, q, k, v, prefix, out_c, lse_c, scale) == 0
    out_p = torch.full_like(q, float("nan"))
    lse_p = torch.full((hq, length), float("nan"), device=q.device, dtype=torch.float32)
    m.mocap_chunk_attn_noalloc(q, k, v, prefix, out_p, lse_p, scale)
    torch.cuda.synchronize()
    assert m.mocap_last_device_status() == m.MOCAP_OK
    assert torch.equal(out_p, out_c) and torch.equal(lse_p, lse_c)
