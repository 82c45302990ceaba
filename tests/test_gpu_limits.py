"""GPU: the size limits and degenerate cases of the attention entry points,
against the float64 oracle.

- A chunk whose Q/O element count passes 2^31 (270000 rows x 64 heads x 128
  dims): rows on both sides of element 2^31 and the ragged last tile.
- Prefixes of about 2^21 keys (sixteen times the longest workload), with
  and without the split-KV scratch, on both kernel forms (CTA pairs at
  d = 128, single CTAs at d = 64), and last-row attention over them.
- An empty chunk (nothing written) and a one-row chunk at position 0, whose
  output is V[0] exactly (one visible key: p = 1, l = 1).

The oracle evaluates each sampled row on its own: chunk-local row r of a
chunk at ``prefix`` is row 0 of a one-row chunk at ``prefix + r`` (same
visible keys), and the query heads of one KV group are a problem with a
single KV head, so only that group's keys are widened to float64."""

import math

import numpy as np
import pytest
import torch

from oracle import attention as A
from tests.parity_utils import assert_close, f64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def m():
    import paper_2606_22968_gb300 as mod
    mod._lib.load()
    return mod


def _oracle_rows(q, k_cache, v_cache, prefix, rows, heads, scale):
    """O [n, H, d] and LSE [H, n] of chunk-local ``rows`` for ``heads``,
    one KV group and one row at a time."""
    n_q, n_kv = q.shape[1], k_cache.shape[1]
    group = n_q // n_kv
    o = np.zeros((len(rows), len(heads), q.shape[2]))
    lse = np.zeros((len(heads), len(rows)))
    for g in sorted({h // group for h in heads}):
        cols = [j for j, h in enumerate(heads) if h // group == g]
        hs = [heads[j] for j in cols]
        end = prefix + int(max(rows)) + 1
        kf = f64(k_cache[:end, g:g + 1])
        vf = f64(v_cache[:end, g:g + 1])
        for i, r in enumerate(rows):
            qr = f64(q[int(r):int(r) + 1, hs])
            o_r, l_r = A.chunk_attention(qr, kf, vf, prefix + int(r), scale)
            o[i, cols] = o_r[0]
            lse[cols, i] = l_r[:, 0]
    return o, lse


def _check(out, lse, q, k, v, prefix, rows, heads, scale, what):
    o_ref, l_ref = _oracle_rows(q, k, v, prefix, rows, heads, scale)
    idx = torch.as_tensor(rows, device=out.device)
    o_gpu = out[idx][:, heads].float().cpu().numpy()
    l_gpu = lse[:, idx][heads].cpu().numpy()
    assert_close(o_gpu, l_gpu, o_ref, l_ref, what)


def test_chunk_past_2_31_output_elements(m):
    """270000 rows x 64 heads x 128 dims = 2.2e9 elements of Q and O: rows
    262143 / 262144 straddle element 2^31, the last tile holds 80 rows.  The
    varlen entry point with the same chunk as its one item gives the same
    bits."""
    hq, hkv, d, length = 64, 8, 128, 270000
    assert length * hq * d > 2 ** 31
    dev = torch.device("cuda")
    gen = torch.Generator(device=dev).manual_seed(270000)
    q = torch.randn((length, hq, d), generator=gen, device=dev, dtype=torch.bfloat16)
    k = torch.randn((length, hkv, d), generator=gen, device=dev, dtype=torch.bfloat16)
    v = torch.randn((length, hkv, d), generator=gen, device=dev, dtype=torch.bfloat16)
    scale = 1.0 / math.sqrt(d)
    out = torch.full((length, hq, d), float("nan"), device=dev, dtype=torch.bfloat16)
    lse = torch.full((hq, length), float("nan"), device=dev, dtype=torch.float32)
    need = m.mocap_chunk_attn_workspace_size(0, length, hq, hkv, d)
    ws = torch.empty((max(need, 16),), device=dev, dtype=torch.uint8)
    m.mocap_chunk_attn(q, k, v, 0, out, lse, scale, workspace=ws)
    torch.cuda.synchronize()
    assert m.mocap_last_device_status() == 0
    edge = 2 ** 31 // (hq * d)
    rows = np.array([0, 1, 127, 128, edge - 129, edge - 1, edge, edge + 1, length - 81,
                     length - 80, length - 1])
    _check(out, lse, q, k, v, 0, rows, [0, 13, 63], scale, "270000-row chunk")
    assert not torch.isnan(out[edge - 2:edge + 2]).any()
    assert not torch.isnan(lse[:, -128:]).any()
    out2 = torch.full_like(out, float("nan"))
    lse2 = torch.full_like(lse, float("nan"))
    m.mocap_chunk_attn_varlen(q, k, v, [(0, 0, 0, length)], out2, lse2, scale, workspace=ws)
    torch.cuda.synchronize()
    assert m.mocap_last_device_status() == 0
    assert torch.equal(out2.view(torch.int16), out.view(torch.int16))
    assert torch.equal(lse2, lse)


@pytest.mark.parametrize("hq,hkv,d", [(4, 1, 128), (2, 1, 64)])
def test_two_million_key_prefix(m, hq, hkv, d):
    """A 301-row chunk after 2^21 - 77 cached keys (ragged on both ends):
    single pass and split key range against the oracle; rows past the
    chunk hold NaN and are never read.  Last-row attention over the same
    keys matches the chunk's last row."""
    prefix, length = 2 ** 21 - 77, 301
    total = prefix + length
    dev = torch.device("cuda")
    gen = torch.Generator(device=dev).manual_seed(total + d)
    k = torch.randn((total + 5, hkv, d), generator=gen, device=dev, dtype=torch.bfloat16)
    v = torch.randn((total + 5, hkv, d), generator=gen, device=dev, dtype=torch.bfloat16)
    k[total:] = float("nan")
    v[total:] = float("nan")
    q = torch.randn((length, hq, d), generator=gen, device=dev, dtype=torch.bfloat16)
    scale = 1.0 / math.sqrt(d)
    need = m.mocap_chunk_attn_workspace_size(prefix, length, hq, hkv, d)
    assert need > 0  # few CTAs and a long key range: the planner splits it
    ws = torch.empty((need,), device=dev, dtype=torch.uint8)
    results = []
    for workspace in (None, ws):
        out = torch.full((length, hq, d), float("nan"), device=dev, dtype=torch.bfloat16)
        lse = torch.full((hq, length), float("nan"), device=dev, dtype=torch.float32)
        m.mocap_chunk_attn(q, k, v, prefix, out, lse, scale, workspace=workspace)
        torch.cuda.synchronize()
        assert m.mocap_last_device_status() == 0
        results.append((out, lse))
    rows = np.array([0, 1, 127, 128, 255, 256, length - 1])
    heads = list(range(hq))
    for (out, lse), what in zip(results, ("single pass", "split")):
        _check(out, lse, q, k, v, prefix, rows, heads, scale, f"2M-key prefix, {what}")
    o_lr = torch.full((1, hq, d), float("nan"), device=dev, dtype=torch.bfloat16)
    l_lr = torch.full((hq, 1), float("nan"), device=dev, dtype=torch.float32)
    m.mocap_last_row_attn(q[length - 1:], k, v, [0], [total], o_lr, l_lr, scale)
    torch.cuda.synchronize()
    assert m.mocap_last_device_status() == 0
    _check(o_lr, l_lr, q[length - 1:], k, v, total - 1, np.array([0]), heads, scale,
           "last row over 2M keys")


def test_empty_chunk_writes_nothing(m):
    """len = 0 is a no-op for the chunk, varlen and append entry points: the
    sentinel bytes of every output survive."""
    dev = torch.device("cuda")
    hq, hkv, d = 8, 2, 128
    q = torch.randn((4, hq, d), device=dev).bfloat16()
    k = torch.randn((64, hkv, d), device=dev).bfloat16()
    v = torch.randn((64, hkv, d), device=dev).bfloat16()
    out = torch.full((4, hq, d), 7.0, device=dev, dtype=torch.bfloat16)
    lse = torch.full((hq, 4), 7.0, device=dev, dtype=torch.float32)
    kc, vc = k.clone(), v.clone()
    lib = m._lib.load()
    stream = torch.cuda.current_stream().cuda_stream
    assert lib.mocap_chunk_attn(q.data_ptr(), k.data_ptr(), v.data_ptr(), 32, 0, hq, hkv, d,
                                0.1, out.data_ptr(), lse.data_ptr(), None, 0, stream) == 0
    m.mocap_chunk_attn_varlen(q, k, v, [(0, 0, 10, 0), (2, 0, 0, 0)], out, lse, 0.1)
    assert lib.mocap_kv_append(k.data_ptr(), v.data_ptr(), kc.data_ptr(), vc.data_ptr(), 64, 3,
                               0, hkv, d, stream) == 0
    torch.cuda.synchronize()
    assert m.mocap_last_device_status() == 0
    assert bool((out.float() == 7.0).all()) and bool((lse == 7.0).all())
    assert torch.equal(kc.view(torch.int16), k.view(torch.int16))
    assert torch.equal(vc.view(torch.int16), v.view(torch.int16))


@pytest.mark.parametrize("hq,hkv,d", [(8, 2, 128), (4, 4, 64), (16, 1, 128)])
def test_first_row_alone_is_v0(m, hq, hkv, d):
    """A one-row chunk at position 0 sees one key: p = 1 and l = 1, so O is
    V[0] of its group bit for bit and LSE is scale * q . k_0."""
    dev = torch.device("cuda")
    gen = torch.Generator(device=dev).manual_seed(hq * d)
    q = torch.randn((1, hq, d), generator=gen, device=dev, dtype=torch.bfloat16)
    k = torch.randn((1, hkv, d), generator=gen, device=dev, dtype=torch.bfloat16)
    v = torch.randn((1, hkv, d), generator=gen, device=dev, dtype=torch.bfloat16)
    scale = 1.0 / math.sqrt(d)
    out = torch.full((1, hq, d), float("nan"), device=dev, dtype=torch.bfloat16)
    lse = torch.full((hq, 1), float("nan"), device=dev, dtype=torch.float32)
    m.mocap_chunk_attn(q, k, v, 0, out, lse, scale)
    torch.cuda.synchronize()
    assert m.mocap_last_device_status() == 0
    group = hq // hkv
    expect = v[0, [h // group for h in range(hq)]]
    assert torch.equal(out[0].view(torch.int16), expect.view(torch.int16))
    qf, kf = f64(q)[0], f64(k)[0]
    ref = np.array([scale * qf[h] @ kf[h // group] for h in range(hq)])
    assert np.abs(lse[:, 0].cpu().numpy() - ref).max() <= 1e-3
