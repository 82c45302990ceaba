"""GPU: attention launches that also append the next chunk's K/V
(mocap_chunk_attn_append, mocap_chunk_attn_varlen_append), through the C ABI.

The chunked prefill walks its chunks in order (Sec. 2.2); chunk i + 1's K/V
rows are written by chunk i's attention launch.  The attention results must
be bitwise those of the plain entry points (the attention work is the same
kernel code), the appended cache rows bitwise the sources, and every other
cache row untouched (sentinel bit patterns, NaN encodings included).
"""

import math

import numpy as np
import pytest
import torch

from oracle import attention as A
from tests.parity_utils import assert_close, check_single_request, f64, sample_rows

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def m():
    import paper_2606_22968_gb300 as mod
    mod._lib.load()
    return mod


def _randn(shape, gen, dev):
    return torch.randn(shape, generator=gen, device=dev, dtype=torch.bfloat16)


def _sentinel(shape, gen, dev):
    """Random bf16 bit patterns (NaN and Inf encodings included)."""
    bits = torch.randint(-32768, 32767, shape, generator=gen, device=dev, dtype=torch.int16)
    return bits.view(torch.bfloat16)


CASES = [
    # (prefix, len, Hq, Hkv, d, append row counts, pair form, forced splits)
    (0, 300, 8, 2, 128, [257], "1", None),
    (1000, 129, 16, 2, 128, [1, 640], "1", None),
    (100000, 256, 8, 2, 128, [2048], "1", None),      # the library splits the key range
    (200, 700, 8, 2, 128, [300, 5, 77], "0", 2),       # single-CTA form, two splits
    (50, 130, 4, 4, 64, [129], "0", None),             # d = 64
    (500, 700, 96, 8, 128, [1000], "1", 3),            # 12:1 heads, three splits
    (3000, 1, 6, 2, 128, [64] * 40, "1", None),        # one row, 40 appends
    (128, 0, 8, 2, 128, [200, 9], "1", None),          # no attention rows: appends only
]


@pytest.mark.parametrize("prefix,length,hq,hkv,d,app_rows,pair,forced", CASES)
def test_fused_append_bitwise(m, monkeypatch, prefix, length, hq, hkv, d, app_rows, pair, forced):
    monkeypatch.setenv("MOCAP_ATTN_PAIR", pair)
    if forced is not None:
        monkeypatch.setenv("MOCAP_SPLIT_KV", str(forced))
    dev = torch.device("cuda")
    gen = torch.Generator(device=dev).manual_seed(prefix + length + sum(app_rows))
    s = prefix + length
    cap = s + sum(app_rows) + 17
    # (slices of one-row tensors when empty, so that every pointer is non-null)
    q = _randn((max(length, 1), hq, d), gen, dev)[:length]
    k_cache = _sentinel((cap, hkv, d), gen, dev)
    v_cache = _sentinel((cap, hkv, d), gen, dev)
    k_cache[:s] = _randn((s, hkv, d), gen, dev)
    v_cache[:s] = _randn((s, hkv, d), gen, dev)
    k_before, v_before = k_cache.clone(), v_cache.clone()
    srcs, appends, row = [], [], s + 3
    for n in app_rows:
        ks, vs = _randn((n, hkv, d), gen, dev), _randn((n, hkv, d), gen, dev)
        srcs.append((ks, vs, row))
        appends.append((ks, vs, row))
        row += n
    scale = 1.0 / math.sqrt(d)
    ws_bytes = m.mocap_chunk_attn_workspace_size(prefix, length, hq, hkv, d)
    ws = torch.full((max(ws_bytes, 16),), 0xFF, device=dev, dtype=torch.uint8)
    out_f = torch.full((max(length, 1), hq, d), float("nan"), device=dev,
                       dtype=torch.bfloat16)[:length]
    lse_f = torch.full((hq, max(length, 1)), float("nan"), device=dev,
                       dtype=torch.float32)[:, :length]
    if length > 0:
        m.mocap_chunk_attn_append(q, k_cache, v_cache, prefix, out_f, lse_f, scale, appends,
                                  workspace=ws)
    else:
        # torch reports a null data pointer for empty tensors, so the C ABI is
        # called directly with the (unused) one-row buffers behind them
        from paper_2606_22968_gb300._lib import AppendItem
        arr = (AppendItem * len(appends))(*[AppendItem(ks.data_ptr(), vs.data_ptr(), r0,
                                                       ks.shape[0]) for ks, vs, r0 in appends])
        base_q = q.untyped_storage().data_ptr()
        base_o = out_f.untyped_storage().data_ptr()
        base_l = lse_f.untyped_storage().data_ptr()
        assert m._lib.load().mocap_chunk_attn_append(
            base_q, k_cache.data_ptr(), v_cache.data_ptr(), prefix, 0, hq, hkv, d, scale, base_o,
            base_l, None, 0, arr, len(appends), cap, torch.cuda.current_stream().cuda_stream) == 0
    torch.cuda.synchronize()
    assert m.mocap_last_device_status() == 0
    # appended rows bitwise, every other row untouched
    k_exp, v_exp = k_before.clone(), v_before.clone()
    for ks, vs, r0 in srcs:
        k_exp[r0:r0 + ks.shape[0]] = ks
        v_exp[r0:r0 + vs.shape[0]] = vs
    assert torch.equal(k_cache.view(torch.int16), k_exp.view(torch.int16))
    assert torch.equal(v_cache.view(torch.int16), v_exp.view(torch.int16))
    if length == 0:
        return
    # the attention results are the plain entry point's, bitwise
    out_p = torch.empty_like(out_f)
    lse_p = torch.empty_like(lse_f)
    m.mocap_chunk_attn(q, k_before, v_before, prefix, out_p, lse_p, scale, workspace=ws)
    torch.cuda.synchronize()
    assert torch.equal(out_f, out_p) and torch.equal(lse_f, lse_p)
    rows = np.arange(length) if length <= 300 else sample_rows(length, every=53)
    idx = torch.as_tensor(rows, device=dev)
    q_rows = np.zeros((int(rows.max()) + 1, hq, d))
    q_rows[rows] = f64(q[idx])
    o_ref, l_ref = A.chunk_attention(q_rows, f64(k_before[:s]), f64(v_before[:s]), prefix, scale,
                                     rows=rows)
    assert_close(out_f[idx].float().cpu().numpy(), lse_f[:, idx].cpu().numpy(), o_ref, l_ref,
                 "fused append")


def test_varlen_fused_append_bitwise(m):
    """Several requests' chunk k attend while chunk k + 1 of each is appended."""
    dev = torch.device("cuda")
    gen = torch.Generator(device=dev).manual_seed(77)
    hq, hkv, d = 8, 2, 128
    lens = [300, 1000, 129, 640]
    cut = [int(0.4 * n) for n in lens]
    cu = np.concatenate([[0], np.cumsum(lens)]).tolist()
    t = cu[-1]
    q, k, v = _randn((t, hq, d), gen, dev), _randn((t, hkv, d), gen, dev), _randn((t, hkv, d), gen, dev)
    kc, vc = _sentinel((t, hkv, d), gen, dev), _sentinel((t, hkv, d), gen, dev)
    for r in range(4):  # chunk 0 of every request is in the cache already
        kc[cu[r]:cu[r] + cut[r]] = k[cu[r]:cu[r] + cut[r]]
        vc[cu[r]:cu[r] + cut[r]] = v[cu[r]:cu[r] + cut[r]]
    kc_before, vc_before = kc.clone(), vc.clone()
    items = [(cu[r], cu[r], 0, cut[r]) for r in range(4)]
    appends = [(k[cu[r] + cut[r]:cu[r + 1]], v[cu[r] + cut[r]:cu[r + 1]], cu[r] + cut[r])
               for r in range(4)]
    out_f = torch.full((t, hq, d), float("nan"), device=dev, dtype=torch.bfloat16)
    lse_f = torch.full((hq, t), float("nan"), device=dev, dtype=torch.float32)
    m.mocap_chunk_attn_varlen_append(q, kc, vc, items, out_f, lse_f, 0.088, appends)
    torch.cuda.synchronize()
    assert m.mocap_last_device_status() == 0
    assert torch.equal(kc, k) and torch.equal(vc, v)  # every request's chunk 1 appended
    out_p = torch.full_like(out_f, float("nan"))
    lse_p = torch.full_like(lse_f, float("nan"))
    m.mocap_chunk_attn_varlen(q, kc_before, vc_before, items, out_p, lse_p, 0.088)
    torch.cuda.synchronize()
    assert torch.equal(out_f.view(torch.int16), out_p.view(torch.int16))
    assert torch.equal(lse_f.view(torch.int32), lse_p.view(torch.int32))
    # rows outside the items keep their NaN fill; the items' rows match the oracle
    for r in range(4):
        a = cu[r]
        assert torch.isnan(out_f[a + cut[r]:cu[r + 1]].float()).all()
        o_ref, l_ref = A.causal_attention(f64(q[a:a + cut[r]]), f64(k[a:a + cut[r]]),
                                          f64(v[a:a + cut[r]]), 0.088)
        assert_close(out_f[a:a + cut[r]].float().cpu().numpy(),
                     lse_f[:, a:a + cut[r]].cpu().numpy(), o_ref, l_ref, f"request {r}")


@pytest.mark.parametrize("mode", ["fused", "overlap"])
@pytest.mark.parametrize("index", [1, 2, 3, 5])
def test_append_modes_equal_serial_pipeline(m, index, mode):
    """The prompt with each next chunk's append in the attention launch
    ("fused") or on a second stream beside it ("overlap") gives bitwise the
    results of one append launch per chunk on one stream ("serial"), eager
    and replayed from a CUDA graph, caches poisoned with NaN first."""
    from paper_2606_22968_gb300 import workloads
    from paper_2606_22968_gb300.pipeline import ChunkedPrefill
    w = workloads.get(index)
    dev = torch.device("cuda")
    q, k, v = workloads.make_qkv(w, dev)
    pu = ChunkedPrefill(w, dev, append_mode="serial")
    pu.run(q, k, v)
    pf = ChunkedPrefill(w, dev, append_mode=mode, chunk_streams=1)
    for t in (pf.out, pf.lse, pf.k_cache, pf.v_cache):
        t.fill_(float("nan"))
    pf.run(q, k, v)
    torch.cuda.synchronize()
    assert m.mocap_last_device_status() == 0
    assert torch.equal(pf.k_cache, k) and torch.equal(pf.v_cache, v)
    assert torch.equal(pf.out, pu.out) and torch.equal(pf.lse, pu.lse)
    graph = pf.capture(q, k, v)
    for _ in range(2):
        for t in (pf.out, pf.lse, pf.k_cache, pf.v_cache):
            t.fill_(float("nan"))
        graph.replay()
        torch.cuda.synchronize()
        assert torch.equal(pf.k_cache, k) and torch.equal(pf.v_cache, v)
        assert torch.equal(pf.out, pu.out) and torch.equal(pf.lse, pu.lse)
    del graph


def test_overlap_pipeline_and_step_graphs_against_oracle(m):
    """The 131072-token workload with its appends on a second stream (caches
    and outputs poisoned first): caches bitwise, every chunk against the
    oracle on its first, tile-edge, middle and last rows (four rotating
    heads); then its per-step attention graphs replayed in order give the
    same bits."""
    from paper_2606_22968_gb300 import workloads
    from paper_2606_22968_gb300.pipeline import ChunkedPrefill
    from tests.parity_utils import rotating_heads
    w = workloads.get(4)
    dev = torch.device("cuda")
    q, k, v = workloads.make_qkv(w, dev)
    pf = ChunkedPrefill(w, dev, append_mode="overlap")
    for t in (pf.out, pf.lse, pf.k_cache, pf.v_cache):
        t.fill_(float("nan"))
    pf.run(q, k, v)
    torch.cuda.synchronize()
    assert m.mocap_last_device_status() == 0
    assert torch.equal(pf.k_cache, k) and torch.equal(pf.v_cache, v)
    check_single_request(pf, q, k, v, rows_fn=lambda n, i: np.array([0, 127, 128, n // 2, n - 1]),
                         heads_fn=rotating_heads(64))
    out_ref, lse_ref = pf.out.clone(), pf.lse.clone()
    graphs = pf.capture_steps(q, k, v)
    pf.out.fill_(float("nan"))
    pf.lse.fill_(float("nan"))
    for g in graphs:
        g.replay()
    torch.cuda.synchronize()
    assert torch.equal(pf.out, out_ref) and torch.equal(pf.lse, lse_ref)
    del graphs


@pytest.mark.parametrize("index", [3, 5])
def test_overlap_mode_from_host_matches_device_run(m, index):
    """Host-streamed prompts with overlapped appends (the second stream waits
    for each step's upload) give bitwise the device-resident results."""
    from paper_2606_22968_gb300 import workloads
    from paper_2606_22968_gb300.pipeline import ChunkedPrefill
    w = workloads.get(index)
    dev = torch.device("cuda")
    q, k, v = workloads.make_qkv(w, dev)
    pf = ChunkedPrefill(w, dev, append_mode="overlap")
    pf.run(q, k, v)
    torch.cuda.synchronize()
    out_ref, lse_ref = pf.out.clone(), pf.lse.clone()
    hq, hk, hv = (t.cpu().pin_memory() for t in (q, k, v))
    outs = []
    for _ in range(3):
        ho = torch.full(pf.out.shape, float("nan"), dtype=pf.out.dtype).pin_memory()
        hl = torch.full(pf.lse.shape, float("nan"), dtype=pf.lse.dtype).pin_memory()
        outs.append((hq, hk, hv, ho, hl))
    bufs = [tuple(torch.full_like(t, float("nan")) for t in (q, k, v)) for _ in range(2)]
    pf.k_cache.fill_(float("nan"))
    pf.v_cache.fill_(float("nan"))
    pf.run_prompts_from_host(outs, bufs)
    torch.cuda.synchronize()
    assert m.mocap_last_device_status() == 0
    for _, _, _, ho, hl in outs:
        assert torch.equal(ho, out_ref.cpu()) and torch.equal(hl, lse_ref.cpu())


def test_fused_launch_after_expired_wait_does_nothing(m):
    dev = torch.device("cuda")
    gen = torch.Generator(device=dev).manual_seed(5)
    q = _randn((300, 8, 128), gen, dev)
    kc = _randn((700, 2, 128), gen, dev)
    vc = _randn((700, 2, 128), gen, dev)
    ks, vs = _randn((200, 2, 128), gen, dev), _randn((200, 2, 128), gen, dev)
    kc_before, vc_before = kc.clone(), vc.clone()
    out = torch.full_like(q, float("nan"))
    lse = torch.full((8, 300), float("nan"), device=dev, dtype=torch.float32)
    m.mocap_selftest_bounded_wait(20000)
    m.mocap_chunk_attn_append(q, kc, vc, 0, out, lse, 0.088, [(ks, vs, 400)])
    torch.cuda.synchronize()
    assert m.mocap_last_device_status() == m.MOCAP_ETIMEOUT
    assert torch.isnan(out.float()).all() and torch.isnan(lse).all()
    assert torch.equal(kc, kc_before) and torch.equal(vc, vc_before)  # no append either
    m.mocap_chunk_attn_append(q, kc, vc, 0, out, lse, 0.088, [(ks, vs, 400)])
    torch.cuda.synchronize()
    assert m.mocap_last_device_status() == m.MOCAP_OK
    assert torch.equal(kc[400:600], ks) and torch.equal(vc[400:600], vs)
    assert not torch.isnan(out.float()).any()


@pytest.mark.parametrize("index", [1, 2, 3, 5])
def test_two_chunk_streams_equal_one(m, index):
    """Attention launches alternating between two compute streams (each with
    its own split-KV scratch; appends on a third) give bitwise the results
    of one stream, eager and replayed from a CUDA graph."""
    from paper_2606_22968_gb300 import workloads
    from paper_2606_22968_gb300.pipeline import ChunkedPrefill
    w = workloads.get(index)
    dev = torch.device("cuda")
    q, k, v = workloads.make_qkv(w, dev)
    p1 = ChunkedPrefill(w, dev, chunk_streams=1)
    p1.run(q, k, v)
    p2 = ChunkedPrefill(w, dev, chunk_streams=2)
    assert ChunkedPrefill(w, dev).chunk_streams == 2  # the default with overlapped appends
    for _ in range(2):
        for t in (p2.out, p2.lse, p2.k_cache, p2.v_cache):
            t.fill_(float("nan"))
        p2.run(q, k, v)
        torch.cuda.synchronize()
        assert m.mocap_last_device_status() == 0
        assert torch.equal(p2.k_cache, k) and torch.equal(p2.v_cache, v)
        assert torch.equal(p2.out, p1.out) and torch.equal(p2.lse, p1.lse)
    graph = p2.capture(q, k, v)
    for t in (p2.out, p2.lse, p2.k_cache, p2.v_cache):
        t.fill_(float("nan"))
    graph.replay()
    torch.cuda.synchronize()
    assert torch.equal(p2.k_cache, k) and torch.equal(p2.v_cache, v)
    assert torch.equal(p2.out, p1.out) and torch.equal(p2.lse, p1.lse)
    del graph


def test_two_chunk_streams_need_overlapped_appends():
    from paper_2606_22968_gb300 import workloads
    from paper_2606_22968_gb300.pipeline import ChunkedPrefill
    for mode in ("serial", "fused"):
        with pytest.raises(ValueError):
            ChunkedPrefill(workloads.get(1), torch.device("cuda"), append_mode=mode,
                           chunk_streams=2)
