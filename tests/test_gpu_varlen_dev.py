"""GPU: mocap_chunk_attn_varlen_dev, the varlen attention whose (request,
chunk) items are read from device memory.  Per item its outputs are
bitwise those of the host-array form (several items never split), rows no
item covers keep their NaN fill, more than 64 items run in one launch and
match the oracle, an invalid device item is reported through the status
word with nothing written, and a CUDA graph replays the call with new item
values written into the same device tensor."""

import math

import numpy as np
import pytest
import torch

from tests.parity_utils import assert_close, chunk_rows_oracle, f64, sample_rows

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def m():
    import paper_2606_22968_gb300 as mod
    mod._lib.load()
    return mod


def _requests(rng, n_req, max_len):
    """Packed requests: lengths, each request's first row, and per request
    chunk boundaries (1..4 chunks, ragged)."""
    lens = [int(x) for x in rng.integers(1, max_len + 1, n_req)]
    starts = np.concatenate([[0], np.cumsum(lens)]).astype(int).tolist()
    bounds = []
    for L in lens:
        k = int(rng.integers(1, 5))
        cuts = sorted(set(int(x) for x in rng.integers(1, L, k - 1))) if L > 1 else []
        bounds.append([0] + cuts + [L])
    return lens, starts, bounds


def _all_chunk_items(starts, bounds):
    """(q_row, kv_row, prefix, len) of every chunk of every request; the
    caches hold every request's rows already, so all chunks may share one
    launch (their output rows do not overlap)."""
    items = []
    for s, b in zip(starts, bounds):
        for c in range(len(b) - 1):
            items.append((s + b[c], s, b[c], b[c + 1] - b[c]))
    return items


def _run_both(m, q, k, v, items, scale, host=True, tight=True):
    """The device-item call (grid bound: the items' total length when
    ``tight``, else every row of q) and the host-array form."""
    dev = q.device
    hq, d = q.shape[1], q.shape[2]
    rows = q.shape[0]
    out_d = torch.full((rows, hq, d), float("nan"), device=dev, dtype=torch.bfloat16)
    lse_d = torch.full((hq, rows), float("nan"), device=dev, dtype=torch.float32)
    it = torch.tensor(items, dtype=torch.int64, device=dev).reshape(-1, 4)
    bound = sum(x[3] for x in items) if tight else None
    m.mocap_chunk_attn_varlen_dev(q, k, v, it, out_d, lse_d, scale, max_rows=bound)
    torch.cuda.synchronize()
    assert m.mocap_last_device_status() == 0
    if not host:
        return out_d, lse_d, None, None
    out_h = torch.full_like(out_d, float("nan"))
    lse_h = torch.full_like(lse_d, float("nan"))
    for a in range(0, len(items), 64):  # the host-array form takes 64 items a launch
        part = items[a:a + 64]
        if sum(1 for x in part if x[3] > 0) == 1:
            part = part + [(0, 0, 0, 0)]  # keep two items: the host form then never splits
        m.mocap_chunk_attn_varlen(q, k, v, part, out_h, lse_h, scale)
    torch.cuda.synchronize()
    assert m.mocap_last_device_status() == 0
    return out_d, lse_d, out_h, lse_h


def _equal_bits(a, b):
    return torch.equal(a.contiguous().view(torch.int16 if a.dtype == torch.bfloat16 else torch.int32),
                       b.contiguous().view(torch.int16 if b.dtype == torch.bfloat16 else torch.int32))


@pytest.mark.parametrize("hq,hkv,d,seed", [
    (32, 8, 128, 1),   # CTA pairs
    (8, 2, 128, 2),    # CTA pairs, 4 heads per group
    (6, 2, 128, 3),    # single CTAs, odd head slot
    (4, 4, 64, 4),     # single CTAs, d = 64
    (16, 1, 128, 5),   # group of 16
])
def test_device_items_bitwise_equal_to_host_items(m, hq, hkv, d, seed):
    rng = np.random.default_rng(seed)
    lens, starts, bounds = _requests(rng, 5, 900)
    total = starts[-1]
    dev = torch.device("cuda")
    gen = torch.Generator(device=dev).manual_seed(seed)
    q = torch.randn((total + 7, hq, d), generator=gen, device=dev, dtype=torch.bfloat16)
    k = torch.randn((total + 7, hkv, d), generator=gen, device=dev, dtype=torch.bfloat16)
    v = torch.randn((total + 7, hkv, d), generator=gen, device=dev, dtype=torch.bfloat16)
    k[total:] = float("nan")
    v[total:] = float("nan")
    items = _all_chunk_items(starts, bounds)
    items.insert(2, (total, 0, 0, 0))  # an empty item in the middle
    scale = 1.0 / math.sqrt(d)
    for tight in (True, False):
        out_d, lse_d, out_h, lse_h = _run_both(m, q, k, v, items, scale, tight=tight)
        assert _equal_bits(out_d, out_h) and _equal_bits(lse_d, lse_h)
        assert torch.isnan(out_d[total:].float()).all() and torch.isnan(lse_d[:, total:]).all()
        assert not torch.isnan(out_d[:total].float()).any()


def test_three_hundred_items_in_one_launch(m):
    """300 (request, chunk) items (beyond the host form's 64): bitwise equal
    to the host form run 64 items at a time, and sampled rows of every tenth
    item against the oracle."""
    hq, hkv, d = 16, 4, 128
    rng = np.random.default_rng(300)
    lens, starts, bounds = _requests(rng, 120, 400)
    items = _all_chunk_items(starts, bounds)
    while len(items) < 300:  # more requests until there are at least 300 chunks
        more_lens, more_starts, more_bounds = _requests(rng, 10, 400)
        off = starts[-1]
        lens += more_lens
        starts = starts[:-1] + [off + s for s in more_starts]
        bounds += more_bounds
        items = _all_chunk_items(starts, bounds)
    total = starts[-1]
    dev = torch.device("cuda")
    gen = torch.Generator(device=dev).manual_seed(300)
    q = torch.randn((total, hq, d), generator=gen, device=dev, dtype=torch.bfloat16)
    k = torch.randn((total, hkv, d), generator=gen, device=dev, dtype=torch.bfloat16)
    v = torch.randn((total, hkv, d), generator=gen, device=dev, dtype=torch.bfloat16)
    scale = 1.0 / math.sqrt(d)
    out_d, lse_d, out_h, lse_h = _run_both(m, q, k, v, items, scale)
    assert _equal_bits(out_d, out_h) and _equal_bits(lse_d, lse_h)
    assert not torch.isnan(out_d.float()).any()
    kf, vf = f64(k), f64(v)
    for i in range(0, len(items), 10):
        q_row, kv_row, prefix, length = items[i]
        rows = sample_rows(length, every=61, edge=2, seed=i)
        idx = torch.as_tensor(rows + q_row, device=dev)
        o_ref, l_ref = chunk_rows_oracle(f64(q[idx]), kf[kv_row:kv_row + prefix + length],
                                         vf[kv_row:kv_row + prefix + length], prefix, rows, scale)
        assert_close(out_d[idx].float().cpu().numpy(), lse_d[:, idx].cpu().numpy(), o_ref, l_ref,
                     f"item {i}")


def test_varlen_workload_steps(m):
    """The 8-request varlen workload step by step (chunk k of every request
    per launch, as the pipeline runs it): device items bitwise equal to the
    host form at every step."""
    from paper_2606_22968_gb300 import workloads
    from paper_2606_22968_gb300.pipeline import ChunkedPrefill
    w = workloads.get(5)
    dev = torch.device("cuda")
    q, k, v = workloads.make_qkv(w, dev)
    pf = ChunkedPrefill(w, dev)
    steps = pf.steps()
    cu = pf.cu
    for st in steps:
        items = [(cu[r] + pf.bounds[r][c], cu[r], pf.bounds[r][c],
                  pf.bounds[r][c + 1] - pf.bounds[r][c]) for r, c in st]
        if len(items) == 1:
            items.append((0, 0, 0, 0))
        out_d, lse_d, out_h, lse_h = _run_both(m, q, k, v, items, w.scale)
        assert _equal_bits(out_d, out_h) and _equal_bits(lse_d, lse_h)


def test_invalid_device_item_is_reported_and_nothing_written(m):
    hq, hkv, d = 8, 2, 128
    dev = torch.device("cuda")
    q = torch.randn((600, hq, d), device=dev).bfloat16()
    k = torch.randn((600, hkv, d), device=dev).bfloat16()
    v = torch.randn((600, hkv, d), device=dev).bfloat16()
    out = torch.full((600, hq, d), float("nan"), device=dev, dtype=torch.bfloat16)
    lse = torch.full((hq, 600), float("nan"), device=dev, dtype=torch.float32)
    for bad in [(0, 0, 500, 200),     # keys past the cache
                (550, 0, 0, 100),     # queries past the buffer
                (0, -1, 0, 10),       # negative field
                (0, 0, 2 ** 31 - 5, 10)]:
        items = torch.tensor([(0, 0, 0, 300), bad], dtype=torch.int64, device=dev)
        m.mocap_chunk_attn_varlen_dev(q, k, v, items, out, lse, 0.1)
        torch.cuda.synchronize()
        assert m.mocap_last_device_status() == m.MOCAP_EINVAL, bad
        assert torch.isnan(out.float()).all() and torch.isnan(lse).all()
    # the status was read and cleared: a valid call runs
    items = torch.tensor([(0, 0, 0, 300), (300, 300, 0, 300)], dtype=torch.int64, device=dev)
    m.mocap_chunk_attn_varlen_dev(q, k, v, items, out, lse, 0.1)
    torch.cuda.synchronize()
    assert m.mocap_last_device_status() == 0
    assert not torch.isnan(out.float()).any()


def test_items_beyond_the_grid_bound_are_rejected(m):
    """Items that need more CTAs than the grid has: overlapping Q rows
    beyond the default bound, or items longer in all than the caller's
    max_rows: reported as invalid, nothing written."""
    hq, hkv, d = 8, 2, 128
    dev = torch.device("cuda")
    q = torch.randn((256, hq, d), device=dev).bfloat16()
    k = torch.randn((256, hkv, d), device=dev).bfloat16()
    v = torch.randn((256, hkv, d), device=dev).bfloat16()
    out = torch.full((256, hq, d), float("nan"), device=dev, dtype=torch.bfloat16)
    lse = torch.full((hq, 256), float("nan"), device=dev, dtype=torch.float32)
    items = torch.tensor([(0, 0, 0, 256)] * 8, dtype=torch.int64, device=dev)
    m.mocap_chunk_attn_varlen_dev(q, k, v, items, out, lse, 0.1)
    torch.cuda.synchronize()
    assert m.mocap_last_device_status() == m.MOCAP_EINVAL
    assert torch.isnan(out.float()).all()
    # a max_rows of 0 leaves one row block per item: 8 items of 32 rows fit
    items = torch.tensor([(32 * i, 0, 0, 32) for i in range(8)], dtype=torch.int64, device=dev)
    m.mocap_chunk_attn_varlen_dev(q, k, v, items, out, lse, 0.1, max_rows=0)
    torch.cuda.synchronize()
    assert m.mocap_last_device_status() == m.MOCAP_OK
    assert not torch.isnan(out.float()).any()
    # two items of 128 and 96 rows (2 row blocks) against max_rows = 0
    # (0 + 2 = 2 blocks): fit; 129 + 95 rows (3 blocks): do not
    for rows_a, ok in ((128, True), (129, False)):
        out.fill_(float("nan"))
        items = torch.tensor([(0, 0, 0, rows_a), (rows_a, 0, 0, 224 - rows_a)],
                             dtype=torch.int64, device=dev)
        m.mocap_chunk_attn_varlen_dev(q, k, v, items, out, lse, 0.1, max_rows=0)
        torch.cuda.synchronize()
        if ok:
            assert m.mocap_last_device_status() == m.MOCAP_OK
            assert not torch.isnan(out[:224].float()).any()
        else:
            assert m.mocap_last_device_status() == m.MOCAP_EINVAL
            assert torch.isnan(out.float()).all()


def test_graph_replay_with_new_device_items(m):
    """The call captured once in a CUDA graph; new item values written into
    the same device tensor between replays change what the replay computes
    (no host round trip), each replay bitwise equal to the host form."""
    hq, hkv, d = 32, 8, 128
    rng = np.random.default_rng(77)
    lens, starts, bounds = _requests(rng, 4, 2000)
    total = starts[-1]
    dev = torch.device("cuda")
    gen = torch.Generator(device=dev).manual_seed(77)
    q = torch.randn((total, hq, d), generator=gen, device=dev, dtype=torch.bfloat16)
    k = torch.randn((total, hkv, d), generator=gen, device=dev, dtype=torch.bfloat16)
    v = torch.randn((total, hkv, d), generator=gen, device=dev, dtype=torch.bfloat16)
    scale = 1.0 / math.sqrt(d)
    # two item sets with the same count: the first chunk, then the last
    first = [(s, s, 0, b[1]) for s, b in zip(starts, bounds)]
    last = [(s + b[-2], s, b[-2], b[-1] - b[-2]) for s, b in zip(starts, bounds)]
    items = torch.tensor(first, dtype=torch.int64, device=dev)
    out = torch.full((total, hq, d), float("nan"), device=dev, dtype=torch.bfloat16)
    lse = torch.full((hq, total), float("nan"), device=dev, dtype=torch.float32)
    need = m.mocap_chunk_attn_varlen_dev_workspace_size(len(first), total, hq, hkv, d)  # max_rows = all rows
    ws = torch.empty((need,), device=dev, dtype=torch.uint8)
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        m.mocap_chunk_attn_varlen_dev(q, k, v, items, out, lse, scale, workspace=ws, stream=side)
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        m.mocap_chunk_attn_varlen_dev(q, k, v, items, out, lse, scale, workspace=ws)
    for chosen in (last, first, last):
        items.copy_(torch.tensor(chosen, dtype=torch.int64))
        out.fill_(float("nan"))
        lse.fill_(float("nan"))
        g.replay()
        torch.cuda.synchronize()
        assert m.mocap_last_device_status() == 0
        _, _, out_h, lse_h = _run_both(m, q, k, v, chosen, scale)
        assert _equal_bits(out, out_h) and _equal_bits(lse, lse_h)


def test_no_items_and_empty_items(m):
    dev = torch.device("cuda")
    q = torch.randn((64, 8, 128), device=dev).bfloat16()
    k = torch.randn((64, 2, 128), device=dev).bfloat16()
    out = torch.full((64, 8, 128), 5.0, device=dev, dtype=torch.bfloat16)
    lse = torch.full((8, 64), 5.0, device=dev, dtype=torch.float32)
    none = torch.zeros((0, 4), dtype=torch.int64, device=dev)
    lib = m._lib.load()
    stream = torch.cuda.current_stream().cuda_stream
    assert lib.mocap_chunk_attn_varlen_dev(q.data_ptr(), k.data_ptr(), k.data_ptr(), None, 0, 64,
                                           64, 64, 8, 2, 128, 0.1, out.data_ptr(), lse.data_ptr(),
                                           None, 0, stream) == 0
    empty = torch.tensor([(0, 0, 10, 0), (5, 3, 0, 0)], dtype=torch.int64, device=dev)
    m.mocap_chunk_attn_varlen_dev(q, k, k, empty, out, lse, 0.1)
    torch.cuda.synchronize()
    assert m.mocap_last_device_status() == 0
    assert bool((out.float() == 5.0).all()) and bool((lse == 5.0).all())
    assert none.numel() == 0


@pytest.mark.parametrize("case", range(20))
def test_random_device_items_sweep(m, monkeypatch, case):
    """Seeded random launches of 1..400 device items (some empty, random
    prefixes, items in random order), heads, head dim and kernel form drawn
    per case: bitwise equal to the host-array form, rows outside every item
    untouched; in a third of the cases one item is made invalid, and then
    the call writes nothing and reports MOCAP_EINVAL."""
    rng = np.random.default_rng(9100 + case)
    heads = [(4, 4), (8, 2), (16, 2), (32, 8), (16, 1), (6, 2)]
    hq, hkv = heads[int(rng.integers(len(heads)))]
    d = 128 if rng.random() < 0.7 else 64
    monkeypatch.setenv("MOCAP_ATTN_PAIR", str(int(rng.integers(2))))
    n_req = int(rng.choice([1, int(rng.integers(2, 65)), int(rng.integers(65, 401))]))
    lens = [int(x) for x in rng.integers(1, 800 if n_req > 64 else 3000, n_req)]
    cu = np.concatenate([[0], np.cumsum(lens)]).tolist()
    t = cu[-1]
    items = []
    for r, n in enumerate(lens):
        pre = int(rng.integers(0, n))
        ln = int(rng.integers(0, n - pre + 1)) if rng.random() < 0.9 else 0
        items.append((cu[r] + pre, cu[r], pre, ln))
    items = [items[i] for i in rng.permutation(len(items))]
    dev = torch.device("cuda")
    gen = torch.Generator(device=dev).manual_seed(9100 + case)
    q = torch.randn((t, hq, d), generator=gen, device=dev, dtype=torch.bfloat16)
    k = torch.randn((t, hkv, d), generator=gen, device=dev, dtype=torch.bfloat16)
    v = torch.randn((t, hkv, d), generator=gen, device=dev, dtype=torch.bfloat16)
    scale = 1.0 / math.sqrt(d)
    if case % 3 == 2:
        j = int(rng.integers(len(items)))
        qr, kr, pre, ln = items[j]
        items[j] = (qr, kr, pre, t + 1)  # rows past both buffers
        out = torch.full((t, hq, d), float("nan"), device=dev, dtype=torch.bfloat16)
        lse = torch.full((hq, t), float("nan"), device=dev, dtype=torch.float32)
        it = torch.tensor(items, dtype=torch.int64, device=dev)
        m.mocap_chunk_attn_varlen_dev(q, k, v, it, out, lse, scale)
        torch.cuda.synchronize()
        assert m.mocap_last_device_status() == m.MOCAP_EINVAL
        assert torch.isnan(out.float()).all() and torch.isnan(lse).all()
        return
    out_d, lse_d, out_h, lse_h = _run_both(m, q, k, v, items, scale)
    assert _equal_bits(out_d, out_h) and _equal_bits(lse_d, lse_h)
    covered = torch.zeros(t, dtype=torch.bool)
    for (qr, _, _, ln) in items:
        covered[qr:qr + ln] = True
    cov = covered.to(dev)
    assert torch.isnan(out_d[~cov].float()).all() and torch.isnan(lse_d[:, ~cov]).all()
    assert torch.isfinite(out_d[cov].float()).all()
