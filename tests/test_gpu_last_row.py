"""GPU parity of the last-row-only attention (each request's final prompt row
against all its keys) with the float64 oracle, and against the chunk kernel
run on the same one-row chunk."""

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


CASES = [
    # (lengths, Hq, Hkv, d)
    ([23168, 9344, 5504, 4224, 7424, 6144, 6528, 8448], 32, 8, 128),  # the varlen workload
    ([131072], 64, 8, 128),
    ([1, 2, 127, 128, 129, 300, 4097], 8, 2, 128),                    # ragged, tiny
    ([1000, 50], 4, 4, 64),
    ([3000], 16, 1, 128),                                              # group of 16
    ([int(x) for x in np.random.default_rng(5).integers(1, 2500, 64)], 16, 4, 64),  # 64 requests
]


@pytest.mark.parametrize("lens,hq,hkv,d", CASES)
def test_last_row_matches_oracle_and_chunk_kernel(m, lens, hq, hkv, d):
    dev = torch.device("cuda")
    gen = torch.Generator(device=dev).manual_seed(sum(lens) + hq)
    cu = np.concatenate([[0], np.cumsum(lens)]).tolist()
    total = cu[-1] + 3
    k = torch.randn((total, hkv, d), generator=gen, device=dev, dtype=torch.bfloat16)
    v = torch.randn((total, hkv, d), generator=gen, device=dev, dtype=torch.bfloat16)
    k[cu[-1]:] = float("nan")   # rows past every request are never read
    v[cu[-1]:] = float("nan")
    n = len(lens)
    q = torch.randn((n, hq, d), generator=gen, device=dev, dtype=torch.bfloat16)
    scale = 1.0 / math.sqrt(d)
    out = torch.full((n, hq, d), float("nan"), device=dev, dtype=torch.bfloat16)
    lse = torch.full((hq, n), float("nan"), device=dev, dtype=torch.float32)
    m.mocap_last_row_attn(q, k, v, cu[:-1], lens, out, lse, scale)
    torch.cuda.synchronize()
    assert m.mocap_last_device_status() == 0
    for r, length in enumerate(lens):
        a = cu[r]
        o_ref, l_ref = A.chunk_attention(f64(q[r:r + 1]), f64(k[a:a + length]),
                                         f64(v[a:a + length]), length - 1, scale)
        assert_close(out[r:r + 1].float().cpu().numpy(), lse[:, r:r + 1].cpu().numpy(), o_ref,
                     l_ref, f"request {r} (len {length})")
        # the chunk kernel on the same one-row chunk agrees
        oc = torch.empty((1, hq, d), device=dev, dtype=torch.bfloat16)
        lc = torch.empty((hq, 1), device=dev, dtype=torch.float32)
        m.mocap_chunk_attn(q[r:r + 1], k[a:a + length], v[a:a + length], length - 1, oc, lc, scale)
        torch.cuda.synchronize()
        assert (oc.float() - out[r:r + 1].float()).abs().max().item() <= 1e-2
        assert (lc - lse[:, r:r + 1]).abs().max().item() <= 1e-4


def test_last_row_rejects_bad_arguments(m):
    dev = torch.device("cuda")
    q = torch.zeros((2, 8, 128), device=dev, dtype=torch.bfloat16)
    k = torch.zeros((100, 2, 128), device=dev, dtype=torch.bfloat16)
    out = torch.zeros_like(q)
    lse = torch.zeros((8, 2), device=dev, dtype=torch.float32)
    with pytest.raises(m.MocapError):   # request past the cache
        m.mocap_last_row_attn(q, k, k, [0, 60], [50, 50], out, lse, 0.1)
    with pytest.raises(m.MocapError):   # empty request
        m.mocap_last_row_attn(q, k, k, [0, 10], [50, 0], out, lse, 0.1)


def test_last_row_workspace_garbage_and_reuse(m):
    """The per-group arrival counters live in the caller's workspace: the call
    zeroes them itself, so a workspace full of garbage, and the same workspace
    reused, give bit-identical results (the merge order does not depend on
    which CTA finishes last)."""
    dev = torch.device("cuda")
    gen = torch.Generator(device=dev).manual_seed(11)
    lens = [131072, 4096]
    hq, hkv, d = 64, 8, 128
    total = sum(lens)
    k = torch.randn((total, hkv, d), generator=gen, device=dev, dtype=torch.bfloat16)
    v = torch.randn((total, hkv, d), generator=gen, device=dev, dtype=torch.bfloat16)
    q = torch.randn((2, hq, d), generator=gen, device=dev, dtype=torch.bfloat16)
    rows = [0, lens[0]]
    need = m.mocap_last_row_attn_workspace_size(lens, hq, hkv, d)
    ws = torch.full((need,), 0xFF, device=dev, dtype=torch.uint8)
    outs = []
    for _ in range(3):
        out = torch.empty((2, hq, d), device=dev, dtype=torch.bfloat16)
        lse = torch.empty((hq, 2), device=dev, dtype=torch.float32)
        m.mocap_last_row_attn(q, k, v, rows, lens, out, lse, 0.088, workspace=ws)
        outs.append((out, lse))
    torch.cuda.synchronize()
    assert m.mocap_last_device_status() == 0
    for out, lse in outs[1:]:
        assert torch.equal(out.view(torch.int16), outs[0][0].view(torch.int16))
        assert torch.equal(lse.view(torch.int32), outs[0][1].view(torch.int32))
    # and the result is the attention of the last row (the oracle, request 1)
    a = lens[0]
    o_ref, l_ref = A.chunk_attention(f64(q[1:2]), f64(k[a:]), f64(v[a:]), lens[1] - 1, 0.088)
    assert_close(outs[0][0][1:2].float().cpu().numpy(), outs[0][1][:, 1:2].cpu().numpy(), o_ref,
                 l_ref, "request 1")


@pytest.mark.parametrize("case", range(30))
def test_random_last_row_sweep(m, case):
    """Seeded random last-row calls: 1..64 requests of 1..20000 keys, group
    sizes up to 16, head dim 64 or 128, NaN cache rows past every request;
    each request's row against the oracle."""
    rng = np.random.default_rng(31337 + case)
    heads = [(4, 4), (8, 2), (16, 2), (32, 8), (16, 1), (64, 8), (64, 4)]
    hq, hkv = heads[int(rng.integers(len(heads)))]
    d = 128 if rng.random() < 0.7 else 64
    n = int(rng.choice([1, int(rng.integers(2, 9)), int(rng.integers(9, 65))]))
    lens = [int(x) for x in rng.integers(1, 20001 if n <= 8 else 3000, n)]
    cu = np.concatenate([[0], np.cumsum(lens)]).tolist()
    dev = torch.device("cuda")
    gen = torch.Generator(device=dev).manual_seed(900 + case)
    total = cu[-1] + 5
    k = torch.randn((total, hkv, d), generator=gen, device=dev, dtype=torch.bfloat16)
    v = torch.randn((total, hkv, d), generator=gen, device=dev, dtype=torch.bfloat16)
    k[cu[-1]:] = float("nan")
    v[cu[-1]:] = float("nan")
    q = torch.randn((n, hq, d), generator=gen, device=dev, dtype=torch.bfloat16)
    scale = 1.0 / math.sqrt(d)
    out = torch.full((n, hq, d), float("nan"), device=dev, dtype=torch.bfloat16)
    lse = torch.full((hq, n), float("nan"), device=dev, dtype=torch.float32)
    m.mocap_last_row_attn(q, k, v, cu[:-1], lens, out, lse, scale)
    torch.cuda.synchronize()
    assert m.mocap_last_device_status() == 0
    for r, length in enumerate(lens):
        a = cu[r]
        o_ref, l_ref = A.chunk_attention(f64(q[r:r + 1]), f64(k[a:a + length]),
                                         f64(v[a:a + length]), length - 1, scale)
        assert_close(out[r:r + 1].float().cpu().numpy(), lse[:, r:r + 1].cpu().numpy(), o_ref,
                     l_ref, f"case {case} request {r} (len {length}, heads {hq}/{hkv}, d {d})")
