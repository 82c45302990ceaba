"""GPU parity of the fused QKV projection + RoPE + KV append against the
float64 oracle (every element), with cache rows outside the chunk kept."""

import math

import numpy as np
import pytest
import torch

from oracle import projection as R
from tests.parity_utils import f64

pytestmark = pytest.mark.gpu

TOL_MAX, TOL_MEAN = 2e-2, 2e-3


@pytest.fixture(scope="module")
def m():
    import paper_2606_22968_gb300 as mod
    mod._lib.load()
    return mod


CASES = [
    # (len, hidden, Hq, Hkv, d, offset, theta)
    (300, 1024, 4, 2, 128, 0, 500000.0),
    (1, 256, 4, 2, 128, 77, 500000.0),
    (129, 200, 8, 8, 64, 1000, 10000.0),      # hidden not a multiple of 64
    (1000, 512, 2, 1, 128, 130000, 500000.0),  # large positions
    (512, 2048, 16, 2, 128, 4096, 500000.0),   # GQA 8:1, several n tiles
]


@pytest.mark.parametrize("length,hidden,hq,hkv,d,offset,theta", CASES)
def test_qkv_rope_append_matches_oracle(m, length, hidden, hq, hkv, d, offset, theta):
    dev = torch.device("cuda")
    gen = torch.Generator(device=dev).manual_seed(length + hidden + offset)
    x = torch.randn((length, hidden), generator=gen, device=dev).bfloat16()
    n_out = (hq + 2 * hkv) * d
    w = (torch.randn((n_out, hidden), generator=gen, device=dev) / math.sqrt(hidden)).bfloat16()
    cap = offset + length + 5
    sentinel = torch.randint(-30000, 30000, (cap, hkv, d), generator=gen, device=dev,
                             dtype=torch.int16)
    kc = sentinel.clone().view(torch.bfloat16)
    vc = (sentinel ^ 0x1234).view(torch.bfloat16)
    k0, v0 = kc.clone(), vc.clone()
    q = torch.full((length, hq, d), float("nan"), device=dev, dtype=torch.bfloat16)
    m.mocap_qkv_rope_append(x, w, q, kc, vc, offset, rope_theta=theta)
    torch.cuda.synchronize()
    assert m.mocap_last_device_status() == 0
    q_ref, k_ref, v_ref = R.qkv_rope(f64(x), f64(w), hq, hkv, d, offset, theta)
    for got, ref, name in [(q, q_ref, "Q"), (kc[offset:offset + length], k_ref, "K"),
                           (vc[offset:offset + length], v_ref, "V")]:
        err = np.abs(got.float().cpu().numpy() - ref)
        assert err.max() <= TOL_MAX and err.mean() <= TOL_MEAN, (name, err.max(), err.mean())
    # rows outside the chunk keep their bytes (compared as bit patterns: the
    # sentinels include NaN encodings)
    bits = lambda t: t.view(torch.int16)  # noqa: E731
    for got, ref in [(kc, k0), (vc, v0)]:
        assert torch.equal(bits(got[:offset]), bits(ref[:offset]))
        assert torch.equal(bits(got[offset + length:]), bits(ref[offset + length:]))


def test_qkv_rope_rejects_bad_shapes(m):
    dev = torch.device("cuda")
    x = torch.zeros((10, 128), device=dev, dtype=torch.bfloat16)
    w = torch.zeros((3 * 64 * 2, 128), device=dev, dtype=torch.bfloat16)  # (2+2*2)*64=384: not /256
    q = torch.zeros((10, 2, 64), device=dev, dtype=torch.bfloat16)
    kc = torch.zeros((20, 2, 64), device=dev, dtype=torch.bfloat16)
    with pytest.raises(m.MocapError):
        m.mocap_qkv_rope_append(x, w, q, kc, kc.clone(), 0)
    x2 = torch.zeros((10, 128), device=dev, dtype=torch.bfloat16)
    w2 = torch.zeros((4 * 128, 128), device=dev, dtype=torch.bfloat16)
    q2 = torch.zeros((10, 2, 128), device=dev, dtype=torch.bfloat16)
    kc2 = torch.zeros((12, 1, 128), device=dev, dtype=torch.bfloat16)
    with pytest.raises(m.MocapError):   # offset + len past the cache
        m.mocap_qkv_rope_append(x2, w2, q2, kc2, kc2.clone(), 5)


@pytest.mark.parametrize("length,offset", [(4096, 61440), (2000, 129024)])
def test_qkv_rope_full_size_sampled_rows(m, length, offset):
    """Llama-3-70B projection shapes as the benchmark launches them (hidden
    8192, 64 + 2 x 8 heads of 128; a 4096-row chunk and a ragged 2000-row one
    near the end of a 131072-token prompt): sampled rows, including the tile
    edges of the 256-row pair tiles and the ragged tail, against the oracle
    row by row (each at its own position)."""
    from tests.parity_utils import sample_rows
    hidden, hq, hkv, d, theta = 8192, 64, 8, 128, 500000.0
    dev = torch.device("cuda")
    gen = torch.Generator(device=dev).manual_seed(length + offset)
    x = torch.randn((length, hidden), generator=gen, device=dev).bfloat16()
    n_out = (hq + 2 * hkv) * d
    w = (torch.randn((n_out, hidden), generator=gen, device=dev) / math.sqrt(hidden)).bfloat16()
    cap = offset + length
    kc = torch.zeros((cap, hkv, d), device=dev, dtype=torch.bfloat16)
    vc = torch.zeros_like(kc)
    q = torch.full((length, hq, d), float("nan"), device=dev, dtype=torch.bfloat16)
    m.mocap_qkv_rope_append(x, w, q, kc, vc, offset, rope_theta=theta)
    torch.cuda.synchronize()
    assert m.mocap_last_device_status() == 0
    rows = sample_rows(length, every=509, edge=2, seed=length)
    rows = np.unique(np.concatenate([rows, [r for r in (255, 256, 511, 512) if r < length]]))
    wf = f64(w)
    for r in rows:
        q_ref, k_ref, v_ref = R.qkv_rope(f64(x[r:r + 1]), wf, hq, hkv, d, offset + int(r), theta)
        for got, ref, name in [(q[r:r + 1], q_ref, "Q"), (kc[offset + r:offset + r + 1], k_ref, "K"),
                               (vc[offset + r:offset + r + 1], v_ref, "V")]:
            err = np.abs(got.float().cpu().numpy() - ref)
            assert err.max() <= TOL_MAX and err.mean() <= TOL_MEAN, (name, int(r), err.max(),
                                                                   err.mean())


@pytest.mark.parametrize("overlap", [False, True])
def test_run_stage_projection_then_attention(m, overlap):
    """ChunkedPrefill.run_stage: per chunk the fused projection writes Q and
    the chunk's K/V rows, then attention reads the cache.  The projection
    outputs match the projection oracle, and the attention matches the
    attention oracle on the exact Q/K/V bits the projection produced (every
    chunk, sampled rows), so positions and cache rows line up across the
    two kernels.  ``overlap``: projections on their own stream, attention
    alternating between two compute streams, each chunk's attention waiting
    only for its own projection."""
    from oracle import attention as A
    from paper_2606_22968_gb300 import workloads
    from paper_2606_22968_gb300.pipeline import ChunkedPrefill
    from tests.parity_utils import assert_close, chunk_rows_oracle, sample_rows
    w = workloads.custom("stage-8k-lbcp8-h16-g4-d128", (8192,), (8,), workloads.MODE_LBCP, 16, 4,
                         128)
    hidden, theta = 256, 500000.0
    dev = torch.device("cuda")
    gen = torch.Generator(device=dev).manual_seed(8192)
    x = torch.randn((8192, hidden), generator=gen, device=dev).bfloat16()
    n_out = (w.n_q_heads + 2 * w.n_kv_heads) * w.head_dim
    wq = (torch.randn((n_out, hidden), generator=gen, device=dev) / math.sqrt(hidden)).bfloat16()
    pf = ChunkedPrefill(w, dev)
    qbuf = torch.full((8192, w.n_q_heads, w.head_dim), float("nan"), device=dev,
                      dtype=torch.bfloat16)
    pf.run_stage(x, wq, qbuf, rope_theta=theta, overlap=overlap)
    torch.cuda.synchronize()
    assert m.mocap_last_device_status() == 0
    q_ref, k_ref, v_ref = R.qkv_rope(f64(x), f64(wq), w.n_q_heads, w.n_kv_heads, w.head_dim, 0,
                                     theta)
    for got, ref, name in [(qbuf, q_ref, "Q"), (pf.k_cache, k_ref, "K"), (pf.v_cache, v_ref, "V")]:
        err = np.abs(got.float().cpu().numpy() - ref)
        assert err.max() <= TOL_MAX and err.mean() <= TOL_MEAN, (name, err.max(), err.mean())
    b = pf.bounds[0]
    kf, vf = f64(pf.k_cache), f64(pf.v_cache)
    for i in range(len(b) - 1):
        rows = sample_rows(b[i + 1] - b[i], every=211, edge=2, seed=i)
        idx = torch.as_tensor(rows, device=dev)
        o_ref, l_ref = chunk_rows_oracle(f64(qbuf[b[i]:b[i + 1]][idx]), kf[:b[i + 1]],
                                         vf[:b[i + 1]], b[i], rows, w.scale)
        assert_close(pf.out[b[i]:b[i + 1]][idx].float().cpu().numpy(),
                     pf.chunk_lse(i)[:, idx].cpu().numpy(), o_ref, l_ref, f"chunk {i}")


def _random_projection_case(i):
    rng = np.random.default_rng(4242 + i)
    while True:
        hkv = int(rng.choice([1, 2, 4, 8]))
        hq = hkv * int(rng.choice([1, 2, 4, 8]))
        d = 128 if rng.random() < 0.7 else 64
        if (hq + 2 * hkv) * d % 256 == 0 and (hq + 2 * hkv) * d <= 4096:
            break
    hidden = 8 * int(rng.integers(1, 129))
    length = int(rng.choice([int(rng.integers(1, 129)), int(rng.integers(129, 1500))]))
    offset = int(rng.choice([0, int(rng.integers(1, 1000)), int(rng.integers(1000, 200000))]))
    theta = float(rng.choice([10000.0, 500000.0, 1000000.0]))
    return length, hidden, hq, hkv, d, offset, theta


@pytest.mark.parametrize("case", range(25))
def test_random_projection_sweep(m, case):
    """Seeded random shapes of the fused QKV projection + RoPE + append
    (any hidden size that keeps 16-byte rows, whole 256-column output
    tiles, positions up to 200000) against the oracle, every element; cache
    rows outside the chunk keep their bytes."""
    length, hidden, hq, hkv, d, offset, theta = _random_projection_case(case)
    test_qkv_rope_append_matches_oracle(m, length, hidden, hq, hkv, d, offset, theta)
