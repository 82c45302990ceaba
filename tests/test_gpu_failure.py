"""GPU failure detection without a GPU fault: a bounded wait that expires
records MOCAP_ETIMEOUT, the host reads (and clears) it, launches made while
it is set do nothing, and the context stays usable."""

import math
import time

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


def _small(dev, seed=3):
    gen = torch.Generator(device=dev).manual_seed(seed)
    q = torch.randn((300, 8, 128), generator=gen, device=dev, dtype=torch.bfloat16)
    k = torch.randn((300, 2, 128), generator=gen, device=dev, dtype=torch.bfloat16)
    v = torch.randn((300, 2, 128), generator=gen, device=dev, dtype=torch.bfloat16)
    return q, k, v


def test_expired_wait_is_reported_and_cleared(m):
    assert m.mocap_last_device_status() == m.MOCAP_OK
    t0 = time.perf_counter()
    m.mocap_selftest_bounded_wait(50000)  # 50 ms
    st = m.mocap_last_device_status()     # synchronises the stream
    elapsed = time.perf_counter() - t0
    assert st == m.MOCAP_ETIMEOUT
    assert elapsed >= 0.045
    assert m.mocap_last_device_status() == m.MOCAP_OK  # read clears it


@pytest.mark.parametrize("pair,split", [("1", None), ("0", None), ("1", 2), ("0", 2)])
def test_launch_after_expired_wait_does_nothing_then_recovers(m, monkeypatch, pair, split):
    # both attention forms: CTA pairs (both CTAs act on the first CTA's
    # reading of the status word) and single CTAs.  With split-KV (rows
    # 128..299 over two key tiles) no split arrives, so nothing is merged,
    # and the next call's counters start at 0 again.
    monkeypatch.setenv("MOCAP_ATTN_PAIR", pair)
    dev = torch.device("cuda")
    q_all, k, v = _small(dev)
    prefix = 0 if split is None else 128
    q = q_all[prefix:].contiguous()
    rows = q.shape[0]
    ws = None
    if split is not None:
        monkeypatch.setenv("MOCAP_SPLIT_KV", str(split))
        need = m.mocap_chunk_attn_workspace_size(prefix, rows, 8, 2, 128)
        assert need > 0
        ws = torch.empty((need,), device=dev, dtype=torch.uint8)
    out = torch.full_like(q, float("nan"))
    lse = torch.full((8, rows), float("nan"), device=dev, dtype=torch.float32)
    m.mocap_selftest_bounded_wait(20000)
    m.mocap_chunk_attn(q, k, v, prefix, out, lse, 0.088, workspace=ws)  # behind the expired wait
    torch.cuda.synchronize()
    assert torch.isnan(out.float()).all() and torch.isnan(lse).all()
    assert m.mocap_last_device_status() == m.MOCAP_ETIMEOUT
    # the context is usable: the same launch now computes the right answer
    m.mocap_chunk_attn(q, k, v, prefix, out, lse, 0.088, workspace=ws)
    torch.cuda.synchronize()
    assert m.mocap_last_device_status() == m.MOCAP_OK
    o_ref, l_ref = A.causal_attention(f64(q_all), f64(k), f64(v), 0.088)
    assert_close(out.float().cpu().numpy(), lse.cpu().numpy(), o_ref[prefix:], l_ref[:, prefix:])


def test_selftest_rejects_bad_limits(m):
    for bad in (0, 1000001):
        with pytest.raises(m.MocapError):
            m.mocap_selftest_bounded_wait(bad)
