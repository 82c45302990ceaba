"""GPU: mocap_kv_append and mocap_kv_append_overlap (the one-warp kernel that
runs beside attention launches) write exactly the chunk rows, bit for bit,
and no other cache byte (sentinel bit patterns, NaN included, must
survive)."""

import numpy as np
import pytest
import torch

from oracle import attention as A

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def m():
    import paper_2606_22968_gb300 as mod
    mod._lib.load()
    return mod


APPENDS = ["mocap_kv_append", "mocap_kv_append_overlap"]


@pytest.mark.parametrize("fn", APPENDS)
@pytest.mark.parametrize("cap,offset,length,hkv,d", [
    (1000, 0, 1000, 8, 128),
    (1000, 3, 1, 8, 128),
    (4099, 1234, 2047, 8, 128),
    (513, 511, 2, 4, 64),
    (300, 17, 250, 1, 8),
    (70000, 65536, 4464, 8, 128),
])
def test_append_bitwise_with_sentinels(m, fn, cap, offset, length, hkv, d):
    dev = torch.device("cuda")
    gen = torch.Generator(device=dev).manual_seed(cap + offset)
    sentinel = torch.randint(-32768, 32767, (cap, hkv, d), generator=gen, device=dev,
                             dtype=torch.int16)
    sentinel[::7] = 0x7FC1  # NaN bit patterns among the sentinels
    kc = sentinel.clone().view(torch.bfloat16)
    vc = (sentinel ^ 0x5555).view(torch.bfloat16)
    k = torch.randint(-32768, 32767, (length, hkv, d), generator=gen, device=dev,
                      dtype=torch.int16).view(torch.bfloat16)
    v = torch.randint(-32768, 32767, (length, hkv, d), generator=gen, device=dev,
                      dtype=torch.int16).view(torch.bfloat16)
    kc0 = kc.view(torch.int16).cpu().numpy()
    vc0 = vc.view(torch.int16).cpu().numpy()
    getattr(m, fn)(k, v, kc, vc, offset)
    torch.cuda.synchronize()
    k_ref = A.kv_append(kc0, k.view(torch.int16).cpu().numpy(), offset)
    v_ref = A.kv_append(vc0, v.view(torch.int16).cpu().numpy(), offset)
    assert np.array_equal(kc.view(torch.int16).cpu().numpy(), k_ref)
    assert np.array_equal(vc.view(torch.int16).cpu().numpy(), v_ref)


@pytest.mark.parametrize("fn", APPENDS)
def test_append_rejects_overflow(m, fn):
    dev = torch.device("cuda")
    kc = torch.zeros((10, 8, 128), device=dev, dtype=torch.bfloat16)
    k = torch.zeros((4, 8, 128), device=dev, dtype=torch.bfloat16)
    with pytest.raises(m.MocapError):
        getattr(m, fn)(k, k, kc, kc.clone(), 7)


@pytest.mark.parametrize("fn", APPENDS)
@pytest.mark.parametrize("case", range(30))
def test_random_append_sweep(m, fn, case):
    """Seeded random appends (rows a whole number of 16-byte vectors):
    bitwise equal to the oracle's copy, every other cache row untouched."""
    rng = np.random.default_rng(60 + case)
    hkv = int(rng.choice([1, 2, 4, 8, 16]))
    d = int(rng.choice([8, 16, 64, 128, 256]))
    length = int(rng.choice([int(rng.integers(1, 64)), int(rng.integers(64, 20000))]))
    offset = int(rng.integers(0, 50000))
    cap = offset + length + int(rng.integers(0, 100))
    test_append_bitwise_with_sentinels(m, fn, cap, offset, length, hkv, d)
