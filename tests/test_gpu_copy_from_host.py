"""GPU: mocap_copy_from_host, host -> device copies by the SMs.  Bytes land
exactly (both launch forms, ragged sizes, several ranges per launch, bytes
around the ranges untouched); sources that are not page-locked host memory,
or destinations that are not device memory, are refused before any launch;
the host-memory pipeline gives the same bits with kernel and copy-engine
uploads."""

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def m():
    import paper_2606_22968_gb300 as mod
    mod._lib.load()
    return mod


@pytest.mark.parametrize("beside", [False, True])
@pytest.mark.parametrize("sizes", [[16], [4096, 16, 48], [1 << 20, 3 << 20, 12345 * 16],
                                   [64 << 20, 16 << 20, 32, 8 << 20, 1024, 48, 160, 5 << 20]])
def test_copies_land_exactly(m, beside, sizes):
    dev = torch.device("cuda")
    rng = np.random.default_rng(sum(sizes) + beside)
    pairs, checks = [], []
    for n in sizes:
        host = torch.from_numpy(rng.integers(0, 256, n + 64, dtype=np.uint8)).pin_memory()
        dst = torch.full((n + 64,), 0xA5, device=dev, dtype=torch.uint8)
        pairs.append((dst[16:16 + n], host[32:32 + n]))
        checks.append((dst, host, n))
    m.mocap_copy_from_host(pairs, beside_kernels=beside)
    torch.cuda.synchronize()
    for dst, host, n in checks:
        got = dst.cpu()
        assert torch.equal(got[16:16 + n], host[32:32 + n])
        assert bool((got[:16] == 0xA5).all()) and bool((got[16 + n:] == 0xA5).all())


def test_refuses_what_is_not_pinned_host_memory(m):
    dev = torch.device("cuda")
    dst = torch.empty(4096, device=dev, dtype=torch.uint8)
    pageable = torch.zeros(4096, dtype=torch.uint8)
    pinned = torch.zeros(4096, dtype=torch.uint8).pin_memory()
    other = torch.zeros(4096, device=dev, dtype=torch.uint8)
    lib = m._lib.load()
    from paper_2606_22968_gb300._lib import CopyItem

    def call(d, s):
        arr = (CopyItem * 1)(CopyItem(d, s, 4096))
        return lib.mocap_copy_from_host(arr, 1, 0, torch.cuda.current_stream().cuda_stream)

    assert call(dst.data_ptr(), pageable.data_ptr()) == m.MOCAP_EINVAL
    assert call(dst.data_ptr(), other.data_ptr()) == m.MOCAP_EINVAL   # device memory as source
    assert call(pinned.data_ptr(), pinned.data_ptr()) == m.MOCAP_EINVAL  # host memory as target
    assert call(dst.data_ptr(), pinned.data_ptr()) == m.MOCAP_OK
    torch.cuda.synchronize()


@pytest.mark.parametrize("index", [3, 5])
def test_pipeline_uploads_kernel_equals_copy_engine(m, index):
    """run_from_host with both upload forms: O and LSE bitwise equal."""
    from paper_2606_22968_gb300 import workloads
    from paper_2606_22968_gb300.pipeline import ChunkedPrefill
    w = workloads.get(index)
    dev = torch.device("cuda")
    q, k, v = workloads.make_qkv(w, dev)
    hq, hk, hv = (t.cpu().pin_memory() for t in (q, k, v))
    outs = []
    for upload in ("kernel", "copy_engine"):
        pf = ChunkedPrefill(w, dev, upload=upload)
        ho = torch.full(pf.out.shape, float("nan"), dtype=pf.out.dtype).pin_memory()
        hl = torch.full(pf.lse.shape, float("nan"), dtype=pf.lse.dtype).pin_memory()
        dq, dk, dv = torch.empty_like(q), torch.empty_like(k), torch.empty_like(v)
        pf.partition()
        pf.run_from_host(hq, hk, hv, ho, hl, dq, dk, dv)
        torch.cuda.synchronize()
        assert m.mocap_last_device_status() == 0
        assert torch.equal(dq, q) and torch.equal(dk, k) and torch.equal(dv, v)
        outs.append((ho.view(torch.int16).clone(), hl.clone()))
    assert torch.equal(outs[0][0], outs[1][0]) and torch.equal(outs[0][1], outs[1][1])
    assert not torch.isnan(outs[0][1]).any()
