"""GPU: mocap_copy_from_host / mocap_copy_to_host, host <-> device copies by
the SMs.  Bytes land exactly (both launch forms, ragged sizes, several
ranges per launch, bytes around the ranges untouched); ranges in the wrong
kind of memory are refused before any launch; the host-memory pipeline
(one prompt, and prompts streamed) gives the same bits with kernel and
copy-engine copies."""

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


@pytest.mark.parametrize("beside", [False, True])
@pytest.mark.parametrize("sizes", [[16], [4096, 16, 48], [3 << 20, 12345 * 16, 64 << 20]])
def test_copies_back_land_exactly(m, beside, sizes):
    dev = torch.device("cuda")
    gen = torch.Generator(device=dev).manual_seed(sum(sizes) + beside)
    pairs, checks = [], []
    for n in sizes:
        src = torch.randint(0, 256, (n + 64,), generator=gen, device=dev, dtype=torch.uint8)
        host = torch.full((n + 64,), 0x5A, dtype=torch.uint8).pin_memory()
        pairs.append((host[16:16 + n], src[32:32 + n]))
        checks.append((host, src, n))
    m.mocap_copy_to_host(pairs, beside_kernels=beside)
    torch.cuda.synchronize()
    for host, src, n in checks:
        assert torch.equal(host[16:16 + n], src[32:32 + n].cpu())
        assert bool((host[:16] == 0x5A).all()) and bool((host[16 + n:] == 0x5A).all())


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

    def back(d, s):
        arr = (CopyItem * 1)(CopyItem(d, s, 4096))
        return lib.mocap_copy_to_host(arr, 1, 1, torch.cuda.current_stream().cuda_stream)

    assert back(pageable.data_ptr(), dst.data_ptr()) == m.MOCAP_EINVAL
    assert back(other.data_ptr(), dst.data_ptr()) == m.MOCAP_EINVAL    # device memory as target
    assert back(pinned.data_ptr(), pinned.data_ptr()) == m.MOCAP_EINVAL  # host memory as source
    assert back(pinned.data_ptr(), dst.data_ptr()) == m.MOCAP_OK
    torch.cuda.synchronize()


@pytest.mark.parametrize("index", [3, 5])
def test_pipeline_host_copies_kernel_equals_copy_engine(m, index):
    """run_from_host and run_prompts_from_host (three prompts) with every
    form of host copies: O and LSE bitwise equal."""
    from paper_2606_22968_gb300 import workloads
    from paper_2606_22968_gb300.pipeline import ChunkedPrefill
    w = workloads.get(index)
    dev = torch.device("cuda")
    q, k, v = workloads.make_qkv(w, dev)
    hq, hk, hv = (t.cpu().pin_memory() for t in (q, k, v))
    outs = []
    for mode in ("kernel", "copy_engine", "auto"):
        pf = ChunkedPrefill(w, dev, host_copies=mode)
        ho = torch.full(pf.out.shape, float("nan"), dtype=pf.out.dtype).pin_memory()
        hl = torch.full(pf.lse.shape, float("nan"), dtype=pf.lse.dtype).pin_memory()
        dq, dk, dv = torch.empty_like(q), torch.empty_like(k), torch.empty_like(v)
        pf.partition()
        pf.run_from_host(hq, hk, hv, ho, hl, dq, dk, dv)
        torch.cuda.synchronize()
        assert m.mocap_last_device_status() == 0
        assert torch.equal(dq, q) and torch.equal(dk, k) and torch.equal(dv, v)
        outs.append((ho.view(torch.int16).clone(), hl.clone()))
        # three prompts streamed (the second and third are the first's inputs
        # with Q scaled, so every prompt's results differ)
        hqs = [hq] + [(q * s).cpu().pin_memory() for s in (0.5, 2.0)]
        prompts = [(x, hk, hv,
                    torch.full(pf.out.shape, float("nan"), dtype=pf.out.dtype).pin_memory(),
                    torch.full(pf.lse.shape, float("nan"), dtype=pf.lse.dtype).pin_memory())
                   for x in hqs]
        bufs = [(dq, dk, dv), (torch.empty_like(q), torch.empty_like(k), torch.empty_like(v))]
        pf.partition()
        pf.run_prompts_from_host(prompts, bufs)
        torch.cuda.synchronize()
        assert m.mocap_last_device_status() == 0
        outs.append(tuple(t.view(torch.int16).clone() if t.dtype == torch.bfloat16 else t.clone()
                          for pr in prompts for t in pr[3:]))
    for j in (2, 4):  # every mode gives the bits of the first
        assert all(torch.equal(a, b) for a, b in zip(outs[0], outs[j]))
        assert all(torch.equal(a, b) for a, b in zip(outs[1], outs[j + 1]))
    assert torch.equal(outs[0][0], outs[1][0]) and torch.equal(outs[0][1], outs[1][1])
    assert not torch.isnan(outs[0][1]).any() and not torch.isnan(outs[1][-1]).any()


def test_pipeline_with_pageable_host_tensors(m):
    """Host tensors that are not page-locked have no device mapping: the
    pipeline moves them with the copy engines instead, same bits."""
    from paper_2606_22968_gb300 import workloads
    from paper_2606_22968_gb300.pipeline import ChunkedPrefill
    w = workloads.get(2)
    dev = torch.device("cuda")
    q, k, v = workloads.make_qkv(w, dev)
    res = []
    for pin in (True, False):
        hq, hk, hv = (t.cpu() for t in (q, k, v))
        pf = ChunkedPrefill(w, dev)
        ho = torch.full(pf.out.shape, float("nan"), dtype=pf.out.dtype)
        hl = torch.full(pf.lse.shape, float("nan"), dtype=pf.lse.dtype)
        if pin:
            hq, hk, hv, ho, hl = (t.pin_memory() for t in (hq, hk, hv, ho, hl))
        dq, dk, dv = torch.empty_like(q), torch.empty_like(k), torch.empty_like(v)
        pf.partition()
        pf.run_from_host(hq, hk, hv, ho, hl, dq, dk, dv)
        torch.cuda.synchronize()
        assert m.mocap_last_device_status() == 0
        res.append((ho.view(torch.int16).clone(), hl.clone()))
    assert torch.equal(res[0][0], res[1][0]) and torch.equal(res[0][1], res[1][1])
    assert not torch.isnan(res[1][1]).any()
