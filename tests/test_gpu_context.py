"""GPU: the library called in a CUDA context the caller created with the
driver API (not the runtime's primary context).  Its per-context state (the
status word's address, kernel attributes, the no-allocation scratch) is set
up in that context, and the results equal, bit for bit, the same calls made
in the primary context.  Every buffer used in the created context is
allocated in it."""

import ctypes
import math

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def m():
    import paper_2606_22968_gb300 as mod
    mod._lib.load()
    return mod


class _CtxCreateParams(ctypes.Structure):
    _fields_ = [("exec_affinity", ctypes.c_void_p), ("n_exec_affinity", ctypes.c_int),
                ("cig", ctypes.c_void_p)]


def _driver():
    cu = ctypes.CDLL("libcuda.so.1")
    u64, sz, vp = ctypes.c_uint64, ctypes.c_size_t, ctypes.c_void_p
    for name, args in [("cuDeviceGet", [ctypes.POINTER(ctypes.c_int), ctypes.c_int]),
                       ("cuCtxCreate_v4", [ctypes.POINTER(vp), ctypes.POINTER(_CtxCreateParams),
                                           ctypes.c_uint, ctypes.c_int]),
                       ("cuCtxPopCurrent_v2", [ctypes.POINTER(vp)]),
                       ("cuCtxDestroy_v2", [vp]),
                       ("cuCtxSynchronize", []),
                       ("cuMemAlloc_v2", [ctypes.POINTER(u64), sz]),
                       ("cuMemFree_v2", [u64]),
                       ("cuMemcpyHtoD_v2", [u64, vp, sz]),
                       ("cuMemcpyDtoH_v2", [vp, u64, sz])]:
        fn = getattr(cu, name)
        fn.argtypes = args
        fn.restype = ctypes.c_int
    return cu


@pytest.mark.parametrize("prefix,length", [(1000, 300), (100000, 256)])
def test_calls_in_a_context_the_caller_created(m, prefix, length):
    hq, hkv, d = 8, 2, 128
    total = prefix + length
    scale = 1.0 / math.sqrt(d)
    dev = torch.device("cuda")
    gen = torch.Generator(device=dev).manual_seed(prefix + length)
    q = torch.randn((length, hq, d), generator=gen, device=dev, dtype=torch.bfloat16)
    k = torch.randn((total, hkv, d), generator=gen, device=dev, dtype=torch.bfloat16)
    v = torch.randn((total, hkv, d), generator=gen, device=dev, dtype=torch.bfloat16)
    need = m.mocap_chunk_attn_workspace_size(prefix, length, hq, hkv, d)
    ws = torch.empty((max(need, 16),), device=dev, dtype=torch.uint8)
    ref = []  # primary context: the workspace call, then the no-allocation call
    for noalloc in (False, True):
        out = torch.full((length, hq, d), float("nan"), device=dev, dtype=torch.bfloat16)
        lse = torch.full((hq, length), float("nan"), device=dev, dtype=torch.float32)
        if noalloc:
            m.mocap_chunk_attn_noalloc(q, k, v, prefix, out, lse, scale)
        else:
            m.mocap_chunk_attn(q, k, v, prefix, out, lse, scale, workspace=ws)
        torch.cuda.synchronize()
        assert m.mocap_last_device_status() == 0
        ref.append((out.view(torch.int16).cpu().numpy(), lse.cpu().numpy()))
    host = {name: t.contiguous().view(torch.int16).cpu().numpy() for name, t in
            (("q", q), ("k", k), ("v", v))}

    cu = _driver()
    lib = m._lib.load()
    dev_h = ctypes.c_int()
    assert cu.cuDeviceGet(ctypes.byref(dev_h), torch.cuda.current_device()) == 0
    ctx = ctypes.c_void_p()
    params = _CtxCreateParams()
    assert cu.cuCtxCreate_v4(ctypes.byref(ctx), ctypes.byref(params), 0, dev_h) == 0
    allocs = []

    def alloc(nbytes):
        p = ctypes.c_uint64()
        assert cu.cuMemAlloc_v2(ctypes.byref(p), nbytes) == 0
        allocs.append(p.value)
        return p.value

    got = []
    try:
        dptr = {}
        for name, arr in host.items():
            dptr[name] = alloc(arr.nbytes)
            assert cu.cuMemcpyHtoD_v2(dptr[name], arr.ctypes.data, arr.nbytes) == 0
        ws_d = alloc(max(need, 16))
        o_bytes, l_bytes = length * hq * d * 2, hq * length * 4
        for noalloc in (False, True):
            o_d, l_d = alloc(o_bytes), alloc(l_bytes)
            if noalloc:
                st = lib.mocap_chunk_attn_noalloc(dptr["q"], dptr["k"], dptr["v"], prefix, length,
                                                  hq, hkv, d, scale, o_d, l_d, None)
            else:
                st = lib.mocap_chunk_attn(dptr["q"], dptr["k"], dptr["v"], prefix, length, hq,
                                          hkv, d, scale, o_d, l_d, ws_d, max(need, 16), None)
            assert st == 0
            assert cu.cuCtxSynchronize() == 0
            assert lib.mocap_last_device_status(None) == 0
            o_h = np.empty((length, hq, d), dtype=np.int16)
            l_h = np.empty((hq, length), dtype=np.float32)
            assert cu.cuMemcpyDtoH_v2(o_h.ctypes.data, o_d, o_bytes) == 0
            assert cu.cuMemcpyDtoH_v2(l_h.ctypes.data, l_d, l_bytes) == 0
            got.append((o_h, l_h))
    finally:
        for p in allocs:
            cu.cuMemFree_v2(p)
        popped = ctypes.c_void_p()
        assert cu.cuCtxPopCurrent_v2(ctypes.byref(popped)) == 0
        assert popped.value == ctx.value
        assert cu.cuCtxDestroy_v2(ctx) == 0
    for (o_r, l_r), (o_g, l_g) in zip(ref, got):
        assert np.array_equal(o_r, o_g)
        assert np.array_equal(l_r.view(np.int32), l_g.view(np.int32))
    # back in the primary context, the library still works there
    out = torch.full((length, hq, d), float("nan"), device=dev, dtype=torch.bfloat16)
    lse = torch.full((hq, length), float("nan"), device=dev, dtype=torch.float32)
    m.mocap_chunk_attn(q, k, v, prefix, out, lse, scale, workspace=ws)
    torch.cuda.synchronize()
    assert m.mocap_last_device_status() == 0
    assert np.array_equal(out.view(torch.int16).cpu().numpy(), ref[0][0])
