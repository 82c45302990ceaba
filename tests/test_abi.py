"""Host-side checks of the C ABI (no GPU needed): the library builds and
exports every entry point include/mocap.h declares, the host partition is
bit-exact against the oracle, and invalid arguments are rejected before any
CUDA call."""

import ctypes
import os
import random
import re

import pytest

from oracle import partition as P

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    names = set()
    inc = os.path.join(ROOT, "include")
    for f in os.listdir(inc):
        if f.endswith(".h"):
            text = open(os.path.join(inc, f)).read()
            text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
            names |= set(re.findall(r"\b(mocap_[a-z0-9_]+)\s*\(", text))
    return names


def test_header_declares_the_boundary():
    names = _declared()
    for n in ["mocap_lbcp_partition", "mocap_kv_append", "mocap_chunk_attn",
              "mocap_chunk_attn_workspace_size", "mocap_chunk_attn_varlen",
              "mocap_last_device_status", "mocap_status_string"]:
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    for name in _declared():
        assert hasattr(lib, name), name


def test_binding_has_every_declared_entry_point():
    # the Python layer carries the C names (argument marshalling only)
    import paper_2606_22968_gb300 as m
    for name in _declared():
        assert callable(getattr(m, name, None)), name


def test_build_entry_compiles_for_sm103a():
    import __graft_entry__  # noqa: F401
    from paper_2606_22968_gb300 import _build
    assert "arch=compute_103a,code=sm_103a" in " ".join(_build.ARCH)
    assert os.path.exists(_build.build())


def _c_partition(lib, s, m, g, mode):
    out = (ctypes.c_int64 * (m + 1))()
    st = lib.mocap_lbcp_partition(s, m, g, mode, out)
    return st, list(out)


def test_partition_bit_exact_vs_oracle_sweep(lib):
    for units in range(1, 2049, 7):
        for m in (1, 2, 3, 4, 5, 8, 16, 31, 32, 64):
            if m > units:
                continue
            for mode in (0, 1):
                s = units * 128
                st, b = _c_partition(lib, s, m, 128, mode)
                assert st == 0
                assert b == P.boundaries(s, m, 128, mode), (s, m, mode)


def test_partition_random_ragged_vs_oracle(lib):
    rnd = random.Random(1)
    for _ in range(3000):
        g = rnd.choice([1, 16, 64, 128, 256])
        s = rnd.randint(1, 1 << 24)
        m = rnd.randint(1, 200)
        if m * g > s:
            continue
        mode = rnd.randint(0, 1)
        st, b = _c_partition(lib, s, m, g, mode)
        assert st == 0 and b == P.boundaries(s, m, g, mode)


def test_partition_large_sequences(lib):
    for s, m in [(1 << 30, 1000), ((1 << 37) - 5, 4096), (131072, 32)]:
        st, b = _c_partition(lib, s, m, 128, 1)
        assert st == 0 and b == P.boundaries(s, m, 128, 1)


def test_partition_invalid(lib):
    out = (ctypes.c_int64 * 10)()
    assert lib.mocap_lbcp_partition(0, 1, 128, 1, out) == 1
    assert lib.mocap_lbcp_partition(1024, 0, 128, 1, out) == 1
    assert lib.mocap_lbcp_partition(1024, 9, 128, 1, out) == 1
    assert lib.mocap_lbcp_partition(1024, 2, 0, 1, out) == 1
    assert lib.mocap_lbcp_partition(1024, 2, 128, 7, out) == 1
    assert lib.mocap_lbcp_partition(1024, 2, 128, 1, None) == 1
    assert lib.mocap_lbcp_partition(1 << 40, 2, 1, 1, out) == 1  # U >= 2^30


def test_status_strings(lib):
    for code in range(5):
        assert lib.mocap_status_string(code).startswith(b"MOCAP_")


FAKE = 1 << 20  # a 16-byte-aligned non-null value; never dereferenced


def test_kv_append_rejects_bad_arguments_before_launch(lib):
    f = lib.mocap_kv_append
    assert f(None, FAKE, FAKE, FAKE, 10, 0, 1, 8, 128, None) == 1
    assert f(FAKE + 2, FAKE, FAKE, FAKE, 10, 0, 1, 8, 128, None) == 1      # misaligned
    assert f(FAKE, FAKE, FAKE, FAKE, 10, 8, 3, 8, 128, None) == 1           # past capacity
    assert f(FAKE, FAKE, FAKE, FAKE, 10, -1, 1, 8, 128, None) == 1
    assert f(FAKE, FAKE, FAKE, FAKE, 10, 0, -1, 8, 128, None) == 1
    assert f(FAKE, FAKE, FAKE, FAKE, 10, 0, 1, 1, 4, None) == 1             # 4 elems: not 16 B
    assert f(FAKE, FAKE, FAKE, FAKE, 10, 3, 0, 8, 128, None) == 0           # empty: no-op


def test_chunk_attn_rejects_bad_arguments_before_launch(lib):
    f = lib.mocap_chunk_attn
    ok = dict(prefix=0, length=128, hq=8, hkv=2, d=128, scale=0.088)

    def call(**kw):
        a = dict(ok, **kw)
        return f(kw.get("q", FAKE), FAKE, FAKE, a["prefix"], a["length"], a["hq"], a["hkv"], a["d"],
                 a["scale"], FAKE, kw.get("lse", FAKE), None, 0, None)

    assert call(q=None) == 1
    assert call(q=FAKE + 8) == 1
    assert call(lse=FAKE + 2) == 1
    assert call(hq=6, hkv=4) == 1
    assert call(hkv=0) == 1
    assert call(scale=0.0) == 1
    assert call(scale=float("nan")) == 1
    assert call(scale=-1.0) == 1
    assert call(prefix=-1) == 1
    assert call(length=-5) == 1
    assert call(prefix=(1 << 31) - 10, length=20) == 1
    assert call(d=96) == 3
    assert call(d=256) == 3
    assert call(length=0) == 0


def test_varlen_rejects_bad_items_before_launch(lib):
    from paper_2606_22968_gb300._lib import VarlenItem
    f = lib.mocap_chunk_attn_varlen

    def call(items, q_rows=1000, kv_rows=1000, n=None):
        arr = (VarlenItem * max(1, len(items)))(*[VarlenItem(*x) for x in items])
        return f(FAKE, FAKE, FAKE, arr, len(items) if n is None else n, q_rows, kv_rows, 8, 2, 128,
                 0.1, FAKE, FAKE, None, 0, None)

    assert call([(0, 0, 0, 10)], q_rows=5) == 1          # q rows past the buffer
    assert call([(0, 0, 995, 10)]) == 1                  # kv rows past the cache
    assert call([(-1, 0, 0, 10)]) == 1
    assert call([(0, 0, 0, 10)], n=65) == 1              # too many items
    assert call([(0, 0, 0, 10)], n=-1) == 1
    assert call([]) == 0
    assert call([(0, 0, 5, 0)]) == 0                     # empty item: no-op


def test_varlen_dev_argument_checks(lib):
    """mocap_chunk_attn_varlen_dev: everything checkable on the host fails
    before any CUDA call; n_items == 0 is a no-op."""
    f = lib.mocap_chunk_attn_varlen_dev
    need = lib.mocap_chunk_attn_varlen_dev_workspace_size(3, 1000, 64, 8, 128)

    def call(n=3, items=FAKE, q_rows=1000, max_rows=1000, ws=FAKE, ws_bytes=None, d=128):
        return f(FAKE, FAKE, FAKE, items, n, q_rows, 1000, max_rows, 64, 8, d, 0.1, FAKE, FAKE,
                 ws, need if ws_bytes is None else ws_bytes, None)

    assert call(n=0) == 0
    assert call(n=65537) == 1
    assert call(n=-1) == 1
    assert call(items=None) == 1
    assert call(items=FAKE + 4) == 1                     # items not 8-byte aligned
    assert call(ws=None) == 1
    assert call(ws=FAKE + 16) == 1                       # workspace not 128-byte aligned
    assert call(ws_bytes=need - 1) == 1
    assert call(q_rows=2 ** 31) == 1
    assert call(max_rows=-1) == 1
    assert call(max_rows=2 ** 31) == 1
    assert call(max_rows=2000) == 1                      # workspace sized for 1000 rows
    assert call(d=96) == 3


def test_varlen_dev_workspace_layout(lib):
    """Tensor maps (3 x 128 B per item), 24-byte item descriptors, one int32
    per CTA of the grid (ceil(max_rows / 128) + n) x Hkv x ceil(group / 2),
    the count; each section 256-byte aligned."""
    def expect(n, max_rows, hq, hkv):
        a = lambda x: (x + 255) // 256 * 256
        ctas = ((max_rows + 127) // 128 + n) * hkv * ((hq // hkv + 1) // 2)
        return a(a(a(n * 384) + n * 24) + ctas * 4) + 256
    for n, max_rows, hq, hkv, d in [(3, 1000, 64, 8, 128), (1, 0, 4, 4, 64),
                                    (300, 70784, 32, 8, 128), (65536, 1 << 20, 6, 2, 128)]:
        assert lib.mocap_chunk_attn_varlen_dev_workspace_size(n, max_rows, hq, hkv, d) == \
            expect(n, max_rows, hq, hkv)
    assert lib.mocap_chunk_attn_varlen_dev_workspace_size(0, 1000, 64, 8, 128) == 0
    assert lib.mocap_chunk_attn_varlen_dev_workspace_size(65537, 1000, 64, 8, 128) == 0
    assert lib.mocap_chunk_attn_varlen_dev_workspace_size(3, 1000, 64, 8, 96) == 0


def test_copy_from_host_argument_checks(lib):
    """mocap_copy_from_host rejects what it can see on the host before any
    CUDA call; an empty batch is a no-op."""
    from paper_2606_22968_gb300._lib import CopyItem
    f = lib.mocap_copy_from_host

    def call(items, n=None):
        arr = (CopyItem * max(1, len(items)))(*[CopyItem(*x) for x in items])
        return f(arr, len(items) if n is None else n, 0, None)

    assert call([]) == 0
    assert f(None, 0, 1, None) == 0
    assert f(None, 1, 0, None) == 1                       # null item array
    assert call([(FAKE, FAKE, 32)], n=9) == 1             # above MOCAP_COPY_MAX_ITEMS
    assert call([(FAKE, FAKE, 32)], n=-1) == 1
    assert call([(FAKE, FAKE, 17)]) == 1                  # not whole 16-byte vectors
    assert call([(FAKE, FAKE, -16)]) == 1
    assert call([(None, FAKE, 32)]) == 1
    assert call([(FAKE, FAKE + 8, 32)]) == 1              # misaligned source
    assert call([(FAKE, FAKE, 0)]) == 0                   # empty item skipped


def test_workspace_size_split_plan(lib):
    # many row blocks: no split; few long row blocks: a split and its layout
    assert lib.mocap_chunk_attn_workspace_size(0, 23168, 64, 8, 128) == 0
    ws = lib.mocap_chunk_attn_workspace_size(129024, 2048, 64, 8, 128)
    if ws:
        splits = None
        for s in (2, 3, 4):
            o = s * 2048 * 64 * 128 * 4
            if ws == (o + 255) // 256 * 256 + s * 64 * 2048 * 4:
                splits = s
        assert splits is not None, ws
    # tiny: one 8-unit chunk with a long prefix always splits
    assert lib.mocap_chunk_attn_workspace_size(100000, 256, 8, 2, 128) > 0
    # invalid shapes report 0
    assert lib.mocap_chunk_attn_workspace_size(0, 100, 6, 4, 128) == 0
    assert lib.mocap_chunk_attn_workspace_size(0, 100, 8, 2, 96) == 0
    assert lib.mocap_chunk_attn_workspace_size(-1, 100, 8, 2, 128) == 0


def test_dp_partition_bit_exact_vs_oracle(lib):
    rnd = random.Random(9)
    for _ in range(60):
        g = rnd.choice([64, 128, 256])
        units = rnd.randint(1, 160)
        m = rnd.randint(1, min(units, 12))
        s = units * g + rnd.choice([0, 0, 1, 63])
        n = rnd.choice([1, 2, 4, 16, 1000])
        model = rnd.randint(0, 1)
        gemm = rnd.choice([0, 5, 1000])
        out = (ctypes.c_int64 * (m + 1))()
        assert lib.mocap_lbcp_partition_dp(s, m, g, n, model, gemm, out) == 0
        assert list(out) == P.dp_boundaries(s, m, g, n, model, gemm), (s, m, g, n, model, gemm)


def test_dp_partition_invalid_and_limits(lib):
    out = (ctypes.c_int64 * 40)()
    assert lib.mocap_lbcp_partition_dp(1024, 2, 128, 0, 0, 0, out) == 1      # N < 1
    assert lib.mocap_lbcp_partition_dp(1024, 2, 128, 4, 5, 0, out) == 1      # model
    assert lib.mocap_lbcp_partition_dp(1024, 2, 128, 4, 0, -1, out) == 1     # weight
    assert lib.mocap_lbcp_partition_dp(1024, 9, 128, 4, 0, 0, out) == 1      # M g > S
    assert lib.mocap_lbcp_partition_dp(1 << 30, 32, 1, 4, 0, 0, out) == 3    # too large
    assert lib.mocap_lbcp_partition_dp(131072, 32, 128, 16, 0, 0, out) == 0


def test_bench_entry_points_exist():
    """bench.py's probe modes and arms are all defined (they are run on the GPU)."""
    import bench
    for name in ["profile_case", "profile_case_append", "profile_case_qkv", "profile_case_last_row",
                 "profile_case_host_copy", "measure_varlen_dev", "ours_arm",
                 "reference_arm", "measure_e2e", "measure_graph", "measure_projection",
                 "measure_last_row", "measure_partitions", "measure_chunk_streams",
                 "measure_fusion", "measure_append_graph"]:
        assert callable(getattr(bench, name)), name


def test_stage_balanced_bounds_weight_and_dp():
    """The GEMM weight follows from the per-chunk stage cost a * pairs + b * rows
    in the DP's doubled 128-row units, and the split is the DP's (bit-exact
    against the oracle's DP with that weight)."""
    from paper_2606_22968_gb300.pipeline import gemm_weight, stage_balanced_bounds
    from oracle import partition as P
    # a chunk of k units at s: pairs ~ 128^2 k (s + k/2), rows 128 k
    # a * 128^2 / 2 * [k (2s + k) + w k] = a * 128^2 k (s + k/2) + b * 128 k  =>  w = 2 b / (128 a)
    assert gemm_weight(1.0, 64.0) == 1
    assert gemm_weight(1.84e-11, 1.06e-7) == 90
    assert gemm_weight(1.0, 0.0) == 0
    for bad in ((0.0, 1.0), (1.0, -1.0)):
        with pytest.raises(ValueError):
            gemm_weight(*bad)
    for a, b in ((1.84e-11, 1.06e-7), (1e-11, 0.0)):
        got = stage_balanced_bounds(32768, 16, a, b)
        assert got == P.dp_boundaries(32768, 16, 128, 16, P.COST_CAUSAL, gemm_weight(a, b))


def test_dp_hand_worked_tie_case_bit_exact(lib):
    """Algorithm 1's tie rule (strict improvement, k ascending) on the case
    worked by hand in tests/golden/dp_tie_case.txt."""
    from tests.golden_utils import dp_tie_case
    case, _, _, bounds = dp_tie_case()
    out = (ctypes.c_int64 * (case["chunks"] + 1))()
    assert lib.mocap_lbcp_partition_dp(case["seq_len"], case["chunks"], case["granularity"],
                                       case["stages"], case["model"], case["gemm"], out) == 0
    assert list(out) == bounds


def test_dp_golden_rows_of_the_workload_shapes(lib):
    """The DP on the 32768/16 and 131072/32 shapes against rows the oracle wrote."""
    from tests.golden_utils import dp_boundary_rows
    rows = dp_boundary_rows()
    assert {r[0] for r in rows} == {32768, 131072}
    for s, m, g, n, model, gemm, b in rows:
        out = (ctypes.c_int64 * (m + 1))()
        assert lib.mocap_lbcp_partition_dp(s, m, g, n, model, gemm, out) == 0
        assert list(out) == b, (s, m, g, n, model, gemm)


def test_dp_rejects_arguments_whose_objective_could_overflow(lib):
    out = (ctypes.c_int64 * 40)()
    big_n = 2 ** 31 - 1
    # U = 1024: N (2 U^2 + w U) with w = 2^40 far beyond 2^62
    assert lib.mocap_lbcp_partition_dp(131072, 32, 128, big_n, 0, 2 ** 40, out) == 1
    assert lib.mocap_lbcp_partition_dp(131072, 32, 128, 2 ** 22, 0, 2 ** 40, out) == 1
    assert lib.mocap_lbcp_partition_dp(131072, 32, 128, 16, 0, 2 ** 40, out) == 0  # 1.8e16
    # U = 63245 (M U^2 < 4e9): 2 U^2 N with N = 2^31 - 1 is about 1.7e19 > 2^62
    assert lib.mocap_lbcp_partition_dp(63245, 1, 1, big_n, 0, 0, out) == 1
    # inside the bound: U = 1024 with the largest N, and a realistic weight
    assert lib.mocap_lbcp_partition_dp(131072, 32, 128, big_n, 0, 0, out) == 0
    assert lib.mocap_lbcp_partition_dp(131072, 32, 128, 16, 1, 90, out) == 0


def test_gemm_weight_entry_point(lib):
    w = ctypes.c_int64(-1)
    assert lib.mocap_lbcp_gemm_weight(1.0, 64.0, 128, ctypes.byref(w)) == 0 and w.value == 1
    assert lib.mocap_lbcp_gemm_weight(1.84e-11, 1.06e-7, 128, ctypes.byref(w)) == 0
    assert w.value == 90
    assert lib.mocap_lbcp_gemm_weight(1.0, 96.0, 128, ctypes.byref(w)) == 0 and w.value == 2
    for bad in ((0.0, 1.0, 128), (1.0, -1.0, 128), (float("nan"), 1.0, 128), (1.0, 1.0, 0),
                (1e-30, 1.0, 128)):
        assert lib.mocap_lbcp_gemm_weight(*bad, ctypes.byref(w)) == 1, bad
    assert lib.mocap_lbcp_gemm_weight(1.0, 1.0, 128, None) == 1


def test_fused_append_argument_checks(lib):
    """mocap_chunk_attn_append / _varlen_append refuse appends that overlap
    the rows the launch reads, each other, or the cache end (nothing is
    launched, so no GPU is needed)."""
    from paper_2606_22968_gb300._lib import AppendItem, VarlenItem
    f = lib.mocap_chunk_attn_append

    def call(apps, prefix=100, length=50, cap=1000, n=None):
        arr = (AppendItem * max(1, len(apps)))(*[AppendItem(*a) for a in apps])
        return f(FAKE, FAKE, FAKE, prefix, length, 8, 2, 128, 0.1, FAKE, FAKE, None, 0,
                 arr if apps else None, len(apps) if n is None else n, cap, None)

    assert call([(FAKE, FAKE, 149, 10)]) == 1            # overlaps the chunk's own rows
    assert call([(FAKE, FAKE, 0, 10)]) == 1              # overlaps the prefix
    assert call([(FAKE, FAKE, 995, 10)]) == 1            # past the cache
    assert call([(FAKE, FAKE, -1, 10)]) == 1
    assert call([(FAKE, FAKE, 200, -1)]) == 1
    assert call([(FAKE + 8, FAKE, 200, 10)]) == 1        # misaligned source
    assert call([(None, FAKE, 200, 10)]) == 1
    assert call([(FAKE, FAKE, 200, 10), (FAKE, FAKE, 205, 10)]) == 1  # appends overlap
    assert call([(FAKE, FAKE, 200, 10)] * 65) == 1       # too many
    assert call([], n=3) == 1                            # a count with a null array
    assert call([(FAKE, FAKE, 200, 10)], cap=120) == 1   # cache shorter than prefix + len
    g = lib.mocap_chunk_attn_varlen_append
    items = (VarlenItem * 2)(VarlenItem(0, 0, 0, 10), VarlenItem(10, 500, 20, 10))
    arr = (AppendItem * 1)(AppendItem(FAKE, FAKE, 515, 4))  # inside item 1's rows [500, 530)
    assert g(FAKE, FAKE, FAKE, items, 2, 100, 1000, 8, 2, 128, 0.1, FAKE, FAKE, None, 0, arr, 1,
             None) == 1


def test_dp_latency_bit_exact_vs_oracle(lib):
    """Algorithm 1 stage 1 with the kernel's latency model: C++ against the
    oracle on random small prompts (windows up to the whole prompt)."""
    rnd = random.Random(23)
    for _ in range(40):
        units = rnd.randint(1, 40)
        m = rnd.randint(1, min(units, 6))
        s = units * 128 + rnd.choice([0, 0, 1, 77])
        hkv = rnd.choice([1, 2, 8])
        hq = hkv * rnd.choice([1, 2, 3, 4, 8])
        d = rnd.choice([64, 128])
        sms = rnd.choice([1, 5, 16, 152])
        n = rnd.choice([1, 2, 16, 10 ** 6])
        window = rnd.choice([0, 1, 3, units])
        out = (ctypes.c_int64 * (m + 1))()
        assert lib.mocap_lbcp_partition_dp_latency(s, m, n, hq, hkv, d, sms, window, out) == 0
        assert list(out) == P.dp_latency_boundaries(s, m, n, hq, hkv, d, sms, window), \
            (s, m, n, hq, hkv, d, sms, window)


def test_dp_latency_golden_rows(lib):
    """The workload shapes' rows the oracle wrote (tests/golden/make_golden.py)."""
    from tests.golden_utils import dp_latency_rows
    rows = dp_latency_rows()
    assert {r[0][0] for r in rows} == {32768, 131072}
    for (s, m, n, hq, hkv, d, sms, window), b in rows:
        out = (ctypes.c_int64 * (m + 1))()
        assert lib.mocap_lbcp_partition_dp_latency(s, m, n, hq, hkv, d, sms, window, out) == 0
        assert list(out) == b


def test_dp_latency_argument_checks(lib):
    out = (ctypes.c_int64 * 40)()
    f = lib.mocap_lbcp_partition_dp_latency
    assert f(32768, 16, 16, 32, 8, 96, 152, 4, out) == 3       # head_dim
    assert f(32768, 16, 16, 32, 6, 128, 152, 4, out) == 1      # Hq % Hkv
    assert f(32768, 16, 0, 32, 8, 128, 152, 4, out) == 1       # stages
    assert f(32768, 16, 16, 32, 8, 128, 0, 4, out) == 1        # SMs
    assert f(32768, 16, 16, 32, 8, 128, 152, -1, out) == 1     # window
    assert f(1024, 9, 16, 32, 8, 128, 152, 4, out) == 1        # M * 128 > S
    assert f(1 << 31, 16, 16, 32, 8, 128, 152, 4, out) == 1    # S
    assert f(32768, 16, 16, 32, 8, 128, 152, 4, None) == 1
    assert f(1 << 30, 8, 16, 64, 8, 128, 152, 10 ** 6, out) == 3  # too much host work
    assert f(32768, 16, 16, 32, 8, 128, 152, 0, out) == 0
    assert list(out)[:17] == P.boundaries(32768, 16, 128)      # window 0: the closed form
