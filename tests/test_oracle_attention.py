"""Pins for the attention oracle (Sec. 2.2, Sec. 3.2 / Eq. 1).

Each check is independent of the oracle's numpy code path: pure-Python brute
force with an explicit mask matrix and no max subtraction, closed forms,
invariants (chunked == unchunked, rows of softmax sum to one) and GQA
bookkeeping with planted head values.
"""

import math
import random

import numpy as np
import pytest
import torch

from oracle import attention as A
from oracle import partition as P


def _rand(shape, seed):
    return np.random.default_rng(seed).standard_normal(shape)


def _brute(q, k, v, scale, prefix=0):
    """Pure Python: explicit -inf mask matrix, exp without max shift, fsum."""
    n, hq, d = q.shape
    hkv = k.shape[1]
    grp = hq // hkv
    kv_len = k.shape[0]
    o = [[[0.0] * d for _ in range(hq)] for _ in range(n)]
    lse = [[0.0] * n for _ in range(hq)]
    for h in range(hq):
        g = h // grp
        for i in range(n):
            t = prefix + i
            mask = [0.0 if j <= t else -math.inf for j in range(kv_len)]
            s = [scale * math.fsum(float(q[i, h, c]) * float(k[j, g, c]) for c in range(d)) + mask[j]
                 for j in range(kv_len)]
            w = [math.exp(x) for x in s]
            tot = math.fsum(w)
            lse[h][i] = math.log(tot)
            for c in range(d):
                o[i][h][c] = math.fsum(w[j] * float(v[j, g, c]) for j in range(kv_len)) / tot
    return np.array(o), np.array(lse)


@pytest.mark.parametrize("hq,hkv,d,s", [(1, 1, 3, 7), (4, 2, 5, 9), (6, 3, 4, 11), (4, 1, 8, 6)])
def test_matches_brute_force_full(hq, hkv, d, s):
    q = _rand((s, hq, d), 1) * 0.7
    k = _rand((s, hkv, d), 2) * 0.7
    v = _rand((s, hkv, d), 3)
    scale = 1.0 / math.sqrt(d)
    o, lse = A.causal_attention(q, k, v, scale)
    ob, lb = _brute(q, k, v, scale)
    assert np.max(np.abs(o - ob)) < 1e-12
    assert np.max(np.abs(lse - lb)) < 1e-12


def test_matches_brute_force_chunk_with_prefix():
    hq, hkv, d = 4, 2, 6
    q = _rand((12, hq, d), 4)
    k = _rand((12, hkv, d), 5)
    v = _rand((12, hkv, d), 6)
    scale = 0.3
    prefix, length = 5, 4
    o, lse = A.chunk_attention(q[prefix:prefix + length], k[:prefix + length],
                               v[:prefix + length], prefix, scale)
    ob, lb = _brute(q[prefix:prefix + length], k[:prefix + length], v[:prefix + length], scale, prefix)
    assert np.max(np.abs(o - ob)) < 1e-12
    assert np.max(np.abs(lse - lb)) < 1e-12


def test_sampled_rows_equal_full_rows():
    q = _rand((300, 4, 8), 7)
    k = _rand((300, 2, 8), 8)
    v = _rand((300, 2, 8), 9)
    o, lse = A.causal_attention(q, k, v, 0.35)
    rows = np.array([0, 1, 17, 255, 256, 299])
    os_, ls_ = A.causal_attention(q, k, v, 0.35, rows=rows)
    assert np.array_equal(os_, o[rows]) or np.max(np.abs(os_ - o[rows])) < 1e-13
    assert np.max(np.abs(ls_ - lse[:, rows])) < 1e-13


def test_sampled_heads_equal_full_heads():
    # head sampling selects heads; against the brute-force definition too
    q = _rand((40, 8, 6), 21)
    k = _rand((40, 2, 6), 22)
    v = _rand((40, 2, 6), 23)
    o, lse = A.chunk_attention(q[10:], k, v, 10, 0.4)
    heads = [7, 0, 4]
    oh, lh = A.chunk_attention(q[10:], k, v, 10, 0.4, rows=[0, 5, 29], heads=heads)
    assert np.max(np.abs(oh - o[[0, 5, 29]][:, heads])) < 1e-13
    assert np.max(np.abs(lh - lse[heads][:, [0, 5, 29]])) < 1e-13
    ob, lb = _brute(q[10:], k, v, 0.4, 10)
    assert np.max(np.abs(oh - ob[[0, 5, 29]][:, heads])) < 1e-12
    with pytest.raises(ValueError):
        A.chunk_attention(q[10:], k, v, 10, 0.4, heads=[8])


def test_chunked_equals_unchunked_random_boundaries():
    rnd = random.Random(11)
    s, hq, hkv, d = 611, 4, 2, 16
    q = _rand((s, hq, d), 12)
    k = _rand((s, hkv, d), 13)
    v = _rand((s, hkv, d), 14)
    scale = 1 / math.sqrt(d)
    o_full, lse_full = A.causal_attention(q, k, v, scale)
    for _ in range(4):
        cuts = sorted(rnd.sample(range(1, s), rnd.randint(1, 9)))
        b = [0] + cuts + [s]
        o, lses, ck, cv = A.chunked_prefill(q, k, v, b, scale)
        assert np.max(np.abs(o - o_full)) < 1e-12
        assert np.max(np.abs(np.concatenate(lses, axis=1) - lse_full)) < 1e-12
        assert np.array_equal(ck, k) and np.array_equal(cv, v)
    # LBCP boundaries too
    b = P.boundaries(512, 3, 128)
    o, lses, _, _ = A.chunked_prefill(q[:512], k[:512], v[:512], b, scale)
    o2, l2 = A.causal_attention(q[:512], k[:512], v[:512], scale)
    assert np.max(np.abs(o - o2)) < 1e-12


def test_softmax_rows_sum_to_one():
    s, hq, hkv, d = 200, 2, 1, 8
    q = _rand((s, hq, d), 15) * 3
    k = _rand((s, hkv, d), 16) * 3
    v = _rand((s, hkv, d), 17)
    scale = 0.5
    _, lse = A.causal_attention(q, k, v, scale)
    for h in range(hq):
        for t in (0, 1, 50, 199):
            sc = scale * (k[:t + 1, 0, :] @ q[t, h, :])
            assert abs(np.exp(sc - lse[h, t]).sum() - 1.0) < 1e-12


def test_zero_queries_give_prefix_mean_and_log_count():
    s, hq, hkv, d = 97, 4, 2, 5
    q = np.zeros((s, hq, d))
    k = _rand((s, hkv, d), 18)
    v = _rand((s, hkv, d), 19)
    o, lse = A.causal_attention(q, k, v, 0.125)
    for h in range(hq):
        g = h // 2
        for t in range(s):
            assert np.max(np.abs(o[t, h] - v[:t + 1, g].mean(axis=0))) < 1e-12
            assert abs(lse[h, t] - math.log(t + 1)) < 1e-12


def test_row_zero_sees_only_key_zero():
    q = _rand((10, 2, 4), 20)
    k = _rand((10, 1, 4), 21)
    v = _rand((10, 1, 4), 22)
    scale = 0.7
    o, lse = A.causal_attention(q, k, v, scale)
    for h in range(2):
        assert np.max(np.abs(o[0, h] - v[0, 0])) < 1e-15
        assert abs(lse[h, 0] - scale * float(q[0, h] @ k[0, 0])) < 1e-12


def test_unit_values_and_equal_keys():
    s, d = 50, 6
    q = _rand((s, 3, d), 23)
    k = _rand((s, 3, d), 24)
    o, _ = A.causal_attention(q, k, np.ones((s, 3, d)), 0.4)
    assert np.max(np.abs(o - 1.0)) < 1e-12
    k_eq = np.repeat(_rand((1, 3, d), 25), s, axis=0)
    v = _rand((s, 3, d), 26)
    o, lse = A.causal_attention(q, k_eq, v, 0.4)
    for t in range(s):
        assert np.max(np.abs(o[t] - v[:t + 1].mean(axis=0))) < 1e-12


def test_gqa_head_to_group_mapping():
    s, hq, hkv, d = 20, 8, 2, 4
    q = _rand((s, hq, d), 27)
    k = _rand((s, hkv, d), 28)
    v = np.zeros((s, hkv, d))
    v[:, 0, :] = 1.0
    v[:, 1, :] = 2.0
    o, _ = A.causal_attention(q, k, v, 0.5)
    for h in range(hq):
        assert np.max(np.abs(o[:, h, :] - (1.0 if h < 4 else 2.0))) < 1e-12


def test_bf16_widening_matches_torch():
    x = torch.randn(1000, dtype=torch.float32).to(torch.bfloat16)
    x = torch.cat([x, torch.tensor([0.0, -0.0, 1e-40, -3.0e38, float("inf")], dtype=torch.bfloat16)])
    bits = x.view(torch.int16).numpy()
    assert np.array_equal(A.bf16_bits_to_f64(bits), x.to(torch.float64).numpy())


def test_kv_append_bytewise():
    cache = np.arange(40, dtype=np.uint16).reshape(10, 2, 2)
    chunk = np.full((3, 2, 2), 7, dtype=np.uint16)
    out = A.kv_append(cache, chunk, 4)
    assert np.array_equal(out[4:7], chunk)
    assert np.array_equal(out[:4], cache[:4]) and np.array_equal(out[7:], cache[7:])
    assert np.array_equal(cache, np.arange(40, dtype=np.uint16).reshape(10, 2, 2))


def _brute_subset(q_row, keys, vals, scale, subset):
    s = [scale * math.fsum(q_row[c] * keys[j][c] for c in range(len(q_row))) for j in subset]
    w = [math.exp(x) for x in s]
    tot = math.fsum(w)
    o = [math.fsum(w[a] * vals[j][c] for a, j in enumerate(subset)) / tot for c in range(len(q_row))]
    return o, math.log(tot)


def test_combine_partials_matches_union():
    s, d = 30, 4
    q = _rand((s, 1, d), 30)
    k = _rand((s, 1, d), 31)
    v = _rand((s, 1, d), 32)
    scale = 0.5
    o_full, lse_full = A.causal_attention(q, k, v, scale)
    rows = range(18, 30)
    o_parts = np.zeros((3, len(rows), 1, d))
    l_parts = np.zeros((3, 1, len(rows)))
    for a, t in enumerate(rows):
        sets = [list(range(0, 8)), list(range(8, 16)), list(range(16, t + 1))]
        for p_i, sub in enumerate(sets):
            o, l = _brute_subset(q[t, 0], k[:, 0], v[:, 0], scale, sub)
            o_parts[p_i, a, 0] = o
            l_parts[p_i, 0, a] = l
    o, lse = A.combine_partials(o_parts, l_parts)
    assert np.max(np.abs(o[:, 0] - o_full[18:, 0])) < 1e-12
    assert np.max(np.abs(lse[0] - lse_full[0, 18:])) < 1e-12
    # an empty part (LSE = -inf) contributes nothing
    o_parts2 = np.concatenate([o_parts, np.full((1, len(rows), 1, d), 123.0)])
    l_parts2 = np.concatenate([l_parts, np.full((1, 1, len(rows)), -np.inf)])
    o2, lse2 = A.combine_partials(o_parts2, l_parts2)
    assert np.max(np.abs(o2 - o)) < 1e-15 and np.max(np.abs(lse2 - lse)) < 1e-15
