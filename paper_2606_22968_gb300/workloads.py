"""Seeded synthetic workloads for chunked prefill attention.

This module holds only workload definitions and seeded random inputs -- no
attention or partition arithmetic -- so that the tests, the bench and the
oracle can all draw the same bits from it.

The paper's own workload (prefill-only traces on Llama3-70B-class models,
Sec. 5.1) is not available; these shapes stand in for it:

1. ``tiny``     1024 tokens, 4 uniform chunks, 4 q-heads / 4 kv-heads, d=64
2. ``8b-8k``    8192 tokens, 8 uniform chunks, 32/8 heads, d=128 (Llama-3-8B)
3. ``8b-32k``   32768 tokens, 16 LBCP chunks, 32/8 heads, d=128
4. ``70b-128k`` 131072 tokens, 32 LBCP chunks, 64/8 heads, d=128 (Llama-3-70B)
5. ``varlen8``  8 requests, lengths log-uniform in [2048, 32768] (multiples of
                128), each split into LBCP chunks of about 2048 tokens, 32/8, d=128

Q, K and V are i.i.d. N(0, 1) rounded to bf16, drawn from a seeded
``torch.Generator`` on the target device (seed = 20261202 + config number).
"""

from __future__ import annotations

import dataclasses
import math
from typing import List, Optional

import numpy as np

SEED_BASE = 20261202
GRANULARITY = 128

MODE_UNIFORM = 0
MODE_LBCP = 1


@dataclasses.dataclass(frozen=True)
class Workload:
    index: int
    name: str
    seq_lens: tuple          # one entry per request
    num_chunks: tuple        # chunks per request
    mode: int                # MODE_UNIFORM or MODE_LBCP
    n_q_heads: int
    n_kv_heads: int
    head_dim: int

    @property
    def seed(self) -> int:
        return SEED_BASE + self.index

    @property
    def scale(self) -> float:
        return 1.0 / math.sqrt(self.head_dim)

    @property
    def total_tokens(self) -> int:
        return int(sum(self.seq_lens))

    def describe(self) -> dict:
        return {
            "workload": self.name,
            "requests": len(self.seq_lens),
            "seq_lens": list(self.seq_lens),
            "num_chunks": list(self.num_chunks),
            "partition": "lbcp" if self.mode == MODE_LBCP else "uniform",
            "granularity": GRANULARITY,
            "n_q_heads": self.n_q_heads,
            "n_kv_heads": self.n_kv_heads,
            "head_dim": self.head_dim,
            "seed": self.seed,
        }


def varlen_lengths(seed: int, n_requests: int = 8) -> List[int]:
    """Request lengths log-uniform in [2048, 32768], rounded to multiples of 128."""
    rng = np.random.Generator(np.random.PCG64(seed))
    u = rng.random(n_requests)
    out = []
    for x in u:
        raw = math.exp(math.log(2048.0) + float(x) * math.log(16.0))
        length = GRANULARITY * int(round(raw / GRANULARITY))
        out.append(min(max(length, 2048), 32768))
    return out


def varlen_chunks(length: int) -> int:
    """Chunk count for a target chunk length of about 2048 tokens."""
    return max(1, (length + 1024) // 2048)


def get(index: int) -> Workload:
    if index == 1:
        return Workload(1, "tiny-1k-4x256-h4-d64", (1024,), (4,), MODE_UNIFORM, 4, 4, 64)
    if index == 2:
        return Workload(2, "llama3-8b-attn-8k-uniform8", (8192,), (8,), MODE_UNIFORM, 32, 8, 128)
    if index == 3:
        return Workload(3, "llama3-8b-attn-32k-lbcp16", (32768,), (16,), MODE_LBCP, 32, 8, 128)
    if index == 4:
        return Workload(4, "llama3-70b-attn-128k-lbcp32", (131072,), (32,), MODE_LBCP, 64, 8, 128)
    if index == 5:
        lens = varlen_lengths(SEED_BASE + 5)
        return Workload(5, "varlen8-logu-2k-32k-lbcp2k", tuple(lens),
                        tuple(varlen_chunks(x) for x in lens), MODE_LBCP, 32, 8, 128)
    raise ValueError(f"unknown workload {index}")


def custom(name: str, seq_lens, num_chunks, mode, n_q_heads, n_kv_heads, head_dim,
           index: int = 100) -> Workload:
    return Workload(index, name, tuple(seq_lens), tuple(num_chunks), mode,
                    n_q_heads, n_kv_heads, head_dim)


def make_qkv(w: Workload, device, seed: Optional[int] = None):
    """Packed bf16 inputs for all requests: Q [T, Hq, d], K/V [T, Hkv, d],
    T = sum of the request lengths (request r owns rows cu[r]..cu[r+1])."""
    import torch

    gen = torch.Generator(device=device)
    gen.manual_seed(w.seed if seed is None else seed)
    total = w.total_tokens
    q = torch.randn((total, w.n_q_heads, w.head_dim), generator=gen, device=device,
                    dtype=torch.bfloat16)
    k = torch.randn((total, w.n_kv_heads, w.head_dim), generator=gen, device=device,
                    dtype=torch.bfloat16)
    v = torch.randn((total, w.n_kv_heads, w.head_dim), generator=gen, device=device,
                    dtype=torch.bfloat16)
    return q, k, v


def request_offsets(w: Workload) -> List[int]:
    cu = [0]
    for length in w.seq_lens:
        cu.append(cu[-1] + int(length))
    return cu
