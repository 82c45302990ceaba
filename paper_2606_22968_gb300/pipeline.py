"""Chunked prefill over a whole prompt on one GPU: partition, append, attend.

This walks the chunks of each request in order, exactly as one stage of the
chunked pipeline does (Sec. 2.2): chunk i's K/V are appended to the request's
KV cache and its queries attend to everything cached so far.  Boundaries come
from LBCP (Sec. 3.2 / Sec. 4.2) or the uniform split.  Every step is a call
into libmocap.so; torch only allocates memory and provides the stream.
"""

from __future__ import annotations

import os
from typing import List, Optional

import torch

from . import (MOCAP_COPY_MAX_ITEMS, MOCAP_COST_CAUSAL, MOCAP_PART_LBCP, MOCAP_PART_UNIFORM,
               mocap_chunk_attn, mocap_chunk_attn_append, mocap_chunk_attn_varlen,
               mocap_chunk_attn_varlen_append, mocap_chunk_attn_workspace_size,
               mocap_copy_from_host, mocap_copy_to_host, mocap_kv_append,
               mocap_kv_append_overlap,
               mocap_lbcp_gemm_weight, mocap_lbcp_partition, mocap_lbcp_partition_dp,
               mocap_lbcp_partition_dp_latency, mocap_qkv_rope_append)
from .workloads import GRANULARITY, Workload, request_offsets


def gemm_weight(attn_s_per_pair: float, gemm_s_per_row: float, granularity: int = 128) -> int:
    """The DP's GEMM weight for a chunk stage costing ``a * pairs + b * rows``
    (Eq. 1 with its GEMM term; a = attention seconds per causal (query, key)
    pair, b = projection seconds per row), computed by the library
    (``mocap_lbcp_gemm_weight``)."""
    return mocap_lbcp_gemm_weight(attn_s_per_pair, gemm_s_per_row, granularity)


def stage_balanced_bounds(seq_len: int, num_chunks: int, attn_s_per_pair: float,
                          gemm_s_per_row: float, num_stages: int = 16,
                          granularity: int = 128) -> List[int]:
    """Boundaries from stage 1 of Algorithm 1 (Sec. 4.2) for chunks whose
    stage is a projection plus attention, given their measured rates."""
    return mocap_lbcp_partition_dp(seq_len, num_chunks, granularity, num_stages,
                                   MOCAP_COST_CAUSAL,
                                   gemm_weight(attn_s_per_pair, gemm_s_per_row, granularity))


APPEND_MODES = ("serial", "fused", "overlap")
HOST_COPY_MODES = ("auto", "kernel", "copy_engine")
# Bandwidth the one-warp-per-SM upload kernel reached beside the attention
# launches (varlen workload on GB300), and the attention rate assumed to
# turn a prompt's FLOP into its compute time, for host_copies="auto".
BESIDE_UPLOAD_BYTES_PER_S = 80e9
ATTENTION_FLOP_PER_S = 1.5e15


def latency_balanced_bounds(seq_len: int, num_chunks: int, n_q_heads: int, n_kv_heads: int,
                            head_dim: int, num_sms: int, num_stages: int = 16,
                            window: int = 8) -> List[int]:
    """Boundaries from stage 1 of Algorithm 1 (Sec. 4.2) with EvaluateChunk =
    the attention kernel's compute-latency model on `num_sms` SMs, each
    boundary within `window` 128-row units of the closed-form split
    (mocap_lbcp_partition_dp_latency)."""
    return mocap_lbcp_partition_dp_latency(seq_len, num_chunks, n_q_heads, n_kv_heads, head_dim,
                                           num_sms, num_stages, window)


class ChunkedPrefill:
    """Buffers and launch sequence for one workload on one device.

    Single-request workloads launch ``mocap_chunk_attn`` once per chunk, with
    chunk i's LSE in its own ``[Hq, c_i]`` block of ``lse`` (offset Hq*b_i).
    Multi-request workloads launch ``mocap_chunk_attn_varlen`` once per chunk
    index k over every request that has a chunk k; ``lse`` is then one
    ``[Hq, T]`` array over the packed rows.
    """

    def __init__(self, w: Workload, device, mode: Optional[int] = None, split_kv: bool = True,
                 bounds: Optional[List[List[int]]] = None, append_mode: str = "overlap",
                 chunk_streams: Optional[int] = None, host_copies: str = "auto"):
        """``bounds`` (one boundary list per request) replaces the workload's
        partition rule, e.g. with the Algorithm 1 stage-1 DP's split.

        ``append_mode`` says how chunk K/V reach the cache (step 0's chunks
        are always appended by a launch of their own before its attention):
          "serial"   each step appends its chunks (mocap_kv_append), then
                     attends, all on one stream;
          "fused"    each step's attention launch also appends the next
                     step's chunks (mocap_chunk_attn_append);
          "overlap"  a second stream appends steps 1.. in order
                     (mocap_kv_append_overlap, a kernel that fits beside the
                     attention CTAs), and step i's attention waits for its
                     own chunks' event only.

        ``chunk_streams`` = 2 (the default with overlapped appends, else 1)
        issues the steps' attention launches alternately
        on the caller's stream and a second compute stream (``run`` only):
        step i + 1 reads no output of step i, only K/V rows already appended,
        so its CTAs may take SMs that step i's last wave leaves idle.  Each
        compute stream has its own split-KV workspace.  Steps are still
        issued in order; per-step events then time overlapping launches.
        Needs append_mode "overlap": every step then waits for an event that
        says its rows (and all earlier rows) are in the cache.

        ``host_copies`` says how ``run_from_host`` / ``run_prompts_from_host``
        move Q/K/V up from pinned host memory and O/LSE back.  The transfers
        nothing hides, a prompt's first upload and its last results, go by
        all SMs (mocap_copy_from_host / mocap_copy_to_host) unless
        "copy_engine"; results returned while attention runs go by the copy
        engines (no SM slots taken).  Uploads while attention runs: "kernel"
        by one warp per SM beside the attention CTAs (about 80 GB/s there);
        "copy_engine" by cudaMemcpyAsync, as every copy then; "auto" by the
        kernel when the prompt needs less than half that bandwidth to keep
        its uploads ahead of its attention (compute-bound prompts), else by
        the copy engines."""
        if append_mode not in APPEND_MODES:
            raise ValueError(f"append_mode must be one of {APPEND_MODES}")
        if host_copies not in HOST_COPY_MODES:
            raise ValueError(f"host_copies must be one of {HOST_COPY_MODES}")
        self.host_copies = host_copies
        if chunk_streams is None:
            chunk_streams = 2 if append_mode == "overlap" else 1
        if chunk_streams not in (1, 2):
            raise ValueError("chunk_streams must be 1 or 2")
        if chunk_streams == 2 and append_mode != "overlap":
            raise ValueError("chunk_streams = 2 needs append_mode 'overlap'")
        self.w = w
        self.append_mode = append_mode
        self.chunk_streams = chunk_streams
        self.device = torch.device(device)
        self.mode = w.mode if mode is None else mode
        self.fixed_bounds = None if bounds is None else [list(b) for b in bounds]
        self.bounds: List[List[int]] = []
        self.partition()
        self.cu = request_offsets(w)
        total = w.total_tokens
        kw = dict(device=self.device, dtype=torch.bfloat16)
        self.k_cache = torch.empty((total, w.n_kv_heads, w.head_dim), **kw)
        self.v_cache = torch.empty((total, w.n_kv_heads, w.head_dim), **kw)
        self.out = torch.empty((total, w.n_q_heads, w.head_dim), **kw)
        self.lse = torch.empty((w.n_q_heads * total,), device=self.device, dtype=torch.float32)
        self.single = len(w.seq_lens) == 1
        # Split-KV scratch: the largest any launch uses.  A single request
        # splits any chunk that gains from it; several requests split only
        # the steps left with one request's chunk (the tail of the longest
        # request), since a launch of several items never splits.
        self.workspace = None
        if split_kv:
            one = [(0, i) for i in range(len(self.bounds[0]) - 1)] if self.single else \
                [step[0] for step in self.steps() if len(step) == 1]
            need = 0
            for r, c in one:
                b = self.bounds[r]
                need = max(need, mocap_chunk_attn_workspace_size(b[c], b[c + 1] - b[c],
                                                                 w.n_q_heads, w.n_kv_heads,
                                                                 w.head_dim))
            if need > 0:
                self.workspace = torch.empty((need,), device=self.device, dtype=torch.uint8)
        # the second compute stream's own split-KV scratch
        self.workspace2 = None
        if chunk_streams == 2 and self.workspace is not None:
            self.workspace2 = torch.empty_like(self.workspace)

    def partition(self):
        """Chunk boundaries of every request (host call into the library)."""
        if self.fixed_bounds is not None:
            self.bounds = [list(b) for b in self.fixed_bounds]
            return self.bounds
        part_mode = MOCAP_PART_LBCP if self.mode == 1 else MOCAP_PART_UNIFORM
        self.bounds = [mocap_lbcp_partition(s, m, GRANULARITY, part_mode)
                       for s, m in zip(self.w.seq_lens, self.w.num_chunks)]
        return self.bounds

    # -- launch plan -----------------------------------------------------------
    def steps(self):
        """List of launch steps; each is a list of (request, chunk index)."""
        n_steps = max(len(b) - 1 for b in self.bounds)
        return [[(r, k) for r in range(len(self.bounds)) if k < len(self.bounds[r]) - 1]
                for k in range(n_steps)]

    def chunk_lse(self, i: int) -> torch.Tensor:
        """Single request: chunk i's LSE block [Hq, c_i]."""
        b = self.bounds[0]
        hq = self.w.n_q_heads
        return self.lse[hq * b[i]:hq * b[i + 1]].view(hq, b[i + 1] - b[i])

    def lse_packed(self) -> torch.Tensor:
        """Multi-request: the [Hq, T] LSE array."""
        return self.lse.view(self.w.n_q_heads, self.w.total_tokens)

    # -- execution ----------------------------------------------------------------
    def run_step(self, q, k, v, i, stream=None, events=None, ready=None, attention_only=False,
                 workspace=None):
        """Step ``i`` of ``steps()`` (one chunk index of every request that has
        it), as ``append_mode`` says.  ``ready`` is the event after which step
        i's chunks are in the cache (overlap mode, from ``launch_appends``);
        without one, step i appends its own chunks first.  ``attention_only``
        skips every append (the caches already hold the rows).  ``events`` is
        an optional triple of CUDA events recorded before the step's own
        appends, before the attention launch, and after it.  With MOCAP_NVTX=1
        in the environment each step is an NVTX range ("mocap chunk <index>")
        for timeline profilers.  ``workspace`` replaces the split-KV scratch
        (default: the prefill's own)."""
        if os.environ.get("MOCAP_NVTX", "0") != "0":
            with torch.cuda.nvtx.range(f"mocap chunk {i}"):
                return self._run_step(q, k, v, i, stream, events, ready, attention_only,
                                      workspace)
        return self._run_step(q, k, v, i, stream, events, ready, attention_only, workspace)

    def _append_rows(self, k, v, r, c):
        """(K rows, V rows, destination cache row) of chunk c of request r."""
        b0, b1 = self.bounds[r][c], self.bounds[r][c + 1]
        base = self.cu[r]
        return k[base + b0:base + b1], v[base + b0:base + b1], base + b0

    def launch_appends(self, k, v, stream=None, landed=None):
        """Overlap mode: on a second stream, the appends of steps 1.. in step
        order (each after ``landed[i]`` if given, e.g. its host upload), each
        step followed by an event.  The second stream starts after the work
        queued so far on ``stream``.  Returns the per-step events (None for
        step 0, which run_step appends itself) and the second stream."""
        main = torch.cuda.current_stream(self.device) if stream is None else stream
        side = torch.cuda.Stream(self.device)
        side.wait_stream(main)
        ready = [None]
        with torch.cuda.stream(side):
            for i, step in enumerate(self.steps()):
                if i == 0:
                    continue
                if landed is not None:
                    side.wait_event(landed[i])
                for r, c in step:
                    kr, vr, dst = self._append_rows(k, v, r, c)
                    mocap_kv_append_overlap(kr, vr, self.k_cache, self.v_cache, dst, stream=side)
                ev = torch.cuda.Event()
                ev.record(side)
                ready.append(ev)
        return ready, side

    def _run_step(self, q, k, v, i, stream=None, events=None, ready=None, attention_only=False,
                  workspace=None):
        w = self.w
        workspace = self.workspace if workspace is None else workspace
        mode = self.append_mode
        steps = self.steps()
        step = steps[i]
        if events is not None:
            events[0].record(stream)
        if not attention_only:
            if ready is not None:
                (torch.cuda.current_stream(self.device) if stream is None else stream).wait_event(
                    ready)
            elif mode != "fused" or i == 0:
                for r, c in step:
                    kr, vr, dst = self._append_rows(k, v, r, c)
                    mocap_kv_append(kr, vr, self.k_cache, self.v_cache, dst, stream=stream)
        nxt = []
        if mode == "fused" and not attention_only and i + 1 < len(steps):
            nxt = [self._append_rows(k, v, r, c) for r, c in steps[i + 1]]
        if events is not None:
            events[1].record(stream)
        if self.single:
            (_, c), = step
            b0, b1 = self.bounds[0][c], self.bounds[0][c + 1]
            if nxt:
                mocap_chunk_attn_append(q[b0:b1], self.k_cache, self.v_cache, b0,
                                        self.out[b0:b1], self.chunk_lse(c), w.scale, nxt,
                                        workspace=workspace, stream=stream)
            else:
                mocap_chunk_attn(q[b0:b1], self.k_cache, self.v_cache, b0, self.out[b0:b1],
                                 self.chunk_lse(c), w.scale, workspace=workspace,
                                 stream=stream)
        else:
            items = []
            for r, c in step:
                b0, b1 = self.bounds[r][c], self.bounds[r][c + 1]
                items.append((self.cu[r] + b0, self.cu[r], b0, b1 - b0))
            if nxt:
                mocap_chunk_attn_varlen_append(q, self.k_cache, self.v_cache, items, self.out,
                                               self.lse_packed(), w.scale, nxt,
                                               workspace=workspace, stream=stream)
            else:
                mocap_chunk_attn_varlen(q, self.k_cache, self.v_cache, items, self.out,
                                        self.lse_packed(), w.scale, workspace=workspace,
                                        stream=stream)
        if events is not None:
            events[2].record(stream)

    def run(self, q, k, v, stream=None, chunk_events=None, landed=None, after_step=None):
        """The whole prompt: every step in order.  ``chunk_events`` optionally
        holds one event triple per step (see run_step); ``landed`` optionally
        one event per step after which its inputs are in q, k, v;
        ``after_step(i, st)`` is called once step i has been enqueued on
        stream ``st`` (e.g. to queue work that waits for it)."""
        main = torch.cuda.current_stream(self.device) if stream is None else stream
        n = len(self.steps())
        ready, side = [None] * n, None
        if self.append_mode == "overlap" and n > 1:
            ready, side = self.launch_appends(k, v, main, landed)
        second = None
        if self.chunk_streams == 2 and n > 1:
            # step 0's chunks go to the cache first, on the caller's stream;
            # the second stream starts after them (and after earlier work)
            if landed is not None:
                main.wait_event(landed[0])
            for r, c in self.steps()[0]:
                kr, vr, dst = self._append_rows(k, v, r, c)
                mocap_kv_append(kr, vr, self.k_cache, self.v_cache, dst, stream=main)
            ready[0] = torch.cuda.Event()
            ready[0].record(main)
            second = torch.cuda.Stream(self.device)
            second.wait_stream(main)
        for i in range(n):
            st, ws = (second, self.workspace2) if (second is not None and i % 2) else (main, None)
            if landed is not None:
                st.wait_event(landed[i])
                if self.append_mode == "fused" and i + 1 < n:
                    st.wait_event(landed[i + 1])  # this launch appends step i + 1's K/V
            with torch.cuda.stream(st):
                self.run_step(q, k, v, i, st, None if chunk_events is None else chunk_events[i],
                              ready[i], workspace=ws)
            if after_step is not None:
                after_step(i, st)
        if second is not None:
            main.wait_stream(second)
        if side is not None:
            main.wait_stream(side)

    def run_stage(self, x, w_qkv, q_buf, stream=None, rope_theta: float = 500000.0,
                  chunk_events=None, overlap: bool = False):
        """One attention layer's chunk stage for a single request (Eq. 1 with
        its GEMM term): per chunk, in order, the fused QKV projection of the
        chunk's hidden states ``x`` [S, hidden] with ``w_qkv`` [(Hq + 2 Hkv) d,
        hidden] (RoPE at the chunk's global positions; Q to ``q_buf`` [S, Hq,
        d], K and V straight into the caches), then the chunk's attention over
        the cache.  ``chunk_events`` optionally holds one (start, end) event
        pair per chunk.

        ``overlap=True``: the projections run in order on a stream of their
        own and each chunk's attention, alternating between two compute
        streams (their own split-KV scratch), waits only for its chunk's
        projection: chunk c + 1's projection writes rows chunk c's attention
        never reads, so the two overlap (no ``chunk_events``)."""
        if not self.single:
            raise ValueError("run_stage takes a single-request workload")
        w, b = self.w, self.bounds[0]
        if overlap:
            if chunk_events is not None:
                raise ValueError("chunk_events need overlap=False")
            return self._run_stage_overlapped(x, w_qkv, q_buf, stream, rope_theta)
        for c in range(len(b) - 1):
            if chunk_events is not None:
                chunk_events[c][0].record(stream)
            mocap_qkv_rope_append(x[b[c]:b[c + 1]], w_qkv, q_buf[b[c]:b[c + 1]], self.k_cache,
                                  self.v_cache, b[c], rope_theta=rope_theta, stream=stream)
            mocap_chunk_attn(q_buf[b[c]:b[c + 1]], self.k_cache, self.v_cache, b[c],
                             self.out[b[c]:b[c + 1]], self.chunk_lse(c), w.scale,
                             workspace=self.workspace, stream=stream)
            if chunk_events is not None:
                chunk_events[c][1].record(stream)

    def _run_stage_overlapped(self, x, w_qkv, q_buf, stream, rope_theta):
        w, b = self.w, self.bounds[0]
        main = torch.cuda.current_stream(self.device) if stream is None else stream
        proj = torch.cuda.Stream(self.device)
        second = torch.cuda.Stream(self.device)
        proj.wait_stream(main)
        second.wait_stream(main)
        if self.workspace is not None and self.workspace2 is None:
            self.workspace2 = torch.empty_like(self.workspace)
        for c in range(len(b) - 1):
            with torch.cuda.stream(proj):
                mocap_qkv_rope_append(x[b[c]:b[c + 1]], w_qkv, q_buf[b[c]:b[c + 1]],
                                      self.k_cache, self.v_cache, b[c], rope_theta=rope_theta,
                                      stream=proj)
            projected = torch.cuda.Event()
            projected.record(proj)
            st, ws = (second, self.workspace2) if c % 2 else (main, self.workspace)
            st.wait_event(projected)
            with torch.cuda.stream(st):
                mocap_chunk_attn(q_buf[b[c]:b[c + 1]], self.k_cache, self.v_cache, b[c],
                                 self.out[b[c]:b[c + 1]], self.chunk_lse(c), w.scale,
                                 workspace=ws, stream=st)
        main.wait_stream(second)
        main.wait_stream(proj)

    # -- from host memory ------------------------------------------------------------
    def _rows(self, r, c):
        b0, b1 = self.bounds[r][c], self.bounds[r][c + 1]
        return slice(self.cu[r] + b0, self.cu[r] + b1), b0, b1

    def _compute_and_return(self, q, k, v, compute, d2h, landed, host_out, host_lse,
                            last_alone=True):
        """Every step on ``compute`` (and the second compute stream) once its
        inputs have landed (events ``landed``), each step's O (and a single
        request's LSE block) copied back on ``d2h`` as soon as that step is
        done.  ``last_alone``: nothing else computes while the last step's
        results go back (no next prompt queued behind this one)."""
        steps = self.steps()
        hq = self.w.n_q_heads

        def copy_back(i, st):
            done = torch.cuda.Event()
            done.record(st)
            d2h.wait_event(done)
            pairs = []
            for r, c in steps[i]:
                rows, b0, b1 = self._rows(r, c)
                pairs.append((host_out[rows], self.out[rows]))
                if self.single:
                    pairs.append((host_lse[hq * b0:hq * b1], self.lse[hq * b0:hq * b1]))
            self._copy_back(pairs, d2h, beside=i + 1 < len(steps) or not last_alone)

        self.run(q, k, v, compute, landed=landed, after_step=copy_back)

    def _beside_uploads_by_kernel(self):
        """host_copies "auto": the upload bandwidth this prompt needs to stay
        ahead of its attention, against half the beside kernel's."""
        if self.host_copies != "auto":
            return self.host_copies == "kernel"
        w = self.w
        flop = sum(4 * w.n_q_heads * w.head_dim * (c * p + c * (c + 1) // 2)
                   for b in self.bounds for p, c in
                   ((b[i], b[i + 1] - b[i]) for i in range(len(b) - 1)))
        up = w.total_tokens * (w.n_q_heads + 2 * w.n_kv_heads) * w.head_dim * 2
        return up / max(flop / ATTENTION_FLOP_PER_S, 1e-9) < 0.5 * BESIDE_UPLOAD_BYTES_PER_S

    def _upload_step(self, step, dev_qkv, host_qkv, stream, beside):
        """Copy one step's Q/K/V rows from pinned host memory on ``stream``."""
        pairs = []
        for r, c in step:
            rows, _, _ = self._rows(r, c)
            pairs += [(d[rows], h[rows]) for d, h in zip(dev_qkv, host_qkv)]
        if beside and self.host_copies != "copy_engine" and not self._beside_uploads_by_kernel():
            with torch.cuda.stream(stream):
                for d, src in pairs:
                    d.copy_(src, non_blocking=True)
            return
        self._host_copy(pairs, stream, beside, mocap_copy_from_host)

    def _copy_back(self, pairs, stream, beside):
        """Copy (pinned host, device) pairs back on ``stream``: by the SMs when
        nothing else runs (``beside`` false: a prompt's last results, which
        nothing hides), else by the copy engines, which then work behind the
        attention launches without taking SM slots from them."""
        if beside and self.host_copies != "copy_engine":
            with torch.cuda.stream(stream):
                for d, src in pairs:
                    d.copy_(src, non_blocking=True)
            return
        self._host_copy(pairs, stream, beside, mocap_copy_to_host)

    def _host_copy(self, pairs, stream, beside, fn):
        # the SM copies read or write the host pages through their device
        # mapping, which only page-locked memory has: other host tensors go
        # by cudaMemcpyAsync (torch stages pageable memory itself)
        pinned = all(t.is_pinned() for pair in pairs for t in pair if not t.is_cuda)
        if self.host_copies == "copy_engine" or not pinned:
            with torch.cuda.stream(stream):
                for d, src in pairs:
                    d.copy_(src, non_blocking=True)
            return
        for a in range(0, len(pairs), MOCAP_COPY_MAX_ITEMS):
            fn(pairs[a:a + MOCAP_COPY_MAX_ITEMS], beside_kernels=beside, stream=stream)

    def run_from_host(self, host_q, host_k, host_v, host_out, host_lse, q, k, v):
        """The whole prompt from (pinned) host memory, overlapping transfers
        with compute.

        Every chunk's Q/K/V rows are copied into the device buffers ``q, k, v``
        on a copy stream, in chunk order; the compute stream starts chunk i as
        soon as its rows (and, with fused appends, chunk i + 1's, which its
        launch appends) have landed, and a third stream copies chunk i's O
        and LSE back to ``host_out`` / ``host_lse`` (shaped like ``self.out``
        and ``self.lse``) as soon as its attention is done.  With several
        requests a chunk's LSE columns are strided in the ``[Hq, T]`` array, so
        the whole LSE (4 Hq T bytes) goes back in one contiguous copy after the
        last step instead.  The caller's current stream waits for everything
        before this returns; the host tensors must stay alive and unchanged
        until that work has finished (with ``host_copies="kernel"`` the GPU
        reads and writes them in place)."""
        compute = torch.cuda.current_stream(self.device)
        h2d = torch.cuda.Stream(self.device)
        d2h = torch.cuda.Stream(self.device)
        steps = self.steps()
        hq = self.w.n_q_heads
        landed = []
        h2d.wait_stream(compute)  # device buffers are free of earlier work
        with torch.cuda.stream(h2d):
            for i, step in enumerate(steps):
                # step 0 goes up with nothing else running; later steps
                # beside the attention launches
                self._upload_step(step, (q, k, v), (host_q, host_k, host_v), h2d, beside=i > 0)
                ev = torch.cuda.Event()
                ev.record(h2d)
                landed.append(ev)
        d2h.wait_stream(compute)
        self._compute_and_return(q, k, v, compute, d2h, landed, host_out, host_lse)
        if not self.single:
            d2h.wait_stream(compute)
            self._copy_back([(host_lse, self.lse)], d2h, beside=False)
        compute.wait_stream(d2h)
        compute.wait_stream(h2d)

    def run_prompts_from_host(self, prompts, buffers):
        """Several prompts of this workload's shape in a row, each from (pinned)
        host memory, with the next prompt's inputs going up while the current
        one computes.

        ``prompts``: a sequence of (host_q, host_k, host_v, host_out,
        host_lse), shaped like ``run_from_host``'s arguments.  ``buffers``: two
        (q, k, v) device buffer sets used alternately; prompt p's inputs go
        into set p % 2 once prompt p - 2 has finished computing from it.
        Within a prompt, chunk i starts as soon as its rows have landed and
        its O and LSE go back as soon as its attention is done, as in
        ``run_from_host``; prompt p + 1's chunks start after prompt p's
        results have left the shared output buffers.  The caller's current
        stream waits for everything before this returns."""
        if len(buffers) != 2:
            raise ValueError("two device buffer sets expected")
        compute = torch.cuda.current_stream(self.device)
        h2d = torch.cuda.Stream(self.device)
        d2h = torch.cuda.Stream(self.device)
        steps = self.steps()
        hq = self.w.n_q_heads
        h2d.wait_stream(compute)
        d2h.wait_stream(compute)
        computed = [None, None]   # per buffer set: the end of the last prompt computed from it
        outputs_gone = None       # the end of the last prompt's D2H copies
        landed = []               # per prompt: per step, the event its inputs landed on

        def upload(p):
            q, k, v = buffers[p % 2]
            host_q, host_k, host_v = prompts[p][:3]
            evs = []
            with torch.cuda.stream(h2d):
                if computed[p % 2] is not None:
                    h2d.wait_event(computed[p % 2])
                for i, step in enumerate(steps):
                    # only the first prompt's first step goes up alone
                    self._upload_step(step, (q, k, v), (host_q, host_k, host_v), h2d,
                                      beside=p > 0 or i > 0)
                    ev = torch.cuda.Event()
                    ev.record(h2d)
                    evs.append(ev)
            landed.append(evs)

        if prompts:
            upload(0)
        for p in range(len(prompts)):
            if p + 1 < len(prompts):
                upload(p + 1)  # overlaps this prompt's compute (other buffer set)
            q, k, v = buffers[p % 2]
            host_out, host_lse = prompts[p][3], prompts[p][4]
            if outputs_gone is not None:
                compute.wait_event(outputs_gone)
            self._compute_and_return(q, k, v, compute, d2h, landed[p], host_out, host_lse,
                                     last_alone=p + 1 == len(prompts))
            end = torch.cuda.Event()
            end.record(compute)
            computed[p % 2] = end
            if not self.single:
                d2h.wait_event(end)
                self._copy_back([(host_lse, self.lse)], d2h, beside=True)
            gone = torch.cuda.Event()
            gone.record(d2h)
            outputs_gone = gone
        compute.wait_stream(d2h)
        compute.wait_stream(h2d)

    # -- CUDA graph ------------------------------------------------------------------
    def capture_steps(self, q, k, v, stream=None):
        """One CUDA graph per step holding that step's attention launch (and
        split-KV combine) only; the caches must already hold the prompt's
        K/V (e.g. from ``run``).  Replaying them in order with events between
        the replays times each chunk's attention without host gaps inside
        it.  Same preconditions as ``capture``."""
        graphs = []
        side = torch.cuda.Stream(self.device) if stream is None else stream
        side.wait_stream(torch.cuda.current_stream(self.device))
        with torch.cuda.stream(side):
            for i in range(len(self.steps())):
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g, stream=side):
                    self.run_step(q, k, v, i, side, attention_only=True)
                graphs.append(g)
        torch.cuda.current_stream(self.device).wait_stream(side)
        return graphs

    def capture(self, q, k, v, stream=None):
        """Record the whole prompt's launch sequence (every append, attention
        launch and split-KV combine) into one CUDA graph.  Replaying it runs
        the same kernels on the same buffers without per-launch host work or
        gaps between launches.  Call ``run`` once first so one-time set-up
        (device attributes, symbol lookups) happens outside the capture; the
        graph holds the current boundaries and buffer addresses."""
        graph = torch.cuda.CUDAGraph()
        side = torch.cuda.Stream(self.device) if stream is None else stream
        side.wait_stream(torch.cuda.current_stream(self.device))
        with torch.cuda.stream(side):
            with torch.cuda.graph(graph, stream=side):
                self.run(q, k, v, side)
        torch.cuda.current_stream(self.device).wait_stream(side)
        return graph
