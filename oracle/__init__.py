"""MOCAP oracle: plain, slow, obviously correct CPU reference (TEST INFRASTRUCTURE).

This package is test infrastructure only.  It may be imported by ``tests/``,
by ``__graft_entry__.smoke()`` and by the ``cpu_baseline`` / ``--impl
reference`` legs of ``bench.py`` -- never by the product package
``paper_2606_22968_gb300``.  It shares no code, header, table or helper with
the CUDA path, and never takes an input or an expected value from it.

Contents
--------
``partition``  Latency-Balanced Chunk Partitioning boundaries (Sec. 3.2, Eq. 1;
               Sec. 4.2 / Algorithm 1 stage 1 objective) in exact Python
               integers.
``attention``  Causal (GQA) prefill attention over a chunked KV prefix in
               float64 numpy (Sec. 2.2: each chunk attends to the KV of all
               earlier chunks plus itself), the KV-append definition
               (Sec. 2.2 / 3.1: KV of earlier chunks stays live) and the
               split-KV log-sum-exp combine.
``projection`` The QKV projection of a chunk (Sec. 3.2 / Eq. 1's GEMM term)
               with the rotary position embedding applied to Q and K.

Every function is pinned by ``tests/test_oracle_*.py`` against brute force,
closed forms and invariants (nothing in this package is "parity unpinned").
"""

from . import attention, partition, projection  # noqa: F401
