"""CPU float64 oracle for the AoH head-heterogeneous attention path.

TEST INFRASTRUCTURE ONLY. This package is the slow, obviously-correct
definition that the CUDA library is checked against. Only ``tests/``,
``__graft_entry__.smoke()`` and the CPU-baseline / reference leg of
``bench.py`` may import it. The product path (``paper_2608_06849_gb300``)
never imports it, and this package imports nothing from the product path:
the two share no code, headers, helpers or constants.

Modules
  attention    masked causal softmax attention with retrieval / streaming
               masks (Sec. 5 "Decode Stage", Eq. 8, and "Chunked-Prefill
               Stage"), the ring-buffer slot model of the streaming cache,
               and the decode step as a row of the same definition.
  kv_memory    KV-cache byte count (Appendix "Details on Baseline Budgets"
               32K KV-memory table; Appendix "Additional Efficiency Results"
               memory columns).
  effective_rank
               the head score of Sec. 4: effective rank of
               M_h = W_K^T W_Q (Eq. 2-4) computed three ways (explicit SVD,
               the d_head proxy C_h of Eq. 5-6, a QR route), and the
               group-level classification of Algorithm 1 plus the GQA
               extension appendix.
  h2share      index-only cross-layer sparse attention (the H2Share
               section): anchor-group importance and top-k selection,
               sparse attention at borrowed positions, the Eq. sim head
               similarity and the group mapping.

Parity status: every function here is pinned by ``tests/test_oracle_*.py``
against closed forms, brute force, a textbook library routine or values the
paper prints. None is "parity unpinned".
"""

from . import attention, effective_rank, h2share, kv_memory  # noqa: F401
