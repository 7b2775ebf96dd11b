"""AoH head-heterogeneous causal attention on GB300 (sm_103a).

Retrieval KV heads run full causal attention over a full KV cache; streaming
KV heads attend to S sink tokens plus a W-token recent window kept in a
fixed-size per-head ring buffer (Sec. 5 of the paper, "Decode Stage" and
"Chunked-Prefill Stage"). The work is done by hand-written CUDA kernels behind
the C ABI declared in ``include/aoh.h``; ``paper_2608_06849_gb300.aoh`` is the
thin ctypes binding, ``paper_2608_06849_gb300.workloads`` the seeded synthetic
inputs.

Importing this package loads nothing; ``aoh.load()`` (called by every binding
function) loads ``libaoh.so`` and raises if it is missing.
"""

__all__ = ["aoh", "workloads"]
