"""KV-cache byte count of a head-heterogeneous cache.

TEST INFRASTRUCTURE ONLY (see the package docstring). Parity status: pinned
by ``tests/test_oracle_kv_memory.py`` against the numbers the paper prints in
the 32K KV-memory table (Appendix "Details on Baseline Budgets") and in the
prefill-memory columns of the efficiency tables (Appendix "Additional
Efficiency Results").

A retrieval KV head keeps K and V for every position (Sec. 5, "Decode
Stage": layer-specific full K/V states); a streaming KV head keeps a fixed
cache of S sink plus W recent positions ("Chunked-Prefill Stage"). Both store
bf16 (2 bytes), K and V.
"""

import math


def kv_cache_bytes(batch, n_retrieval, n_streaming, max_seq, S, W, d_head, elem_bytes=2):
    """Bytes of K and V for one layer: B * (n_R * max_seq + n_S * (S + W)) * d * 2 * elem."""
    tokens = n_retrieval * max_seq + n_streaming * (S + W)
    return batch * tokens * d_head * 2 * elem_bytes


def retrieval_groups(n_kv_groups, sparsity_pct):
    """k = ceil((1 - s) * G) with s given in percent, in integer arithmetic.

    The paper prints the budget as ``k = ceil((1-s),G)`` (Sec. 4,
    "Group-level Classification"); the comma is read as a product.
    """
    num = (100 - int(sparsity_pct)) * int(n_kv_groups)
    return -(-num // 100)


def model_kv_bytes(layers, n_kv_heads, sparsity_pct, ctx, S, W, d_head, batch=1):
    """Whole-model KV bytes for a uniform per-layer retrieval budget."""
    k = retrieval_groups(n_kv_heads, sparsity_pct)
    return layers * kv_cache_bytes(batch, k, n_kv_heads - k, ctx, S, W, d_head)


def gib(nbytes):
    return nbytes / float(1 << 30)


def gb(nbytes):
    return nbytes / 1e9


def round_half_up(x, decimals):
    """Round the way a printed table does (ties away from zero)."""
    f = 10 ** decimals
    return math.floor(x * f + 0.5) / f
