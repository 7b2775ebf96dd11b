"""The work counts bench.py divides by: attended (query, key) pairs of a
prefill, per-token and under the chunk-eviction rule, checked against the
oracle's masks on small prompts (every allowed pair counted once)."""

import os
import sys

import numpy as np
import pytest

from oracle import attention as oatt

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
import bench  # noqa: E402


@pytest.mark.parametrize("T,S,W", [(1, 0, 1), (50, 3, 7), (64, 0, 64), (90, 8, 20), (17, 20, 4)])
def test_attended_pairs_per_token(T, S, W):
    for streaming in (False, True):
        m = oatt.allowed_mask(np.arange(T), np.arange(T), streaming, S, W)
        assert bench.attended_pairs(T, S, W, streaming) == int(m.sum())


@pytest.mark.parametrize("T,S,W,K", [(50, 3, 7, 8), (33, 0, 5, 1), (40, 4, 10, 100), (129, 2, 30, 64)])
def test_attended_pairs_chunk_rule(T, S, W, K):
    for streaming in (False, True):
        m = oatt.allowed_mask(np.arange(T), np.arange(T), streaming, S, W, K)
        assert bench.attended_pairs_chunk(T, S, W, K, streaming) == int(m.sum())


def test_reuse_bytes_reduce_to_decode_bytes():
    """With top_k covering every row, a reuse step moves the decode step's
    bytes plus its index lists (4 bytes per borrowed row)."""
    from paper_2608_06849_gb300.workloads import DECODE_128K, labels_for
    wl = DECODE_128K
    labels = labels_for(wl)
    lens = [1000, 37, 5000]
    n_r = sum(1 for x in labels if x == 0)
    big = bench.reuse_bytes(lens, labels, wl, 10 ** 9)
    assert big == bench.decode_bytes(lens, labels, wl) + 4 * n_r * sum(t + 1 for t in lens)
    small = bench.reuse_bytes(lens, labels, wl, 8)
    assert small < big


@pytest.mark.parametrize("lens,S,W", [([0, 5, 40], 2, 8), ([100], 0, 1), ([3, 300], 16, 300)])
def test_decode_bytes_from_the_oracle_mask(lens, S, W):
    """Bytes of one decode step counted from the keys the oracle lets the new
    token see: every visible cached row read once (K and V), the new token's
    K/V read and appended, q read and out written."""
    import dataclasses

    from paper_2608_06849_gb300.workloads import DECODE_128K
    wl = dataclasses.replace(DECODE_128K, batch=len(lens), sink=S, window=W)
    labels = [0, 1, 1, 0, 1, 0, 0, 1]
    row = wl.d_head * 2
    want = 0
    for t in lens:
        for lab in labels:
            seen = int(oatt.allowed_mask(np.array([t]), np.arange(t + 1), lab == 1, S, W).sum())
            want += (seen - 1) * row * 2 + row * 2 * 2
        want += wl.n_q_heads * wl.d_head * 2 * 2
    assert bench.decode_bytes(lens, labels, wl) == want
