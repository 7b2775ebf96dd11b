"""Masked causal softmax attention for retrieval and streaming KV heads.

TEST INFRASTRUCTURE ONLY (see the package docstring): the plain float64
definition that the CUDA path is compared with. Parity status: pinned
(brute force, closed forms, a library attention routine, invariants, and
both forms of the mask against the rule written out pair by pair) by
``tests/test_oracle_attention.py``.

What the paper fixes (Sec. 5, "Decode Stage", Eq. 8 and "Chunked-Prefill
Stage"; Appendix "GQA Extension"):
  * every KV head carries one label, retrieval or streaming, and the query
    heads of its GQA group inherit it;
  * retrieval heads attend to the whole causal prefix;
  * streaming heads keep only ``S`` sink tokens and ``W`` recent tokens;
  * each head is computed on its own and the outputs sit side by side on the
    head axis (the concatenation of Eq. 8; the W_O projection is not part of
    attention and is not modelled).

Readings taken where the paper is silent:
  * the recent window counts the query's own position, so a streaming query
    at position i sees key j iff ``j <= i and (j < S or i - j < W)``;
  * prefill uses that per-token rule for every row by default, which makes
    prefill row t and a decode step at position t the same computation;
  * the literal chunk rule of the "Chunked-Prefill Stage" (evict all but the
    sinks and the W most recent tokens after each chunk of K tokens) is the
    ``chunk=K`` option of the prefill functions: a streaming query at
    position i in chunk c = i // K sees key j iff ``j <= i and (j < S or
    j >= c*K - W)`` (the cache as it stood after chunk c - 1, plus chunk c
    itself). Decode keeps the per-token rule in both modes;
  * query head h belongs to KV head ``h // (Hq // Hkv)``;
  * the score scale is ``1/sqrt(d_head)``.
"""

import numpy as np

RETRIEVAL = 0
STREAMING = 1


def allowed(i, j, streaming, S, W, chunk=0):
    """True iff query position i may attend key position j (scalar form).
    chunk = 0: the per-token window; chunk = K > 0: eviction after each
    K-token chunk (see the module docstring)."""
    if j > i:
        return False
    if not streaming:
        return True
    if chunk:
        return j < S or j >= (i // chunk) * chunk - W
    return j < S or i - j < W


def allowed_mask(q_pos, k_pos, streaming, S, W, chunk=0):
    """Boolean [len(q_pos), len(k_pos)] mask; the vector form of ``allowed``."""
    i = np.asarray(q_pos, dtype=np.int64)[:, None]
    j = np.asarray(k_pos, dtype=np.int64)[None, :]
    causal = j <= i
    if not streaming:
        return causal
    if chunk:
        return causal & ((j < S) | (j >= (i // chunk) * chunk - W))
    return causal & ((j < S) | (i - j < W))


def attend(q_rows, q_pos, k, v, labels, S, W, chunk=0):
    """Attention output for a set of query rows of one sequence.

    q_rows  [R, Hq, d]   queries, float64
    q_pos   [R]          their positions in the sequence
    k, v    [Tk, Hkv, d] keys / values at positions 0..Tk-1
    labels  [Hkv]        RETRIEVAL (0) or STREAMING (1) per KV head
    returns [R, Hq, d]   float64

    For each query head the steps are those of softmax attention:
    scores = q k^T / sqrt(d); disallowed scores set to -inf; subtract the row
    maximum; exponentiate; normalise by the row sum; multiply by V.
    """
    q_rows = np.asarray(q_rows, dtype=np.float64)
    k = np.asarray(k, dtype=np.float64)
    v = np.asarray(v, dtype=np.float64)
    R, Hq, d = q_rows.shape
    Tk, Hkv, _ = k.shape
    if Hq % Hkv != 0:
        raise ValueError("n_q_heads must be a multiple of n_kv_heads")
    g = Hq // Hkv
    q_pos = np.asarray(q_pos, dtype=np.int64)
    if R and int(q_pos.max()) >= Tk:
        raise ValueError("a query position has no key at its own position")
    out = np.zeros((R, Hq, d), dtype=np.float64)
    k_pos = np.arange(Tk)
    scale = 1.0 / np.sqrt(d)
    for kv in range(Hkv):
        streaming = int(labels[kv]) == STREAMING
        mask = allowed_mask(q_pos, k_pos, streaming, S, W, chunk)
        for h in range(kv * g, (kv + 1) * g):
            s = (q_rows[:, h, :] @ k[:, kv, :].T) * scale
            s = np.where(mask, s, -np.inf)
            m = s.max(axis=1, keepdims=True)
            p = np.exp(s - m)
            p = p / p.sum(axis=1, keepdims=True)
            out[:, h, :] = p @ v[:, kv, :]
    return out


def prefill(q, k, v, labels, S, W, rows=None, chunk=0):
    """Prefill output of one sequence: rows of ``attend`` over its own keys.

    q [T, Hq, d], k/v [T, Hkv, d]. ``rows`` selects the query positions to
    compute (all T when None); every row only ever sees keys at positions
    <= itself, so any subset is computed exactly as in the full matrix.
    ``chunk``: 0 for the per-token streaming window, K > 0 for eviction
    after each K-token chunk.
    """
    T = q.shape[0]
    rows = np.arange(T) if rows is None else np.asarray(rows, dtype=np.int64)
    return attend(np.asarray(q)[rows], rows, k, v, labels, S, W, chunk)


def decode_step(q_new, k_seq, v_seq, labels, S, W):
    """One decode step: the new token sits at position t = len(k_seq) - 1.

    q_new [Hq, d]; k_seq/v_seq [t+1, Hkv, d] hold positions 0..t, the new
    token's key/value last. The result is row t of ``prefill`` over the same
    sequence (Eq. 8 applied to the token being generated).
    """
    t = k_seq.shape[0] - 1
    return attend(np.asarray(q_new)[None], np.array([t]), k_seq, v_seq, labels, S, W)[0]


# --------------------------------------------------------------------------
# Streaming-head cache: S sink slots followed by a W-slot ring (Sec. 5,
# "Chunked-Prefill Stage": persistent storage bounded by s_sink + s_recent).


def ring_slot(p, S, W):
    """Cache slot that position p is written to in a streaming head's cache."""
    if p < S:
        return p
    return S + (p - S) % W


def streaming_slots_after(t, S, W):
    """slot -> position held after positions 0..t have been written in order."""
    held = {}
    for p in range(t + 1):
        held[ring_slot(p, S, W)] = p
    return held


def streaming_cache_image(k_seq, S, W):
    """Contents of one streaming head's cache after writing k_seq[0..T-1].

    k_seq [T, d]. Returns ([S + W, d] array, [S + W] bool written-flags).
    Unwritten slots are left as zeros and flagged False.
    """
    T, d = k_seq.shape
    img = np.zeros((S + W, d), dtype=k_seq.dtype)
    written = np.zeros(S + W, dtype=bool)
    for slot, p in streaming_slots_after(T - 1, S, W).items():
        img[slot] = k_seq[p]
        written[slot] = True
    return img, written
