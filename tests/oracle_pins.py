"""Checks that pin the attention oracle to things other than itself.

Each ``pin_*`` function takes an oracle attention module (the real one, or a
mutated copy built by ``test_oracle_mutants.py``) and raises AssertionError if
the module disagrees with what the paper and the mathematics fix:
  * brute force: scalar loops over the mask conditions written out here;
  * a textbook library routine: torch's float64 scaled-dot-product attention;
  * closed forms: S=0, W=1 returns V itself; S=1, W=1 is a two-key softmax;
  * invariants: a window that covers the whole sequence equals retrieval;
    a decode step equals the matching prefill row;
  * the ring-buffer slot model holds exactly the attended positions;
  * the chunk-eviction option against a step-by-step simulation of the
    procedure of the "Chunked-Prefill Stage" (process a chunk against the
    cache, then evict all but the sinks and the W most recent tokens), plus
    two closed forms (chunks of one token; one chunk covering the prompt);
  * the scalar and the vector form of the mask against the mask conditions
    written out here, over every (query, key) pair of small cases.
"""

import math

import numpy as np


def _rng(seed):
    return np.random.default_rng(seed)


def _qkv(rng, T, Hq, Hkv, d, peaky=1.0):
    q = rng.standard_normal((T, Hq, d))
    k = rng.standard_normal((T, Hkv, d)) * peaky
    v = rng.standard_normal((T, Hkv, d))
    return q, k, v


def brute_force(q, k, v, labels, S, W):
    """Scalar loops; the mask is written as the paper states it, not called."""
    T, Hq, d = q.shape
    Hkv = k.shape[1]
    g = Hq // Hkv
    out = np.zeros_like(q)
    for h in range(Hq):
        kv = h // g
        for i in range(T):
            keys = []
            for j in range(T):
                if j > i:
                    continue
                if labels[kv] == 1 and not (j < S or i - j < W):
                    continue
                keys.append(j)
            scores = []
            for j in keys:
                acc = 0.0
                for e in range(d):
                    acc += q[i, h, e] * k[j, kv, e]
                scores.append(acc / math.sqrt(d))
            mx = max(scores)
            ws = [math.exp(s - mx) for s in scores]
            tot = sum(ws)
            for e in range(d):
                acc = 0.0
                for w, j in zip(ws, keys):
                    acc += w * v[j, kv, e]
                out[i, h, e] = acc / tot
    return out


def pin_brute_force(att):
    rng = _rng(1)
    cases = [
        (23, 4, 2, 8, [0, 1], 3, 4),
        (17, 4, 2, 8, [1, 0], 0, 7),
        (29, 6, 3, 4, [1, 1, 0], 1, 1),
        (12, 2, 1, 8, [1], 3, 7),
        (40, 4, 2, 8, [1, 1], 1, 4),
    ]
    for T, Hq, Hkv, d, labels, S, W in cases:
        q, k, v = _qkv(rng, T, Hq, Hkv, d, peaky=2.0)
        got = att.prefill(q, k, v, labels, S, W)
        want = brute_force(q, k, v, labels, S, W)
        np.testing.assert_allclose(got, want, rtol=0, atol=1e-12)


def pin_library_sdpa(att):
    """All-retrieval labels against torch's float64 causal SDPA; streaming
    labels against SDPA with a boolean mask built here from the paper's rule."""
    import torch
    import torch.nn.functional as F

    rng = _rng(2)
    T, Hq, Hkv, d = 37, 6, 2, 16
    q, k, v = _qkv(rng, T, Hq, Hkv, d, peaky=1.5)
    g = Hq // Hkv
    qt = torch.from_numpy(q).permute(1, 0, 2)[None]
    kt = torch.from_numpy(k).permute(1, 0, 2)[None].repeat_interleave(g, dim=1)
    vt = torch.from_numpy(v).permute(1, 0, 2)[None].repeat_interleave(g, dim=1)
    dense = F.scaled_dot_product_attention(qt, kt, vt, is_causal=True)[0].permute(1, 0, 2).numpy()
    got = att.prefill(q, k, v, [0, 0], 5, 3)
    np.testing.assert_allclose(got, dense, rtol=0, atol=1e-12)

    S, W = 2, 5
    mask = torch.zeros(T, T, dtype=torch.bool)
    for i in range(T):
        for j in range(i + 1):
            mask[i, j] = j < S or i - j < W
    sw = F.scaled_dot_product_attention(qt, kt, vt, attn_mask=mask)[0].permute(1, 0, 2).numpy()
    got = att.prefill(q, k, v, [1, 0], S, W)
    np.testing.assert_allclose(got[:, :g], sw[:, :g], rtol=0, atol=1e-12)
    np.testing.assert_allclose(got[:, g:], dense[:, g:], rtol=0, atol=1e-12)


def pin_window_one(att):
    """S = 0, W = 1: each query sees only itself, so the output is V exactly."""
    rng = _rng(3)
    T, Hq, Hkv, d = 19, 4, 2, 8
    q, k, v = _qkv(rng, T, Hq, Hkv, d, peaky=3.0)
    got = att.prefill(q, k, v, [1, 1], 0, 1)
    g = Hq // Hkv
    for h in range(Hq):
        np.testing.assert_allclose(got[:, h], v[:, h // g], rtol=0, atol=1e-14)


def pin_sink_one_window_one(att):
    """S = 1, W = 1: query i >= 1 sees keys {0, i}; a two-way softmax."""
    rng = _rng(4)
    T, Hq, Hkv, d = 15, 2, 1, 8
    q, k, v = _qkv(rng, T, Hq, Hkv, d, peaky=2.0)
    got = att.prefill(q, k, v, [1], 1, 1)
    for h in range(Hq):
        np.testing.assert_allclose(got[0, h], v[0, 0], rtol=0, atol=1e-14)
        for i in range(1, T):
            a = float(q[i, h] @ k[0, 0]) / math.sqrt(d)
            b = float(q[i, h] @ k[i, 0]) / math.sqrt(d)
            w0 = 1.0 / (1.0 + math.exp(b - a))
            want = w0 * v[0, 0] + (1.0 - w0) * v[i, 0]
            np.testing.assert_allclose(got[i, h], want, rtol=0, atol=1e-13)


def pin_full_window_is_retrieval(att):
    """A streaming head whose S + W covers the sequence is a retrieval head."""
    rng = _rng(5)
    T, Hq, Hkv, d = 33, 4, 2, 8
    q, k, v = _qkv(rng, T, Hq, Hkv, d)
    for S, W in [(0, T), (5, T - 5), (T, 1), (10, 40)]:
        a = att.prefill(q, k, v, [1, 1], S, W)
        b = att.prefill(q, k, v, [0, 0], S, W)
        np.testing.assert_array_equal(a, b)
    # one short of covering must differ for a late row
    a = att.prefill(q, k, v, [1, 1], 4, T - 5, rows=[T - 1])
    b = att.prefill(q, k, v, [0, 0], 4, T - 5, rows=[T - 1])
    assert np.abs(a - b).max() > 1e-6


def pin_decode_is_prefill_row(att):
    rng = _rng(6)
    T, Hq, Hkv, d = 26, 4, 2, 8
    q, k, v = _qkv(rng, T, Hq, Hkv, d)
    labels, S, W = [1, 0], 2, 5
    full = att.prefill(q, k, v, labels, S, W)
    for t in [0, 1, 2, 6, 7, 8, T - 1]:
        got = att.decode_step(q[t], k[: t + 1], v[: t + 1], labels, S, W)
        # same arithmetic; only the BLAS blocking of a 1-row product differs
        np.testing.assert_allclose(got, full[t], rtol=0, atol=1e-14)


def pin_ring_holds_attended_set(att):
    """After positions 0..t are written, the streaming cache holds exactly the
    positions a streaming query at t attends, and never more than S + W."""
    for S in [0, 1, 3, 8]:
        for W in [1, 2, 5, 8]:
            for t in range(0, 3 * (S + W) + 4):
                held = att.streaming_slots_after(t, S, W)
                want = {j for j in range(t + 1) if j < S or t - j < W}
                assert set(held.values()) == want, (S, W, t)
                assert all(0 <= s < S + W for s in held), (S, W, t)
                assert len(held) == len(want)


def pin_ring_slot_layout(att):
    """The cache layout the library documents: sinks in slots 0..S-1; position
    S goes to slot S and each later position to the next slot, wrapping from
    S + W - 1 back to S (a ring of W slots)."""
    for S in [0, 1, 4]:
        for W in [1, 3, 8]:
            for p in range(S):
                assert att.ring_slot(p, S, W) == p
            slot = S
            for p in range(S, S + 4 * W + 3):
                assert att.ring_slot(p, S, W) == slot, (S, W, p)
                slot = S if slot == S + W - 1 else slot + 1


def chunked_prefill_simulation(q, k, v, labels, S, W, K):
    """The chunked-prefill procedure run step by step for streaming heads:
    chunk c's queries attend to the cached positions plus the chunk's own
    positions up to themselves; after the chunk every cached position except
    the S sinks and the W most recent is evicted. Retrieval heads keep all."""
    T, Hq, d = q.shape
    Hkv = k.shape[1]
    g = Hq // Hkv
    out = np.zeros_like(q)
    for kv in range(Hkv):
        cache = []                       # positions held before the current chunk
        for c0 in range(0, T, K):
            chunk = list(range(c0, min(c0 + K, T)))
            for i in chunk:
                keys = cache + [j for j in chunk if j <= i]
                if labels[kv] == 0:
                    keys = list(range(i + 1))
                for h in range(kv * g, (kv + 1) * g):
                    sc = np.array([q[i, h] @ k[j, kv] for j in keys]) / math.sqrt(d)
                    w = np.exp(sc - sc.max())
                    out[i, h] = (w[:, None] * v[keys, kv]).sum(axis=0) / w.sum()
            held = cache + chunk
            recent = sorted(p for p in held if p >= S)[-W:] if W > 0 else []
            cache = [p for p in held if p < S] + recent
    return out


def pin_chunk_eviction_simulation(att):
    rng = _rng(8)
    cases = [
        (30, 4, 2, 8, [1, 0], 2, 5, 7),
        (41, 2, 1, 8, [1], 0, 3, 4),
        (25, 4, 2, 4, [1, 1], 3, 2, 10),
        (20, 2, 1, 8, [1], 1, 1, 1),
        (33, 4, 2, 8, [0, 1], 4, 6, 40),
    ]
    for T, Hq, Hkv, d, labels, S, W, K in cases:
        q, k, v = _qkv(rng, T, Hq, Hkv, d, peaky=2.0)
        got = att.prefill(q, k, v, labels, S, W, chunk=K)
        want = chunked_prefill_simulation(q, k, v, labels, S, W, K)
        np.testing.assert_allclose(got, want, rtol=0, atol=1e-12)


def pin_chunk_closed_forms(att):
    """Chunks of one token see the sinks plus the W positions before the
    query and the query itself: the per-token rule with a window of W + 1.
    One chunk covering the prompt sees everything causally (retrieval)."""
    rng = _rng(9)
    T, Hq, Hkv, d = 29, 4, 2, 8
    q, k, v = _qkv(rng, T, Hq, Hkv, d, peaky=2.0)
    for S, W in [(0, 1), (2, 4), (3, 9)]:
        a = att.prefill(q, k, v, [1, 0], S, W, chunk=1)
        b = att.prefill(q, k, v, [1, 0], S, W + 1)
        np.testing.assert_array_equal(a, b)
        a = att.prefill(q, k, v, [1, 1], S, W, chunk=T)
        b = att.prefill(q, k, v, [0, 0], S, W)
        np.testing.assert_array_equal(a, b)
    # chunk = 0 is the per-token rule
    np.testing.assert_array_equal(att.prefill(q, k, v, [1, 0], 2, 4, chunk=0), att.prefill(q, k, v, [1, 0], 2, 4))


def _mask_written_out(i, j, streaming, S, W, chunk):
    """The visibility rule as Sec. 5 states it, with the readings of the
    module docstring: causal; a streaming head keeps the S sinks and either
    the W positions up to the query (per-token window) or, with eviction
    after each chunk of K tokens, the W positions before the query's chunk
    plus the chunk itself."""
    if j > i:
        return False
    if not streaming or j < S:
        return True
    if chunk == 0:
        return j > i - W
    chunk_start = i - i % chunk
    return j >= chunk_start - W


def pin_scalar_mask(att):
    """``allowed`` (scalar) and ``allowed_mask`` (vector) over every pair
    (i, j) of small cases, with and without the chunk rule, against the
    conditions written out above."""
    for streaming in (False, True):
        for S in (0, 1, 3):
            for W in (1, 2, 5):
                for chunk in (0, 1, 3, 4):
                    T = 3 * (S + W) + 2 * max(chunk, 1) + 1
                    mask = att.allowed_mask(np.arange(T), np.arange(T), streaming, S, W, chunk)
                    assert mask.shape == (T, T)
                    for i in range(T):
                        for j in range(T):
                            want = _mask_written_out(i, j, streaming, S, W, chunk)
                            assert bool(att.allowed(i, j, streaming, S, W, chunk)) == want, (
                                "allowed", i, j, streaming, S, W, chunk)
                            assert bool(mask[i, j]) == want, ("allowed_mask", i, j, streaming, S, W, chunk)


ALL_PINS = [
    pin_brute_force,
    pin_library_sdpa,
    pin_window_one,
    pin_sink_one_window_one,
    pin_full_window_is_retrieval,
    pin_decode_is_prefill_row,
    pin_ring_holds_attended_set,
    pin_ring_slot_layout,
    pin_chunk_eviction_simulation,
    pin_chunk_closed_forms,
    pin_scalar_mask,
]
