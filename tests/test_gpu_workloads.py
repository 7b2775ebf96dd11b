"""The five workloads at full size, checked on sampled outputs that the
oracle computes one by one (rows of the prefill, sequences of a decode
step), in the launch configuration bench.py times."""

import numpy as np
import pytest
import torch

from gpu_cases import assert_matches, ensure_lib, f64
from oracle import attention as oatt
from paper_2608_06849_gb300 import aoh
from paper_2608_06849_gb300.workloads import (DECODE_128K, PREFILL_32K, RAGGED, STACK_256K, decode_inputs,
                                             labels_for, prefill_inputs, randn_bf16, seq_lens)

pytestmark = pytest.mark.gpu


def _check_prefill_rows(q, k, v, out, labels, S, W, rows, g):
    qn = f64(q[0, rows])
    for kv, lab in enumerate(labels):
        kk = f64(k[0, :, kv:kv + 1])
        vv = f64(v[0, :, kv:kv + 1])
        hs = slice(kv * g, (kv + 1) * g)
        want = oatt.attend(qn[:, hs], rows, kk, vv, [lab], S, W)
        mag = oatt.attend(qn[:, hs], rows, kk, np.abs(vv), [lab], S, W)
        assert_matches(f64(out[0, rows][:, hs]), want, f"rows kv={kv}", mag)


def test_prefill_32k_qwen25_shape_sampled_rows():
    wl = PREFILL_32K
    ensure_lib()
    labels = labels_for(wl)
    q, k, v = prefill_inputs(wl, device="cuda")
    T = wl.prefill_len
    cache = aoh.Cache(1, wl.n_q_heads, wl.n_kv_heads, wl.d_head, T, wl.sink, wl.window, labels)
    out = torch.full_like(q, float("nan"))
    cache.prefill(q, k, v, out)
    torch.cuda.synchronize()
    cache.check()
    gen = np.random.default_rng(0)
    rows = np.unique(np.concatenate([np.arange(0, 130), np.arange(wl.sink - 2, wl.sink + 2),
                                     np.arange(wl.window - 2, wl.window + 130), gen.integers(0, T, 96),
                                     np.arange(T - 64, T)]))
    assert not torch.isnan(out).any()
    _check_prefill_rows(q, k, v, out, labels, wl.sink, wl.window, rows, wl.g)
    cache.close()


def _decode_check(cache, wl, labels, kfill, vfill, lens, steps, sample_b):
    g = wl.g
    hist_k = {b: [f64(kfill[b, :lens[b]])] for b in sample_b}
    hist_v = {b: [f64(vfill[b, :lens[b]])] for b in sample_b}
    for step in range(steps):
        dq, dk, dv = decode_inputs(wl, step, device="cuda")
        out = torch.full_like(dq, float("nan"))
        cache.decode_step(dq, dk, dv, out)
        torch.cuda.synchronize()
        for b in sample_b:
            hist_k[b].append(f64(dk[b])[None])
            hist_v[b].append(f64(dv[b])[None])
            kk = np.concatenate(hist_k[b], axis=0)
            vv = np.concatenate(hist_v[b], axis=0)
            hist_k[b], hist_v[b] = [kk], [vv]
            qn = f64(dq[b])
            for kv, lab in enumerate(labels):
                hs = slice(kv * g, (kv + 1) * g)
                want = oatt.decode_step(qn[hs], kk[:, kv:kv + 1], vv[:, kv:kv + 1], [lab], wl.sink, wl.window)
                mag = oatt.decode_step(qn[hs], kk[:, kv:kv + 1], np.abs(vv[:, kv:kv + 1]), [lab], wl.sink, wl.window)
                assert_matches(f64(out[b, hs]), want, f"decode step={step} b={b} kv={kv}", mag)
    cache.check()


def test_decode_128k_llama3_shape_b16_sampled():
    """Llama-3-8B-shaped decode: 16 sequences at 128K cached tokens; the cache
    is filled by prefill without output (as bench.py does); two steps; three
    sequences checked on every head."""
    wl = DECODE_128K
    ensure_lib()
    labels = labels_for(wl)
    B, T = wl.batch, wl.prefill_len
    cache = aoh.Cache(B, wl.n_q_heads, wl.n_kv_heads, wl.d_head, T + 8, wl.sink, wl.window, labels)
    kfill = randn_bf16((B, T, wl.n_kv_heads, wl.d_head), 7001, "cuda")
    vfill = randn_bf16((B, T, wl.n_kv_heads, wl.d_head), 7002, "cuda")
    cache.prefill(None, kfill, vfill, None)
    torch.cuda.synchronize()
    _decode_check(cache, wl, labels, kfill, vfill, [T] * B, 2, [0, 7, 15])
    cache.close()


@pytest.mark.parametrize("frac,W", [(0.5, 2048), (0.75, 512), (0.0, 8192), (0.25, 8192)])
def test_ragged_decode_b64_sweep_points(frac, W):
    """Ragged batch of 64 sequences with lengths uniform in [4K, 32K], S=64,
    streaming fraction and window from the sweep; every sequence checked."""
    import dataclasses
    wl = dataclasses.replace(RAGGED, n_streaming=int(frac * RAGGED.n_kv_heads), window=W)
    ensure_lib()
    labels = labels_for(wl)
    lens = seq_lens(wl)
    B, T = wl.batch, max(lens)
    cache = aoh.Cache(B, wl.n_q_heads, wl.n_kv_heads, wl.d_head, T + 4, wl.sink, wl.window, labels)
    kfill = randn_bf16((B, T, wl.n_kv_heads, wl.d_head), 7101, "cuda")
    vfill = randn_bf16((B, T, wl.n_kv_heads, wl.d_head), 7102, "cuda")
    cache.prefill(None, kfill, vfill, None, seq_lens=lens)
    torch.cuda.synchronize()
    sample = list(range(B)) if frac in (0.5, 0.75) else [0, 31, 63]
    _decode_check(cache, wl, labels, kfill, vfill, lens, 1, sample)
    cache.close()


def test_stack_256k_one_layer_sampled():
    """One layer of the 28-layer Qwen2.5-7B-shaped stack: 256K prefill with
    sampled rows, then two decode steps; the KV bytes of the whole stack
    against the all-retrieval layout."""
    import dataclasses
    wl = STACK_256K
    ensure_lib()
    labels = labels_for(wl, layer=0)
    T = wl.prefill_len
    q, k, v = prefill_inputs(wl, device="cuda")
    cache = aoh.Cache(1, wl.n_q_heads, wl.n_kv_heads, wl.d_head, T + wl.decode_steps, wl.sink, wl.window, labels)
    out = torch.full_like(q, float("nan"))
    cache.prefill(q, k, v, out)
    torch.cuda.synchronize()
    cache.check()
    gen = np.random.default_rng(1)
    rows = np.unique(np.concatenate([np.arange(0, 8), gen.integers(0, T, 24), np.arange(T - 8, T)]))
    _check_prefill_rows(q, k, v, out, labels, wl.sink, wl.window, rows, wl.g)
    del q, out
    _decode_check(cache, wl, labels, k, v, [T], 2, [0])
    total = sum(aoh.aoh_cache_bytes(cache.cfg, labels_for(wl, layer=L)) for L in range(wl.layers))
    full = wl.layers * aoh.aoh_cache_bytes(cache.cfg, [0] * wl.n_kv_heads)
    assert total == 28 * (2 * (T + wl.decode_steps) + 2 * (wl.sink + wl.window)) * wl.d_head * 4
    assert full / total > 1.96
    cache.close()


def test_h2share_at_decode_128k_sampled():
    """H2Share at the size bench.py times it (Llama-3-8B shape, B=16, 128K
    cached tokens, top_k 2048): one anchor step, then one reuse step on the
    same cache borrowing the anchor's positions. Sampled sequences: the
    anchor's selections form a valid top-k set of the oracle's importance
    (up to fp32 score error) and its outputs match the decode step; the reuse
    outputs match the oracle's attention over the borrowed positions."""
    from oracle import h2share as ohs
    wl = DECODE_128K
    ensure_lib()
    labels = labels_for(wl)
    B, T, D, g = wl.batch, wl.prefill_len, wl.d_head, wl.g
    top_k = 2048
    cache = aoh.Cache(B, wl.n_q_heads, wl.n_kv_heads, D, T + 4, wl.sink, wl.window, labels)
    kfill = randn_bf16((B, T, wl.n_kv_heads, D), 7001, "cuda")
    vfill = randn_bf16((B, T, wl.n_kv_heads, D), 7002, "cuda")
    cache.prefill(None, kfill, vfill, None)
    retr = [h for h in range(wl.n_kv_heads) if labels[h] == 0]
    idx = torch.full((B, len(retr), top_k), -7, dtype=torch.int32, device="cuda")
    dq, dk, dv = decode_inputs(wl, 0, device="cuda")
    out = torch.full_like(dq, float("nan"))
    cache.decode_step_anchor(dq, dk, dv, out, top_k, idx)
    rq, rk, rv = decode_inputs(wl, 1, device="cuda")
    rout = torch.full_like(rq, float("nan"))
    cache.decode_step_reuse(rq, rk, rv, rout, idx, top_k, list(range(len(retr))))
    torch.cuda.synchronize()
    cache.check()
    sel = idx.cpu().numpy()
    for b in (0, 9, 15):
        kk = np.concatenate([f64(kfill[b]), f64(dk[b])[None]])
        vv = np.concatenate([f64(vfill[b]), f64(dv[b])[None]])
        q = f64(dq[b])
        for i, kv in enumerate(retr):
            hs = slice(kv * g, (kv + 1) * g)
            imp = ohs.group_importance(q[hs], kk[:, kv])
            s = sel[b, i]
            assert np.all(np.diff(s) > 0) and s.min() >= 0 and s.max() <= T and len(s) == top_k
            thr = np.sort(imp)[::-1][top_k - 1]
            rest = np.setdiff1d(np.arange(T + 1), s)
            assert imp[s].min() >= thr * (1 - 1e-4) and imp[rest].max() <= thr * (1 + 1e-4)
            want = oatt.decode_step(q[hs], kk[:, kv:kv + 1], vv[:, kv:kv + 1], [0], wl.sink, wl.window)
            mag = oatt.decode_step(q[hs], kk[:, kv:kv + 1], np.abs(vv[:, kv:kv + 1]), [0], wl.sink, wl.window)
            assert_matches(f64(out[b, hs]), want, f"anchor b={b} kv={kv}", mag)
        # reuse step at position T + 1: its own new K/V appended after the anchor's
        kr = np.concatenate([kk, f64(rk[b])[None]])
        vr = np.concatenate([vv, f64(rv[b])[None]])
        qr = f64(rq[b])
        for i, kv in enumerate(retr):
            hs = slice(kv * g, (kv + 1) * g)
            pos = sel[b, i]
            want = ohs.sparse_attend(qr[hs], kr[:, kv], vr[:, kv], pos)
            mag = ohs.sparse_attend(qr[hs], kr[:, kv], np.abs(vr[:, kv]), pos)
            assert_matches(f64(rout[b, hs]), want, f"reuse b={b} kv={kv}", mag)
        for kv in range(wl.n_kv_heads):
            if labels[kv] == 0:
                continue
            hs = slice(kv * g, (kv + 1) * g)
            want = oatt.decode_step(qr[hs], kr[:, kv:kv + 1], vr[:, kv:kv + 1], [1], wl.sink, wl.window)
            mag = oatt.decode_step(qr[hs], kr[:, kv:kv + 1], np.abs(vr[:, kv:kv + 1]), [1], wl.sink, wl.window)
            assert_matches(f64(rout[b, hs]), want, f"reuse streaming b={b} kv={kv}", mag)
    cache.close()
