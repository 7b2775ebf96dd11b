"""The five workloads at full size, checked on sampled outputs that the
oracle computes one by one (rows of the prefill, sequences of a decode
step), in the launch configuration bench.py times."""

import numpy as np
import pytest
import torch

from gpu_cases import assert_matches, assert_raw, ensure_lib, f64
from oracle import attention as oatt
from paper_2608_06849_gb300 import aoh
from paper_2608_06849_gb300.workloads import (DECODE_128K, PREFILL_32K, RAGGED, STACK_256K, decode_inputs,
                                             labels_for, prefill_inputs, randn_bf16, seq_lens)

pytestmark = pytest.mark.gpu


def _check_prefill_rows(q, k, v, out, labels, S, W, rows, g, name):
    qn = f64(q[0, rows])
    for kv, lab in enumerate(labels):
        kk = f64(k[0, :, kv:kv + 1])
        vv = f64(v[0, :, kv:kv + 1])
        hs = slice(kv * g, (kv + 1) * g)
        want = oatt.attend(qn[:, hs], rows, kk, vv, [lab], S, W)
        mag = oatt.attend(qn[:, hs], rows, kk, np.abs(vv), [lab], S, W)
        got = f64(out[0, rows][:, hs])
        assert_matches(got, want, f"{name} rows kv={kv}", mag)
        assert_raw(got, want, name)


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
    _check_prefill_rows(q, k, v, out, labels, wl.sink, wl.window, rows, wl.g, "prefill_32k")
    cache.close()


def _decode_run_and_check(cache, wl, labels, kfill, vfill, lens, steps, check_steps, sample_b, name):
    """Run `steps` decode steps back to back (as bench.py does), keeping the
    outputs of `check_steps`; then, per sampled sequence and KV head, the
    oracle computes those steps' outputs as rows of one attention over the
    sequence's keys (cached prefix + every new token; a row at position t sees
    only positions <= t)."""
    g, Hkv, D = wl.g, wl.n_kv_heads, wl.d_head
    kept, qs = {}, {}
    new_k = np.zeros((steps, wl.batch, Hkv, D))
    new_v = np.zeros((steps, wl.batch, Hkv, D))
    out = torch.empty(wl.batch, wl.n_q_heads, D, dtype=torch.bfloat16, device="cuda")
    for step in range(steps):
        dq, dk, dv = decode_inputs(wl, step, device="cuda")
        out.fill_(float("nan"))
        cache.decode_step(dq, dk, dv, out)
        new_k[step], new_v[step] = f64(dk), f64(dv)
        if step in check_steps:
            kept[step] = out.clone()
            qs[step] = dq.clone()
    torch.cuda.synchronize()
    cache.check()
    assert cache.lens() == [L + steps for L in lens]
    cs = sorted(check_steps)
    for b in sample_b:
        pos = np.array([lens[b] + s for s in cs])
        for kv, lab in enumerate(labels):
            hs = slice(kv * g, (kv + 1) * g)
            kk = np.concatenate([f64(kfill[b, :lens[b], kv]), new_k[:, b, kv]])[:, None]
            vv = np.concatenate([f64(vfill[b, :lens[b], kv]), new_v[:, b, kv]])[:, None]
            qrows = np.stack([f64(qs[s][b, hs]) for s in cs])
            want = oatt.attend(qrows, pos, kk, vv, [lab], wl.sink, wl.window)
            mag = oatt.attend(qrows, pos, kk, np.abs(vv), [lab], wl.sink, wl.window)
            got = np.stack([f64(kept[s][b, hs]) for s in cs])
            assert_matches(got, want, f"{name} steps={cs} b={b} kv={kv}", mag)
            assert_raw(got, want, name)


def test_decode_128k_llama3_shape_b16_all_sequences():
    """Llama-3-8B-shaped decode: 16 sequences at 128K cached tokens, the
    cache filled by prefill without output (as bench.py does), then the
    workload's 64 steps back to back. Every sequence and KV head is checked
    at steps 0 and 63 and at two steps in between."""
    wl = DECODE_128K
    ensure_lib()
    labels = labels_for(wl)
    B, T = wl.batch, wl.prefill_len
    cache = aoh.Cache(B, wl.n_q_heads, wl.n_kv_heads, wl.d_head, T + wl.decode_steps, wl.sink, wl.window, labels)
    kfill = randn_bf16((B, T, wl.n_kv_heads, wl.d_head), 7001, "cuda")
    vfill = randn_bf16((B, T, wl.n_kv_heads, wl.d_head), 7002, "cuda")
    cache.prefill(None, kfill, vfill, None)
    torch.cuda.synchronize()
    _decode_run_and_check(cache, wl, labels, kfill, vfill, [T] * B, wl.decode_steps, {0, 1, 31, 63},
                          list(range(B)), "decode_128k")
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
    _decode_run_and_check(cache, wl, labels, kfill, vfill, lens, 2, {0, 1}, sample, "ragged_b64")
    cache.close()


def test_stack_256k_two_layers_sampled():
    """Two layers of the 28-layer Qwen2.5-7B-shaped stack (each with its own
    labels and inputs): 256K prefill with sampled rows; then the workload's
    128 decode steps on the second layer, checked at the first, a middle and
    the last step; the KV bytes of the whole stack against the all-retrieval
    layout."""
    wl = STACK_256K
    ensure_lib()
    T = wl.prefill_len
    gen = np.random.default_rng(1)
    for layer in (0, 1):
        labels = labels_for(wl, layer=layer)
        q, k, v = prefill_inputs(wl, device="cuda", seed_offset=layer)
        cache = aoh.Cache(1, wl.n_q_heads, wl.n_kv_heads, wl.d_head, T + wl.decode_steps, wl.sink, wl.window,
                          labels)
        out = torch.full_like(q, float("nan"))
        cache.prefill(q, k, v, out)
        torch.cuda.synchronize()
        cache.check()
        rows = np.unique(np.concatenate([np.arange(0, 8), np.arange(wl.window - 2, wl.window + 2),
                                         gen.integers(0, T, 24), np.arange(T - 8, T)]))
        _check_prefill_rows(q, k, v, out, labels, wl.sink, wl.window, rows, wl.g, "stack_256k_prefill")
        del q, out
        if layer == 1:
            _decode_run_and_check(cache, wl, labels, k, v, [T], wl.decode_steps, {0, 63, 127}, [0],
                                  "stack_256k_decode")
        cache.close()
        del k, v
        torch.cuda.empty_cache()
    cfg = aoh.make_config(1, wl.n_q_heads, wl.n_kv_heads, wl.d_head, T + wl.decode_steps, wl.sink, wl.window)
    total = sum(aoh.aoh_cache_bytes(cfg, labels_for(wl, layer=L)) for L in range(wl.layers))
    full = wl.layers * aoh.aoh_cache_bytes(cfg, [0] * wl.n_kv_heads)
    assert total == 28 * (2 * (T + wl.decode_steps) + 2 * (wl.sink + wl.window)) * wl.d_head * 4
    assert full / total > 1.96


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
            assert_raw(f64(out[b, hs]), want, "h2share_anchor_128k")
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
            assert_raw(f64(rout[b, hs]), want, "h2share_reuse_128k")
        for kv in range(wl.n_kv_heads):
            if labels[kv] == 0:
                continue
            hs = slice(kv * g, (kv + 1) * g)
            want = oatt.decode_step(qr[hs], kr[:, kv:kv + 1], vr[:, kv:kv + 1], [1], wl.sink, wl.window)
            mag = oatt.decode_step(qr[hs], kr[:, kv:kv + 1], np.abs(vr[:, kv:kv + 1]), [1], wl.sink, wl.window)
            assert_matches(f64(rout[b, hs]), want, f"reuse streaming b={b} kv={kv}", mag)
    cache.close()
