"""The allocation-free decode entry point, held to the oracle.

Some callers cannot allocate device memory once they are running (a server
whose memory arena is planned at start-up, a loop that cannot take
cudaMalloc's device-wide synchronisation). aoh_decode_step_noalloc serves
them: its scratch is a static device array inside the library and the caller
passes the KV buffer and the device lengths. These tests drive it through the
C ABI for several calls in a row and compare every output with the float64
oracle on the same bf16 inputs (and with aoh_decode_step on an identical
cache); they also check the device-side capacity guard and the sticky status
word. The file is named to be collected last."""

import numpy as np
import pytest
import torch

from gpu_cases import MAX_ABS, MEAN_ABS, assert_matches, ensure_lib, f64
from oracle import attention as oatt
from paper_2608_06849_gb300 import aoh
from paper_2608_06849_gb300.workloads import Workload, decode_inputs, randn_bf16

pytestmark = pytest.mark.gpu


def _oracle_check(out, q, kk, vv, labels, S, W, g, what):
    """Every (sequence, KV head) of a decode output against the oracle;
    kk / vv: per sequence the float64 keys / values of positions 0..t."""
    for b in range(len(kk)):
        qn = f64(q[b])
        for kv, lab in enumerate(labels):
            hs = slice(kv * g, (kv + 1) * g)
            want = oatt.decode_step(qn[hs], kk[b][:, kv:kv + 1], vv[b][:, kv:kv + 1], [lab], S, W)
            mag = oatt.decode_step(qn[hs], kk[b][:, kv:kv + 1], np.abs(vv[b][:, kv:kv + 1]), [lab], S, W)
            assert_matches(f64(out[b, hs]), want, f"{what} b={b} kv={kv}", mag)


@pytest.mark.parametrize("B,Hq,Hkv,D,T,S,W,labels", [
    (4, 32, 8, 128, 9000, 64, 1000, [1, 0, 0, 1, 1, 0, 0, 1]),
    (2, 8, 2, 64, 700, 16, 100, [0, 1]),
    (2, 28, 4, 128, 5000, 32, 700, [0, 1, 1, 0]),
])
def test_noalloc_decode_matches_oracle(B, Hq, Hkv, D, T, S, W, labels):
    """Three calls in a row; each output against the oracle, and against the
    handle API's step on an identical cache."""
    ensure_lib()
    steps = 3
    wl = Workload("noalloc", B, Hq, Hkv, D, T, steps, S, W, sum(labels), seed=3)
    cache = aoh.Cache(B, Hq, Hkv, D, T + 4, S, W, labels)
    k = randn_bf16((B, T, Hkv, D), 11, "cuda")
    v = randn_bf16((B, T, Hkv, D), 12, "cuda")
    cache.prefill(None, k, v, None)
    torch.cuda.synchronize()
    kv_copy = cache.buffer.clone()                       # identical cache for the no-alloc path
    lens = torch.full((B,), T, dtype=torch.int32, device="cuda")
    kk = [f64(k[b]) for b in range(B)]
    vv = [f64(v[b]) for b in range(B)]
    g = Hq // Hkv
    for step in range(steps):
        q, kn, vn = decode_inputs(wl, step, device="cuda")
        out_ref = torch.full_like(q, float("nan"))
        out_na = torch.full_like(q, float("nan"))
        cache.decode_step(q, kn, vn, out_ref)
        aoh.aoh_decode_step_noalloc(cache.cfg, labels, kv_copy, lens, T + step, q, kn, vn, out_na)
        torch.cuda.synchronize()
        assert torch.isfinite(out_na.float()).all()
        assert lens.tolist() == [T + step + 1] * B
        for b in range(B):
            kk[b] = np.concatenate([kk[b], f64(kn[b])[None]])
            vv[b] = np.concatenate([vv[b], f64(vn[b])[None]])
        _oracle_check(out_na, q, kk, vv, labels, S, W, g, f"noalloc step={step}")
        _oracle_check(out_ref, q, kk, vv, labels, S, W, g, f"handle step={step}")
        err = (out_na.float() - out_ref.float()).abs()
        assert err.max().item() <= MAX_ABS, err.max().item()
        assert err.mean().item() <= MEAN_ABS, err.mean().item()
    cache.check()
    assert torch.equal(kv_copy, cache.buffer)            # the same rows were appended
    assert aoh.aoh_decode_step_noalloc_status() == (aoh.AOH_OK, 0)
    cache.close()


def test_noalloc_decode_replays_from_a_cuda_graph():
    """Decode steps captured once in a CUDA graph (the launch-bound inner loop
    of a server) and replayed give the same outputs as the handle API step by
    step; the device lengths advance on replay."""
    ensure_lib()
    B, Hq, Hkv, D, T, S, W, labels = 2, 32, 8, 128, 5000, 64, 700, [1, 0, 0, 1, 1, 0, 0, 1]
    steps = 3
    wl = Workload("graph", B, Hq, Hkv, D, T, steps + 1, S, W, sum(labels), seed=4)
    cache = aoh.Cache(B, Hq, Hkv, D, T + steps + 2, S, W, labels)
    k = randn_bf16((B, T, Hkv, D), 21, "cuda")
    v = randn_bf16((B, T, Hkv, D), 22, "cuda")
    cache.prefill(None, k, v, None)
    torch.cuda.synchronize()
    kv_copy = cache.buffer.clone()
    lens = torch.full((B,), T, dtype=torch.int32, device="cuda")
    inputs = [decode_inputs(wl, s, device="cuda") for s in range(steps + 1)]
    # step 0 outside the graph: the first call sets the library up (symbol
    # address, kernel attributes)
    ref0 = torch.empty_like(inputs[0][0])
    na0 = torch.empty_like(inputs[0][0])
    cache.decode_step(*inputs[0], ref0)
    aoh.aoh_decode_step_noalloc(cache.cfg, labels, kv_copy, lens, T, *inputs[0], na0)
    torch.cuda.synchronize()
    outs = [torch.full_like(inputs[0][0], float("nan")) for _ in range(steps)]
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        for s in range(steps):
            aoh.aoh_decode_step_noalloc(cache.cfg, labels, kv_copy, lens, T + 1 + s, *inputs[s + 1], outs[s])
    torch.cuda.synchronize()
    assert lens.tolist() == [T + 1] * B            # capture ran nothing
    graph.replay()
    torch.cuda.synchronize()
    assert lens.tolist() == [T + 1 + steps] * B
    for s in range(steps):
        ref = torch.empty_like(outs[s])
        cache.decode_step(*inputs[s + 1], ref)
        torch.cuda.synchronize()
        assert torch.isfinite(outs[s].float()).all()
        err = (outs[s].float() - ref.float()).abs()
        assert err.max().item() <= MAX_ABS, (s, err.max().item())
        assert err.mean().item() <= MEAN_ABS, (s, err.mean().item())
    assert torch.equal(kv_copy, cache.buffer)
    cache.close()


@pytest.mark.parametrize("labels", [[0, 1], [0, 0]])
def test_noalloc_skips_a_full_sequence(labels):
    """A caller whose host bound has gone stale (max_len below the device
    lengths, as when one captured graph is replayed for many steps) reaches a
    sequence already holding max_seq tokens. The kernel skips that sequence
    (nothing appended, no output, length kept), decodes the others, and the
    sticky status reports CAPACITY once. The KV buffer is passed with a
    padded tail, so even a missing guard would write inside the tensor; the
    test checks the region after the full sequence's rows and the padding."""
    ensure_lib()
    B, Hq, Hkv, D, S, W, max_seq = 3, 8, 2, 128, 16, 100, 600
    g = Hq // Hkv
    fill = [600, 300, 599]                     # sequence 0 is full; 2 has one row left
    wl = Workload("capacity", B, Hq, Hkv, D, max_seq, 2, S, W, sum(labels), seed=5)
    cache = aoh.Cache(B, Hq, Hkv, D, max_seq, S, W, labels)
    k = randn_bf16((B, max_seq, Hkv, D), 31, "cuda")
    v = randn_bf16((B, max_seq, Hkv, D), 32, "cuda")
    cache.prefill(None, k, v, None, seq_lens=fill)
    torch.cuda.synchronize()
    pad = 1 << 20
    kv = torch.full((cache.nbytes + pad,), 0x5A, dtype=torch.uint8, device="cuda")
    kv[:cache.nbytes] = cache.buffer
    before = kv.clone()
    lens = torch.tensor(fill, dtype=torch.int32, device="cuda")
    assert aoh.aoh_decode_step_noalloc_status()[0] == aoh.AOH_OK   # clears anything earlier
    kk = [f64(k[b, :fill[b]]) for b in range(B)]
    vv = [f64(v[b, :fill[b]]) for b in range(B)]
    for step in range(2):
        q, kn, vn = decode_inputs(wl, step, device="cuda")
        out = torch.full_like(q, float("nan"))
        # a stale host bound: 598 passes the host check (598 + 1 <= 600)
        aoh.aoh_decode_step_noalloc(cache.cfg, labels, kv, lens, 598, q, kn, vn, out)
        torch.cuda.synchronize()
        want_lens = [600, 300 + step + 1, 600]
        assert lens.tolist() == want_lens, (step, lens.tolist())
        assert torch.isnan(out[0].float()).all()                 # skipped: not written
        live = [1, 2] if step == 0 else [1]                       # sequence 2 fills at step 0
        if step == 1:
            assert torch.isnan(out[2].float()).all()
        for b in live:
            kk[b] = np.concatenate([kk[b], f64(kn[b])[None]])
            vv[b] = np.concatenate([vv[b], f64(vn[b])[None]])
            qn = f64(q[b])
            for kv_h, lab in enumerate(labels):
                hs = slice(kv_h * g, (kv_h + 1) * g)
                want = oatt.decode_step(qn[hs], kk[b][:, kv_h:kv_h + 1], vv[b][:, kv_h:kv_h + 1], [lab], S, W)
                mag = oatt.decode_step(qn[hs], kk[b][:, kv_h:kv_h + 1], np.abs(vv[b][:, kv_h:kv_h + 1]), [lab],
                                       S, W)
                assert_matches(f64(out[b, hs]), want, f"capacity step={step} b={b} kv={kv_h}", mag)
        st, flags = aoh.aoh_decode_step_noalloc_status()
        assert st == 2 and flags == 2, (st, flags)                # CAPACITY, reported once
        assert aoh.aoh_decode_step_noalloc_status() == (aoh.AOH_OK, 0)
    # nothing outside the rows the live sequences appended has changed
    changed = (kv != before).nonzero().flatten()
    allowed = torch.zeros_like(kv, dtype=torch.bool)
    for b, rows in ((1, [300, 301]), (2, [599])):
        for h in range(Hkv):
            ko, vo, cap = aoh.aoh_cache_region(cache.handle, b, h)
            for p in rows:
                r = p if labels[h] == 0 else oatt.ring_slot(p, S, W)
                for base in (ko, vo):
                    allowed[base + r * D * 2: base + (r + 1) * D * 2] = True
    assert allowed[changed].all(), changed[~allowed[changed]][:8].tolist()
    assert torch.equal(kv[cache.nbytes:], before[cache.nbytes:])
    cache.close()


def test_noalloc_recovers_from_a_timeout():
    """A bounded wait that runs out inside an allocation-free step: the call
    itself cannot report it (it returns before the kernel runs), so the
    status word must; and the launch must leave the static scratch clean, or
    the next step's merges would start from stale arrival counts. The
    self-test entry point stalls one CTA until its wait gives up (about
    2 s); the cache and lengths are then restored from copies (the stalled
    CTA may not have appended the new token) and a plain call must match
    the oracle."""
    ensure_lib()
    B, Hq, Hkv, D, T, S, W, labels = 2, 32, 8, 128, 3000, 64, 500, [1, 0, 0, 1, 1, 0, 0, 1]
    g = Hq // Hkv
    wl = Workload("timeout", B, Hq, Hkv, D, T, 1, S, W, sum(labels), seed=13)
    cache = aoh.Cache(B, Hq, Hkv, D, T + 4, S, W, labels)
    k = randn_bf16((B, T, Hkv, D), 41, "cuda")
    v = randn_bf16((B, T, Hkv, D), 42, "cuda")
    cache.prefill(None, k, v, None)
    torch.cuda.synchronize()
    saved = cache.buffer.clone()
    q, kn, vn = decode_inputs(wl, 0, device="cuda")
    aoh.aoh_decode_step_noalloc_status()                      # clear anything earlier
    kv = saved.clone()
    lens = torch.full((B,), T, dtype=torch.int32, device="cuda")
    junk = torch.empty_like(q)
    aoh.aoh_decode_step_noalloc(cache.cfg, labels, kv, lens, T, q, kn, vn, junk, _selftest=True)
    st, flags = aoh.aoh_decode_step_noalloc_status()
    assert st == 4 and flags & 1, (st, flags)                  # TIMEOUT, reported once
    assert aoh.aoh_decode_step_noalloc_status() == (aoh.AOH_OK, 0)
    assert lens.tolist() == [T + 1] * B
    kv = saved.clone()
    lens.fill_(T)
    out = torch.full_like(q, float("nan"))
    aoh.aoh_decode_step_noalloc(cache.cfg, labels, kv, lens, T, q, kn, vn, out)
    torch.cuda.synchronize()
    assert aoh.aoh_decode_step_noalloc_status() == (aoh.AOH_OK, 0)
    kk = [np.concatenate([f64(k[b]), f64(kn[b])[None]]) for b in range(B)]
    vv = [np.concatenate([f64(v[b]), f64(vn[b])[None]]) for b in range(B)]
    _oracle_check(out, q, kk, vv, labels, S, W, g, "after a timeout")
    cache.close()
