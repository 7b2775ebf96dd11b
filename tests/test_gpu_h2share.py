"""H2Share on the GPU (the paper's H2Share section, GQA extension appendix)
against the oracle on the same bf16 inputs.

Anchor step: the decode output as in every decode test; the selected
positions form a valid top-k set of the oracle's float64 importance. The
GPU ranks fp32 scores, so positions whose importance lies within the fp32
error of the k-th value may legitimately differ: every selected position
must be at least the k-th importance and every other at most it, each up
to that error (1e-4 relative). Reuse step: retrieval groups against the
oracle's sparse attention over the given positions (the lists the anchor
produced, or synthetic lists), streaming groups against the decode step;
the cache image is checked bit-exactly.
"""

import numpy as np
import pytest
import torch

from gpu_cases import assert_matches, check_cache_image, ensure_lib, f64
from oracle import attention as oatt
from oracle import h2share as ohs
from paper_2608_06849_gb300 import aoh
from paper_2608_06849_gb300.workloads import Workload, decode_inputs, randn_bf16

pytestmark = pytest.mark.gpu
REL = 1e-4


def _filled_cache(B, Hq, Hkv, D, T, S, W, labels, steps, seed):
    cache = aoh.Cache(B, Hq, Hkv, D, T + steps, S, W, labels)
    k = randn_bf16((B, T, Hkv, D), seed + 1, "cuda")
    v = randn_bf16((B, T, Hkv, D), seed + 2, "cuda")
    k[:, 0] *= 8
    cache.prefill(None, k, v, None)
    torch.cuda.synchronize()
    return cache, k, v


def _check_selection(sel, imp, k):
    n = imp.shape[0]
    m = min(k, n)
    assert np.all(sel[m:] == -1)
    s = sel[:m]
    assert np.all(np.diff(s) > 0) and s.min() >= 0 and s.max() < n
    if m == n:
        return
    thr = np.sort(imp)[::-1][m - 1]
    tol = REL * thr + 1e-12
    rest = np.setdiff1d(np.arange(n), s)
    assert imp[s].min() >= thr - tol, (imp[s].min(), thr)
    assert imp[rest].max() <= thr + tol, (imp[rest].max(), thr)


@pytest.mark.parametrize("B,Hq,Hkv,T,labels,top_k", [
    (2, 8, 2, 700, [0, 1], 64),
    (1, 14, 2, 1500, [0, 0], 300),
    (2, 16, 4, 257, [0, 1, 0, 1], 1000),      # top_k beyond the rows held
    (1, 8, 2, 4000, [0, 0], 1),
    (1, 2, 2, 900, [0, 1], 100),       # one query head per group
    (1, 8, 4, 700, [0, 0, 1, 0], 50),  # groups of 2
    (1, 32, 2, 600, [0, 1], 128),      # groups of 16
    (1, 8, 2, 5, [0, 1], 2),           # one slice holds every row, the others none
])
def test_anchor_step_selects_top_k(B, Hq, Hkv, T, labels, top_k):
    ensure_lib()
    D, S, W, steps = 128, 4, 64, 2
    g = Hq // Hkv
    cache, k, v = _filled_cache(B, Hq, Hkv, D, T, S, W, labels, steps, 31)
    wl = Workload("anchor", B, Hq, Hkv, D, T, steps, S, W, sum(labels), seed=4)
    retr = [h for h in range(Hkv) if labels[h] == 0]
    kall = [f64(k[b]) for b in range(B)]
    vall = [f64(v[b]) for b in range(B)]
    for step in range(steps):
        dq, dk, dv = decode_inputs(wl, step, device="cuda")
        out = torch.full_like(dq, float("nan"))
        idx = torch.full((B, len(retr), top_k), -7, dtype=torch.int32, device="cuda")
        cache.decode_step_anchor(dq, dk, dv, out, top_k, idx)
        torch.cuda.synchronize()
        sel = idx.cpu().numpy()
        for b in range(B):
            kall[b] = np.concatenate([kall[b], f64(dk[b])[None]])
            vall[b] = np.concatenate([vall[b], f64(dv[b])[None]])
            qb = f64(dq[b])
            want = oatt.decode_step(qb, kall[b], vall[b], labels, S, W)
            mag = oatt.decode_step(qb, kall[b], np.abs(vall[b]), labels, S, W)
            assert_matches(f64(out[b]), want, f"anchor decode {step} b={b}", mag)
            for i, kvh in enumerate(retr):
                imp = ohs.group_importance(qb[kvh * g:(kvh + 1) * g], kall[b][:, kvh])
                _check_selection(sel[b, i], imp, top_k)
    cache.check()
    cache.close()


def test_anchor_selection_when_length_crosses_top_k():
    """Steps with t + 1 <= top_k keep every row; the first step beyond it
    must rank from that step's importances alone."""
    ensure_lib()
    B, Hq, Hkv, D, T, S, W, top_k, steps = 2, 8, 2, 128, 60, 4, 16, 62, 4
    labels = [0, 1]
    g = Hq // Hkv
    cache, k, v = _filled_cache(B, Hq, Hkv, D, T, S, W, labels, steps, 81)
    wl = Workload("cross", B, Hq, Hkv, D, T, steps, S, W, 1, seed=9)
    kall = [f64(k[b]) for b in range(B)]
    for step in range(steps):
        dq, dk, dv = decode_inputs(wl, step, device="cuda")
        idx = torch.full((B, 1, top_k), -7, dtype=torch.int32, device="cuda")
        cache.decode_step_anchor(dq, dk, dv, torch.empty_like(dq), top_k, idx)
        torch.cuda.synchronize()
        sel = idx.cpu().numpy()
        for b in range(B):
            kall[b] = np.concatenate([kall[b], f64(dk[b])[None]])
            imp = ohs.group_importance(f64(dq[b])[:g], kall[b][:, 0])
            _check_selection(sel[b, 0], imp, top_k)
    cache.close()


def test_anchor_selection_with_one_crowded_bucket():
    """Identical keys give every cached position the same importance (the
    new token's differs): one histogram bucket holds more rows than the
    candidate list, so the threshold comes from full passes, and the tied
    rows are taken in position order across several chunks."""
    ensure_lib()
    B, Hq, Hkv, D, T, S, W, top_k = 1, 8, 2, 128, 20000, 4, 64, 9000
    labels = [0, 1]
    g = Hq // Hkv
    cache = aoh.Cache(B, Hq, Hkv, D, T + 1, S, W, labels)
    k = randn_bf16((B, 1, Hkv, D), 91, "cuda").expand(B, T, Hkv, D).contiguous()
    v = randn_bf16((B, T, Hkv, D), 92, "cuda")
    cache.prefill(None, k, v, None)
    wl = Workload("crowd", B, Hq, Hkv, D, T, 1, S, W, 1, seed=10)
    dq, dk, dv = decode_inputs(wl, 0, device="cuda")
    idx = torch.full((B, 1, top_k), -7, dtype=torch.int32, device="cuda")
    cache.decode_step_anchor(dq, dk, dv, torch.empty_like(dq), top_k, idx)
    torch.cuda.synchronize()
    sel = idx.cpu().numpy()[0, 0]
    kk = np.concatenate([f64(k[0]), f64(dk[0])[None]])
    imp = ohs.group_importance(f64(dq[0])[:g], kk[:, 0])
    _check_selection(sel, imp, top_k)
    # the tied positions are taken lowest first
    tied = sel[sel < T]
    assert np.array_equal(tied[: len(tied)], np.arange(len(tied))) or imp[T] < imp[0]


def test_anchor_selection_past_the_shared_memory_slices():
    """200K cached rows: each of a cluster's eight slices holds more rows
    than its CTA keeps in shared memory, so the rest of the importances go
    through global memory."""
    ensure_lib()
    B, Hq, Hkv, D, T, S, W, top_k, steps = 1, 8, 2, 128, 200000, 4, 64, 2048, 2
    labels = [0, 1]
    g = Hq // Hkv
    cache, k, v = _filled_cache(B, Hq, Hkv, D, T, S, W, labels, steps, 131)
    wl = Workload("long", B, Hq, Hkv, D, T, steps, S, W, 1, seed=13)
    kall = f64(k[0])
    for step in range(steps):
        dq, dk, dv = decode_inputs(wl, step, device="cuda")
        idx = torch.full((B, 1, top_k), -7, dtype=torch.int32, device="cuda")
        cache.decode_step_anchor(dq, dk, dv, torch.empty_like(dq), top_k, idx)
        torch.cuda.synchronize()
        kall = np.concatenate([kall, f64(dk[0])[None]])
        imp = ohs.group_importance(f64(dq[0])[:g], kall[:, 0])
        _check_selection(idx.cpu().numpy()[0, 0], imp, top_k)
    cache.close()


def test_anchor_selection_ties_across_slices_and_overflow():
    """180K identical keys: every cached row ties, and the top_k rows are
    the lowest positions, taken across several slices and past the rows a
    CTA keeps in shared memory."""
    ensure_lib()
    B, Hq, Hkv, D, T, S, W, top_k = 1, 8, 2, 128, 180000, 4, 64, 100000
    labels = [0, 1]
    g = Hq // Hkv
    cache = aoh.Cache(B, Hq, Hkv, D, T + 1, S, W, labels)
    k = randn_bf16((B, 1, Hkv, D), 141, "cuda").expand(B, T, Hkv, D).contiguous()
    v = randn_bf16((B, T, Hkv, D), 142, "cuda")
    cache.prefill(None, k, v, None)
    wl = Workload("ties", B, Hq, Hkv, D, T, 1, S, W, 1, seed=14)
    dq, dk, dv = decode_inputs(wl, 0, device="cuda")
    idx = torch.full((B, 1, top_k), -7, dtype=torch.int32, device="cuda")
    cache.decode_step_anchor(dq, dk, dv, torch.empty_like(dq), top_k, idx)
    torch.cuda.synchronize()
    sel = idx.cpu().numpy()[0, 0]
    kk = np.concatenate([f64(k[0]), f64(dk[0])[None]])
    imp = ohs.group_importance(f64(dq[0])[:g], kk[:, 0])
    _check_selection(sel, imp, top_k)
    tied = sel[sel < T]
    want = top_k if imp[T] < imp[0] else top_k - 1
    assert len(tied) == want and np.array_equal(tied, np.arange(want))
    cache.close()


def _reuse_case(B, Hq, Hkv, D, T, S, W, labels, top_k, n_anchor, group_map, steps=2, seed=41):
    ensure_lib()
    g = Hq // Hkv
    cache, k, v = _filled_cache(B, Hq, Hkv, D, T, S, W, labels, steps, seed)
    wl = Workload("reuse", B, Hq, Hkv, D, T, steps, S, W, sum(labels), seed=6)
    retr = [h for h in range(Hkv) if labels[h] == 0]
    rng = np.random.default_rng(seed)
    kall = [f64(k[b]) for b in range(B)]
    vall = [f64(v[b]) for b in range(B)]
    ktn = [k[b].cpu() for b in range(B)]
    vtn = [v[b].cpu() for b in range(B)]
    for step in range(steps):
        t = T + step                       # the new token's position
        lists = np.full((B, n_anchor, top_k), -1, dtype=np.int32)
        for b in range(B):
            for a in range(n_anchor):
                m = min(top_k, t + 1)
                pick = rng.choice(t + 1, size=m, replace=False)
                if a == 0 and m < t + 1:
                    pick[0] = t            # the new token among the borrowed rows
                    pick = np.unique(pick)
                    while len(pick) < m:
                        pick = np.unique(np.concatenate([pick, rng.choice(t, size=m - len(pick))]))
                lists[b, a, :m] = np.sort(pick)[:m]
        idx = torch.from_numpy(lists).cuda()
        dq, dk, dv = decode_inputs(wl, step, device="cuda")
        out = torch.full_like(dq, float("nan"))
        cache.decode_step_reuse(dq, dk, dv, out, idx, top_k, group_map)
        torch.cuda.synchronize()
        for b in range(B):
            kall[b] = np.concatenate([kall[b], f64(dk[b])[None]])
            vall[b] = np.concatenate([vall[b], f64(dv[b])[None]])
            ktn[b] = torch.cat([ktn[b], dk[b][None].cpu()])
            vtn[b] = torch.cat([vtn[b], dv[b][None].cpu()])
            qb = f64(dq[b])
            full = oatt.decode_step(qb, kall[b], vall[b], labels, S, W)
            fmag = oatt.decode_step(qb, kall[b], np.abs(vall[b]), labels, S, W)
            for kvh in range(Hkv):
                hs = slice(kvh * g, (kvh + 1) * g)
                if labels[kvh] == 0:
                    pos = lists[b, group_map[retr.index(kvh)]]
                    pos = pos[pos >= 0]
                    want = ohs.sparse_attend(qb[hs], kall[b][:, kvh], vall[b][:, kvh], pos)
                    mag = ohs.sparse_attend(qb[hs], kall[b][:, kvh], np.abs(vall[b][:, kvh]), pos)
                else:
                    want, mag = full[hs], fmag[hs]
                assert_matches(f64(out[b, hs]), want, f"reuse step {step} b={b} kv={kvh}", mag)
    cache.check()
    assert cache.lens() == [T + steps] * B
    kpad = torch.stack(ktn)
    vpad = torch.stack(vtn)
    check_cache_image(cache, kpad, vpad, [T + steps] * B, labels, S, W)
    cache.close()


@pytest.mark.parametrize("D,Hq,Hkv,labels,top_k,n_anchor,gmap", [
    (128, 8, 2, [0, 1], 200, 3, [2]),
    (128, 14, 2, [0, 0], 97, 2, [1, 0]),
    (128, 16, 4, [0, 1, 0, 0], 5000, 1, [0, 0, 0]),   # every row borrowed: a full decode
    (64, 16, 2, [1, 0], 33, 4, [3]),
    (128, 2, 2, [0, 1], 120, 2, [1]),            # groups of 1, gathered on the tensor cores
    (128, 32, 2, [0, 0], 300, 2, [1, 1]),        # groups of 16
    (128, 4, 2, [0, 1], 180, 2, [1]),            # groups of 2 (sixteen gather warps)
    (128, 6, 2, [1, 0], 260, 1, [0]),            # groups of 3
    (128, 10, 2, [0, 0], 150, 2, [0, 1]),        # groups of 5 (eight gather warps)
    (128, 16, 2, [0, 1], 400, 3, [2]),           # groups of 8
])
def test_reuse_step_attends_to_borrowed_rows(D, Hq, Hkv, labels, top_k, n_anchor, gmap):
    _reuse_case(2, Hq, Hkv, D, 900, 4, 50, labels, top_k, n_anchor, gmap)


@pytest.mark.parametrize("D,Hq,Hkv,labels", [
    (128, 8, 2, [0, 1]),       # tensor-core kernel, gathered rows
    (128, 14, 2, [0, 0]),
    (64, 8, 2, [1, 0]),        # CUDA-core kernel
])
def test_reuse_step_ragged_lengths(D, Hq, Hkv, labels):
    """Sequences of different lengths, so items of different sizes share the
    CTAs' weighted split; one list holds the new token, one sequence holds
    fewer rows than top_k."""
    ensure_lib()
    B, S, W, top_k = 3, 4, 40, 200
    lens = [300, 1100, 37]
    T = max(lens)
    g = Hq // Hkv
    retr = [h for h in range(Hkv) if labels[h] == 0]
    n_anchor = len(retr)
    cache = aoh.Cache(B, Hq, Hkv, D, T + 2, S, W, labels)
    k = randn_bf16((B, T, Hkv, D), 201, "cuda")
    v = randn_bf16((B, T, Hkv, D), 202, "cuda")
    cache.prefill(None, k, v, None, seq_lens=lens)
    wl = Workload("ragged-reuse", B, Hq, Hkv, D, T, 1, S, W, sum(labels), seed=12)
    dq, dk, dv = decode_inputs(wl, 0, device="cuda")
    rng = np.random.default_rng(5)
    lists = np.full((B, n_anchor, top_k), -1, dtype=np.int32)
    for b in range(B):
        t = lens[b]
        for a in range(n_anchor):
            m = min(top_k, t + 1)
            pick = np.sort(rng.choice(t + 1, size=m, replace=False))
            if b == 1 and a == 0 and t not in pick:
                pick[-1] = t               # the new token among the borrowed rows
            lists[b, a, :m] = np.sort(pick)
    out = torch.full_like(dq, float("nan"))
    gmap = list(range(n_anchor))[::-1]
    cache.decode_step_reuse(dq, dk, dv, out, torch.from_numpy(lists).cuda(), top_k, gmap)
    torch.cuda.synchronize()
    for b in range(B):
        t = lens[b]
        kk = np.concatenate([f64(k[b, :t]), f64(dk[b])[None]])
        vv = np.concatenate([f64(v[b, :t]), f64(dv[b])[None]])
        q = f64(dq[b])
        full = oatt.decode_step(q, kk, vv, labels, S, W)
        fmag = oatt.decode_step(q, kk, np.abs(vv), labels, S, W)
        for kvh in range(Hkv):
            hs = slice(kvh * g, (kvh + 1) * g)
            if labels[kvh] == 0:
                pos = lists[b, gmap[retr.index(kvh)]]
                pos = pos[pos >= 0]
                want = ohs.sparse_attend(q[hs], kk[:, kvh], vv[:, kvh], pos)
                mag = ohs.sparse_attend(q[hs], kk[:, kvh], np.abs(vv[:, kvh]), pos)
            else:
                want, mag = full[hs], fmag[hs]
            assert_matches(f64(out[b, hs]), want, f"ragged reuse b={b} kv={kvh}", mag)
    assert cache.lens() == [x + 1 for x in lens]
    cache.check()
    cache.close()


def test_anchor_then_reuse():
    """An anchor layer and a reuse layer of one block at the same step: the
    reuse layer attends to its own K/V at the positions the anchor chose."""
    ensure_lib()
    B, Hq, Hkv, D, T, S, W, top_k = 2, 8, 2, 128, 1200, 4, 64, 128
    labels = [0, 1]
    g = Hq // Hkv
    anchor, _, _ = _filled_cache(B, Hq, Hkv, D, T, S, W, labels, 1, 51)
    reuse, k, v = _filled_cache(B, Hq, Hkv, D, T, S, W, labels, 1, 61)
    wa = Workload("a", B, Hq, Hkv, D, T, 1, S, W, 1, seed=7)
    wr = Workload("r", B, Hq, Hkv, D, T, 1, S, W, 1, seed=8)
    qa, ka, va = decode_inputs(wa, 0, device="cuda")
    qr, kr, vr = decode_inputs(wr, 0, device="cuda")
    idx = torch.empty((B, 1, top_k), dtype=torch.int32, device="cuda")
    oa = torch.empty_like(qa)
    orr = torch.empty_like(qr)
    anchor.decode_step_anchor(qa, ka, va, oa, top_k, idx)
    reuse.decode_step_reuse(qr, kr, vr, orr, idx, top_k, [0])
    torch.cuda.synchronize()
    sel = idx.cpu().numpy()
    for b in range(B):
        kk = np.concatenate([f64(k[b]), f64(kr[b])[None]])
        vv = np.concatenate([f64(v[b]), f64(vr[b])[None]])
        q = f64(qr[b])
        want = ohs.sparse_attend(q[:g], kk[:, 0], vv[:, 0], sel[b, 0])
        mag = ohs.sparse_attend(q[:g], kk[:, 0], np.abs(vv[:, 0]), sel[b, 0])
        assert_matches(f64(orr[b, :g]), want, f"reuse after anchor b={b}", mag)
        full = oatt.decode_step(q, kk, vv, labels, S, W)
        fmag = oatt.decode_step(q, kk, np.abs(vv), labels, S, W)   # the bf16-P bound, as for every decode
        assert_matches(f64(orr[b, g:]), full[g:], f"reuse streaming b={b}", fmag[g:])
    anchor.close()
    reuse.close()


@pytest.mark.parametrize("D", [128, 64])
def test_reuse_step_without_retrieval_heads_is_a_decode_step(D):
    """All KV heads streaming: no list is borrowed, and the reuse step
    equals a plain decode step on an identical cache (bit for bit: the same
    kernel and split)."""
    ensure_lib()
    B, Hq, Hkv, T, S, W = 2, 8, 2, 300, 4, 50
    labels = [1, 1]
    c1, k, v = _filled_cache(B, Hq, Hkv, D, T, S, W, labels, 1, 91)
    c2 = aoh.Cache(B, Hq, Hkv, D, T + 1, S, W, labels)
    c2.prefill(None, k, v, None)
    wl = Workload("no-retrieval", B, Hq, Hkv, D, T, 1, S, W, 2, seed=13)
    dq, dk, dv = decode_inputs(wl, 0, device="cuda")
    o1, o2 = torch.empty_like(dq), torch.empty_like(dq)
    c1.decode_step_reuse(dq, dk, dv, o1, None, 16, [])
    c2.decode_step(dq, dk, dv, o2)
    torch.cuda.synchronize()
    assert torch.equal(o1, o2)
    for b in range(B):
        kk = np.concatenate([f64(k[b]), f64(dk[b])[None]])
        vv = np.concatenate([f64(v[b]), f64(dv[b])[None]])
        want = oatt.decode_step(f64(dq[b]), kk, vv, labels, S, W)
        mag = oatt.decode_step(f64(dq[b]), kk, np.abs(vv), labels, S, W)
        assert_matches(f64(o1[b]), want, f"no-retrieval reuse b={b}", mag)
    c1.close()
    c2.close()


def test_anchor_step_without_retrieval_heads_is_a_decode_step():
    ensure_lib()
    B, Hq, Hkv, D, T, S, W = 2, 8, 2, 128, 300, 4, 50
    labels = [1, 1]
    c1, k, v = _filled_cache(B, Hq, Hkv, D, T, S, W, labels, 1, 93)
    c2 = aoh.Cache(B, Hq, Hkv, D, T + 1, S, W, labels)
    c2.prefill(None, k, v, None)
    wl = Workload("no-retrieval-anchor", B, Hq, Hkv, D, T, 1, S, W, 2, seed=14)
    dq, dk, dv = decode_inputs(wl, 0, device="cuda")
    o1, o2 = torch.empty_like(dq), torch.empty_like(dq)
    c1.decode_step_anchor(dq, dk, dv, o1, 8, None)
    c2.decode_step(dq, dk, dv, o2)
    torch.cuda.synchronize()
    assert torch.equal(o1, o2)
    assert c1.lens() == c2.lens() == [T + 1] * B
    c1.close()
    c2.close()


def test_chunked_prefill_then_anchor_and_reuse():
    """A cache filled by two prefill chunks, then an anchor step and a reuse
    step (on a second layer's cache filled the same way) at the same
    position: the reuse output follows the anchor's selection."""
    ensure_lib()
    B, Hq, Hkv, D, S, W, top_k = 1, 8, 2, 128, 4, 64, 96
    labels = [0, 1]
    g = Hq // Hkv
    chunks = [700, 333]
    T = sum(chunks)
    caches, ks, vs = [], [], []
    for layer in range(2):
        cache = aoh.Cache(B, Hq, Hkv, D, T + 1, S, W, labels)
        k = randn_bf16((B, T, Hkv, D), 300 + 2 * layer, "cuda")
        v = randn_bf16((B, T, Hkv, D), 301 + 2 * layer, "cuda")
        q = randn_bf16((B, T, Hq, D), 350 + layer, "cuda")
        off = 0
        for c in chunks:
            out = torch.empty(B, c, Hq, D, dtype=torch.bfloat16, device="cuda")
            cache.prefill(q[:, off:off + c].contiguous(), k[:, off:off + c].contiguous(),
                          v[:, off:off + c].contiguous(), out)
            off += c
        caches.append(cache)
        ks.append(k)
        vs.append(v)
    wa = Workload("chunk-anchor", B, Hq, Hkv, D, T, 1, S, W, 1, seed=15)
    wr = Workload("chunk-reuse", B, Hq, Hkv, D, T, 1, S, W, 1, seed=16)
    qa, ka, va = decode_inputs(wa, 0, device="cuda")
    qr, kr, vr = decode_inputs(wr, 0, device="cuda")
    idx = torch.empty((B, 1, top_k), dtype=torch.int32, device="cuda")
    oa, orr = torch.empty_like(qa), torch.empty_like(qr)
    caches[0].decode_step_anchor(qa, ka, va, oa, top_k, idx)
    caches[1].decode_step_reuse(qr, kr, vr, orr, idx, top_k, [0])
    torch.cuda.synchronize()
    sel = idx.cpu().numpy()[0, 0]
    kk0 = np.concatenate([f64(ks[0][0]), f64(ka[0])[None]])
    _check_selection(sel, ohs.group_importance(f64(qa[0])[:g], kk0[:, 0]), top_k)
    kk = np.concatenate([f64(ks[1][0]), f64(kr[0])[None]])
    vv = np.concatenate([f64(vs[1][0]), f64(vr[0])[None]])
    q = f64(qr[0])
    want = ohs.sparse_attend(q[:g], kk[:, 0], vv[:, 0], sel)
    mag = ohs.sparse_attend(q[:g], kk[:, 0], np.abs(vv[:, 0]), sel)
    assert_matches(f64(orr[0, :g]), want, "reuse after chunked prefill", mag)
    for c in caches:
        c.check()
        c.close()


def test_reuse_rejects_bad_maps():
    ensure_lib()
    cache, _, _ = _filled_cache(1, 8, 2, 128, 64, 4, 16, [0, 1], 1, 71)
    q = torch.zeros(1, 8, 128, dtype=torch.bfloat16, device="cuda")
    kv = torch.zeros(1, 2, 128, dtype=torch.bfloat16, device="cuda")
    idx = torch.zeros((1, 2, 8), dtype=torch.int32, device="cuda")
    with pytest.raises(aoh.AohError) as e:
        cache.decode_step_reuse(q, kv, kv, torch.empty_like(q), idx, 8, [2])
    assert e.value.status == 1
    with pytest.raises(aoh.AohError) as e:
        cache.decode_step_anchor(q, kv, kv, torch.empty_like(q), 0, idx)
    assert e.value.status == 1
    assert cache.lens() == [64]
    cache.close()


def test_anchor_selection_splits_ties_at_the_threshold():
    """60 copies of one dominant key at random positions, top_k 30: the
    threshold is the copies' shared importance and exactly the 30 lowest
    copies are kept. The copies are few enough for the selection's fast
    path (their bucket's members go to one CTA) and spread over several
    CTAs and warps, which split the tied rows in position order."""
    ensure_lib()
    B, Hq, Hkv, D, T, S, W, top_k = 1, 8, 2, 128, 50000, 4, 64, 30
    labels = [0, 1]
    g = Hq // Hkv
    wl = Workload("split", B, Hq, Hkv, D, T, 1, S, W, 1, seed=15)
    dq, dk, dv = decode_inputs(wl, 0, device="cuda")
    k = randn_bf16((B, T, Hkv, D), 151, "cuda")
    v = randn_bf16((B, T, Hkv, D), 152, "cuda")
    # a key along the group's summed query direction scores far above the rest
    qs = dq[0, :g].float().sum(0)
    k0 = (qs / qs.norm() * 40.0).to(torch.bfloat16)
    gen = torch.Generator().manual_seed(16)
    copies = torch.randperm(T, generator=gen)[:60].sort().values
    k[0, copies.to("cuda"), 0] = k0
    cache = aoh.Cache(B, Hq, Hkv, D, T + 1, S, W, labels)
    cache.prefill(None, k, v, None)
    idx = torch.full((B, 1, top_k), -7, dtype=torch.int32, device="cuda")
    cache.decode_step_anchor(dq, dk, dv, torch.empty_like(dq), top_k, idx)
    torch.cuda.synchronize()
    sel = idx.cpu().numpy()[0, 0]
    kk = np.concatenate([f64(k[0]), f64(dk[0])[None]])
    imp = ohs.group_importance(f64(dq[0])[:g], kk[:, 0])
    _check_selection(sel, imp, top_k)
    assert np.array_equal(sel, copies.numpy()[:top_k]), (sel, copies.numpy()[:top_k])
    cache.close()
