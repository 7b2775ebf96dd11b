"""Chunked prefill (Sec. 5, "Chunked-Prefill Stage"): a sequence is
prefilled in several calls; each chunk's rows attend to the cached prefix
(retrieval: every earlier position; streaming: sinks + the window, read from
the sink and ring slots) and to the chunk itself. Each chunk's outputs are
checked against the oracle's rows of one prefill over the whole sequence;
the cache image is checked bit-exactly and decode steps follow."""

import numpy as np
import pytest
import torch

from gpu_cases import assert_matches, check_cache_image, ensure_lib, f64
from oracle import attention as oatt
from paper_2608_06849_gb300 import aoh
from paper_2608_06849_gb300.workloads import Workload, decode_inputs, randn_bf16

pytestmark = pytest.mark.gpu


def run_chunked(B, Hq, Hkv, D, chunk_lens, S, W, labels, decode_steps=2, seed=5):
    """chunk_lens: list over chunks of per-sequence lengths (lists of B ints)."""
    ensure_lib()
    totals = [sum(c[b] for c in chunk_lens) for b in range(B)]
    T = max(totals)
    q = randn_bf16((B, T, Hq, D), seed + 1, "cuda")
    k = randn_bf16((B, T, Hkv, D), seed + 2, "cuda")
    v = randn_bf16((B, T, Hkv, D), seed + 3, "cuda")
    k[:, 0] *= 8
    cache = aoh.Cache(B, Hq, Hkv, D, T + decode_steps, S, W, labels)
    qn, kn, vn = f64(q), f64(k), f64(v)
    off = [0] * B
    for ci, lens in enumerate(chunk_lens):
        Tc = max(lens)
        qc = torch.zeros(B, Tc, Hq, D, dtype=torch.bfloat16, device="cuda")
        kc = torch.zeros(B, Tc, Hkv, D, dtype=torch.bfloat16, device="cuda")
        vc = torch.zeros_like(kc)
        for b in range(B):
            qc[b, :lens[b]] = q[b, off[b]:off[b] + lens[b]]
            kc[b, :lens[b]] = k[b, off[b]:off[b] + lens[b]]
            vc[b, :lens[b]] = v[b, off[b]:off[b] + lens[b]]
        out = torch.full_like(qc, float("nan"))
        cache.prefill(qc, kc, vc, out, seq_lens=lens)
        torch.cuda.synchronize()
        cache.check()
        for b in range(B):
            rows = np.arange(off[b], off[b] + lens[b])
            L = off[b] + lens[b]
            want = oatt.prefill(qn[b, :L], kn[b, :L], vn[b, :L], labels, S, W, rows=rows)
            mag = oatt.prefill(qn[b, :L], kn[b, :L], np.abs(vn[b, :L]), labels, S, W, rows=rows)
            assert_matches(f64(out[b, :lens[b]]), want, f"chunk {ci} b={b}", mag)
            off[b] += lens[b]
    assert cache.lens() == totals
    check_cache_image(cache, k, v, totals, labels, S, W)
    wl = Workload("chunked", B, Hq, Hkv, D, T, decode_steps, S, W, sum(labels), seed=seed)
    kall = [kn[b, :totals[b]] for b in range(B)]
    vall = [vn[b, :totals[b]] for b in range(B)]
    for step in range(decode_steps):
        dq, dk, dv = decode_inputs(wl, step, device="cuda")
        dout = torch.empty_like(dq)
        cache.decode_step(dq, dk, dv, dout)
        torch.cuda.synchronize()
        for b in range(B):
            kall[b] = np.concatenate([kall[b], f64(dk[b])[None]])
            vall[b] = np.concatenate([vall[b], f64(dv[b])[None]])
            want = oatt.decode_step(f64(dq[b]), kall[b], vall[b], labels, S, W)
            mag = oatt.decode_step(f64(dq[b]), kall[b], np.abs(vall[b]), labels, S, W)
            assert_matches(f64(dout[b]), want, f"decode {step} b={b}", mag)
    cache.check()
    cache.close()


CASES = {
    # name: (B, Hq, Hkv, D, chunk_lens, S, W, labels)
    "ring_wraps_across_chunks": (1, 8, 2, 128, [[300], [200], [517]], 16, 100, [1, 0]),
    "sinks_span_chunks": (1, 8, 2, 128, [[64], [64], [64], [70]], 200, 50, [0, 1]),
    "window_not_full_yet": (1, 8, 2, 128, [[300], [300]], 4, 1000, [1, 1]),
    "no_sinks": (1, 4, 2, 128, [[129], [255], [1]], 0, 64, [1, 0]),
    "single_token_chunks": (1, 8, 2, 128, [[40]] + [[1]] * 5, 3, 17, [1, 0]),
    "group7_d128": (1, 14, 2, 128, [[257], [300]], 8, 130, [0, 1]),
    "d64": (1, 8, 2, 64, [[200], [333]], 16, 128, [1, 0]),
    # 24 sequences: the second chunk's 192 retrieval items, each reading its
    # sequence's 1024-token prefix, outnumber the SMs
    "many_sequences": (24, 8, 2, 128, [[1024] * 24, [512] * 24], 4, 64, [0, 1]),
    "ragged_two_seqs": (2, 8, 2, 128, [[300, 77], [100, 400], [260, 5]], 16, 128, [1, 0]),
    "window_equals_chunk": (1, 8, 2, 128, [[256], [256], [256]], 0, 256, [1, 1]),
}


@pytest.mark.parametrize("name", sorted(CASES))
def test_chunked_prefill(name):
    B, Hq, Hkv, D, chunks, S, W, labels = CASES[name]
    run_chunked(B, Hq, Hkv, D, chunks, S, W, labels)


def test_chunk_past_capacity_is_refused():
    ensure_lib()
    cache = aoh.Cache(1, 8, 2, 128, 300, 4, 16, [0, 1])
    k = randn_bf16((1, 200, 2, 128), 1, "cuda")
    q = randn_bf16((1, 200, 8, 128), 2, "cuda")
    cache.prefill(q, k, k, torch.empty_like(q))
    with pytest.raises(aoh.AohError) as e:
        cache.prefill(q, k, k, torch.empty_like(q))
    assert e.value.status == 2
    assert cache.lens() == [200]
    cache.close()


def test_nan_in_unwritten_cache_and_padding_is_ignored():
    """Cache rows not yet written and chunk rows past seq_lens are read by the
    tile copies but must not reach the outputs (a zero weight times NaN is
    NaN): fill both with NaN and check every output against the oracle."""
    ensure_lib()
    B, Hq, Hkv, D, S, W, labels = 2, 8, 2, 128, 16, 100, [1, 0]
    cache = aoh.Cache(B, Hq, Hkv, D, 600, S, W, labels)
    cache.buffer.fill_(0xFF)                      # every bf16 of the cache is NaN
    lens1, lens2 = [150, 77], [211, 300]
    T1, T2 = 256, 384
    q = randn_bf16((B, T1 + T2, Hq, D), 21, "cuda")
    k = randn_bf16((B, T1 + T2, Hkv, D), 22, "cuda")
    v = randn_bf16((B, T1 + T2, Hkv, D), 23, "cuda")
    qn, kn, vn = f64(q), f64(k), f64(v)
    off = [0, 0]
    for lens, Tc in [(lens1, T1), (lens2, T2)]:
        nan = float("nan")
        qc = torch.full((B, Tc, Hq, D), nan, dtype=torch.bfloat16, device="cuda")
        kc = torch.full((B, Tc, Hkv, D), nan, dtype=torch.bfloat16, device="cuda")
        vc = torch.full((B, Tc, Hkv, D), nan, dtype=torch.bfloat16, device="cuda")
        for b in range(B):
            qc[b, :lens[b]] = q[b, off[b]:off[b] + lens[b]]
            kc[b, :lens[b]] = k[b, off[b]:off[b] + lens[b]]
            vc[b, :lens[b]] = v[b, off[b]:off[b] + lens[b]]
        out = torch.zeros_like(qc)
        cache.prefill(qc, kc, vc, out, seq_lens=lens)
        torch.cuda.synchronize()
        for b in range(B):
            L = off[b] + lens[b]
            rows = np.arange(off[b], L)
            want = oatt.prefill(qn[b, :L], kn[b, :L], vn[b, :L], labels, S, W, rows=rows)
            mag = oatt.prefill(qn[b, :L], kn[b, :L], np.abs(vn[b, :L]), labels, S, W, rows=rows)
            assert_matches(f64(out[b, :lens[b]]), want, f"b={b}", mag)
            off[b] = L
    cache.check()
    cache.close()
