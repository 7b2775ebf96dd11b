"""Chunk-eviction rule for streaming heads in prefill (Sec. 5,
"Chunked-Prefill Stage": after each chunk of K tokens a streaming head keeps
only its sinks and the W most recent tokens). With aoh_config.chunk = K, a
prefill row at position i of chunk c = i // K sees keys j <= i with j < S
or j >= c*K - W. Each case is compared row by row with the oracle's
``prefill(..., chunk=K)``; decode steps that follow use the per-token rule
(oracle ``decode_step``); the cache image is checked bit-exactly."""

import numpy as np
import pytest
import torch

from gpu_cases import assert_matches, check_cache_image, ensure_lib, f64
from oracle import attention as oatt
from paper_2608_06849_gb300 import aoh
from paper_2608_06849_gb300.workloads import Workload, decode_inputs, randn_bf16

pytestmark = pytest.mark.gpu


def run_chunk_mode(Hq, Hkv, D, T, S, W, K, labels, calls, decode_steps=3, seed=21):
    """One sequence of T tokens prefilled in calls of the given lengths (each
    a multiple of K but the last), chunk = K; then decode steps."""
    ensure_lib()
    assert sum(calls) == T
    q = randn_bf16((1, T, Hq, D), seed + 1, "cuda")
    k = randn_bf16((1, T, Hkv, D), seed + 2, "cuda")
    v = randn_bf16((1, T, Hkv, D), seed + 3, "cuda")
    k[:, 0] *= 8
    cache = aoh.Cache(1, Hq, Hkv, D, T + decode_steps, S, W, labels, chunk=K)
    qn, kn, vn = f64(q[0]), f64(k[0]), f64(v[0])
    off = 0
    for n in calls:
        out = torch.full((1, n, Hq, D), float("nan"), dtype=torch.bfloat16, device="cuda")
        cache.prefill(q[:, off:off + n].contiguous(), k[:, off:off + n].contiguous(),
                      v[:, off:off + n].contiguous(), out)
        torch.cuda.synchronize()
        cache.check()
        rows = np.arange(off, off + n)
        L = off + n
        want = oatt.prefill(qn[:L], kn[:L], vn[:L], labels, S, W, rows=rows, chunk=K)
        mag = oatt.prefill(qn[:L], kn[:L], np.abs(vn[:L]), labels, S, W, rows=rows, chunk=K)
        assert_matches(f64(out[0]), want, f"chunk mode K={K} call at {off}", mag)
        off = L
    assert cache.lens() == [T]
    check_cache_image(cache, k, v, [T], labels, S, W)
    wl = Workload("chunk-mode", 1, Hq, Hkv, D, T, decode_steps, S, W, sum(labels), seed=seed)
    kall, vall = kn, vn
    for step in range(decode_steps):
        dq, dk, dv = decode_inputs(wl, step, device="cuda")
        dout = torch.empty_like(dq)
        cache.decode_step(dq, dk, dv, dout)
        torch.cuda.synchronize()
        kall = np.concatenate([kall, f64(dk[0])[None]])
        vall = np.concatenate([vall, f64(dv[0])[None]])
        want = oatt.decode_step(f64(dq[0]), kall, vall, labels, S, W)
        mag = oatt.decode_step(f64(dq[0]), kall, np.abs(vall), labels, S, W)
        assert_matches(f64(dout[0]), want, f"decode {step} after chunk mode", mag)
    cache.check()
    cache.close()


CASES = {
    # name: (Hq, Hkv, D, T, S, W, K, labels, calls)
    "k64_one_call": (8, 2, 128, 700, 4, 100, 64, [1, 0], [700]),
    "k100_one_call_unaligned_tiles": (8, 2, 128, 777, 16, 150, 100, [0, 1], [777]),
    "k256_one_call": (8, 2, 128, 900, 8, 300, 256, [1, 1], [900]),
    "k_beyond_prompt_is_causal": (4, 1, 128, 300, 2, 40, 512, [1], [300]),
    "k1_tokens": (4, 1, 128, 200, 3, 20, 1, [1], [200]),
    "calls_of_k_ring_wraps": (8, 2, 128, 640, 4, 60, 128, [1, 0], [128, 128, 256, 128]),
    "calls_of_k_small_window": (8, 2, 128, 600, 2, 16, 200, [1, 0], [200, 200, 200]),
    "group7_calls": (14, 2, 128, 512, 8, 130, 128, [0, 1], [256, 256]),
    "d64_calls": (8, 2, 64, 450, 4, 70, 150, [1, 0], [150, 300]),
}


@pytest.mark.parametrize("name", sorted(CASES))
def test_chunk_eviction_prefill(name):
    Hq, Hkv, D, T, S, W, K, labels, calls = CASES[name]
    run_chunk_mode(Hq, Hkv, D, T, S, W, K, labels, calls)


def test_call_off_a_chunk_boundary_is_refused():
    ensure_lib()
    K = 64
    cache = aoh.Cache(1, 8, 2, 128, 512, 4, 100, [1, 0], chunk=K)
    x = randn_bf16((1, 100, 8, 128), 3, "cuda")
    kv = randn_bf16((1, 100, 2, 128), 4, "cuda")
    cache.prefill(x, kv, kv)                     # 100 tokens: not a multiple of 64
    with pytest.raises(aoh.AohError) as e:
        cache.prefill(x, kv, kv)
    assert e.value.status == 1
    assert cache.lens() == [100]
    cache.close()
