"""Failure detection without a GPU fault: every kernel's waits on mbarriers
are bounded by %globaltimer. The self-test makes one such wait run out (a
barrier that nothing arrives at, a 50 ms limit) and checks that the library
reports it, clears it, and keeps working."""

import time

import pytest
import torch

from gpu_cases import assert_matches, ensure_lib, f64
from oracle import attention as oatt
from paper_2608_06849_gb300 import aoh
from paper_2608_06849_gb300.workloads import Workload, decode_inputs, randn_bf16

pytestmark = pytest.mark.gpu


def test_bounded_wait_times_out_and_the_cache_stays_usable():
    ensure_lib()
    B, Hq, Hkv, D, T, S, W, labels = 1, 8, 2, 128, 300, 4, 40, [0, 1]
    cache = aoh.Cache(B, Hq, Hkv, D, T + 2, S, W, labels)
    k = randn_bf16((B, T, Hkv, D), 81, "cuda")
    v = randn_bf16((B, T, Hkv, D), 82, "cuda")
    cache.prefill(None, k, v, None)
    cache.check()
    limit = 50_000_000
    t0 = time.perf_counter()
    elapsed = aoh.aoh_cache_selftest_wait(cache.handle, limit)
    wall = time.perf_counter() - t0
    assert elapsed >= limit, elapsed
    assert elapsed < 20 * limit and wall < 5.0
    with pytest.raises(aoh.AohError) as e:
        cache.check()
    assert e.value.status == 4                    # AOH_ERR_TIMEOUT
    cache.check()                                 # reported once, then cleared
    # the context and the cache still work: a decode step against the oracle
    wl = Workload("after-timeout", B, Hq, Hkv, D, T, 1, S, W, 1, seed=9)
    dq, dk, dv = decode_inputs(wl, 0, device="cuda")
    out = torch.empty_like(dq)
    cache.decode_step(dq, dk, dv, out)
    torch.cuda.synchronize()
    cache.check()
    kk = torch.cat([k[0], dk[0][None]]).float().cpu().double().numpy()
    vv = torch.cat([v[0], dv[0][None]]).float().cpu().double().numpy()
    q = f64(dq[0])
    want = oatt.decode_step(q, kk, vv, labels, S, W)
    import numpy as np
    mag = oatt.decode_step(q, kk, np.abs(vv), labels, S, W)
    assert_matches(f64(out[0]), want, "decode after a timeout", mag)
    cache.close()


def test_selftest_rejects_limits_outside_the_range():
    ensure_lib()
    cache = aoh.Cache(1, 8, 2, 64, 16, 2, 4, [0, 1])
    for bad in (0, 999_999, 3_000_000_000):
        with pytest.raises(aoh.AohError) as e:
            aoh.aoh_cache_selftest_wait(cache.handle, bad)
        assert e.value.status == 1
    cache.close()
