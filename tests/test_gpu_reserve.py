"""After aoh_cache_init and aoh_cache_reserve, a serving loop's calls
allocate no device memory: a prefill of the longest chunk the cache can take
(its work list was sized at init) and H2Share anchor steps (workspace
reserved). Device memory is read with cudaMemGetInfo before and after; every
kernel is loaded first on a small cache of the same shape class, since the
first launch of a kernel loads its code (which takes device memory)."""

import pytest
import torch

from gpu_cases import ensure_lib
from paper_2608_06849_gb300 import aoh
from paper_2608_06849_gb300.workloads import Workload, decode_inputs, prefill_inputs

pytestmark = pytest.mark.gpu


def _steps(cache, wl, T, top_k, n_r):
    q, k, v = prefill_inputs(wl, device="cuda")
    out = torch.empty_like(q)
    dq, dk, dv = decode_inputs(wl, 0, device="cuda")
    dout = torch.empty_like(dq)
    idx = torch.empty((wl.batch, n_r, top_k), dtype=torch.int32, device="cuda")
    torch.cuda.synchronize()
    return (q, k, v, out), (dq, dk, dv, dout), idx


def test_reserved_handle_calls_allocate_nothing():
    ensure_lib()
    B, Hq, Hkv, D, S, W, labels, top_k = 2, 32, 8, 128, 64, 500, [1, 0, 0, 1, 1, 0, 0, 1], 256
    n_r = labels.count(0)
    # warm-up on a small cache: loads the prefill, append, decode and top-k kernels
    small = Workload("warm", B, Hq, Hkv, D, 300, 1, S, W, sum(labels), seed=8)
    wcache = aoh.Cache(B, Hq, Hkv, D, 302, S, W, labels)
    (q, k, v, out), (dq, dk, dv, dout), idx = _steps(wcache, small, 300, top_k, n_r)
    wcache.prefill(q, k, v, out)
    wcache.decode_step_anchor(dq, dk, dv, dout, top_k, idx)
    torch.cuda.synchronize()
    wcache.check()
    wcache.close()

    max_seq = 4097
    wl = Workload("reserve", B, Hq, Hkv, D, max_seq - 1, 1, S, W, sum(labels), seed=9)
    cache = aoh.Cache(B, Hq, Hkv, D, max_seq, S, W, labels)
    cache.reserve(max_seq, anchor_workspace=True)
    (q, k, v, out), (dq, dk, dv, dout), idx = _steps(cache, wl, max_seq - 1, top_k, n_r)
    free0, _ = torch.cuda.mem_get_info()
    cache.prefill(q, k, v, out)                     # the longest chunk this cache takes
    cache.decode_step_anchor(dq, dk, dv, dout, top_k, idx)
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    cache.check()
    assert cache.lens() == [max_seq] * B
    assert torch.isfinite(dout.float()).all()
    assert free1 == free0, f"device memory moved by {free0 - free1} bytes"
    cache.close()


def test_reserve_rejects_bad_arguments():
    ensure_lib()
    cache = aoh.Cache(1, 8, 2, 64, 100, 4, 8, [0, 1])
    with pytest.raises(aoh.AohError):
        cache.reserve(-1)
    with pytest.raises(aoh.AohError):            # the anchor step needs d_head 128
        cache.reserve(100, anchor_workspace=True)
    cache.reserve(100)
    cache.close()
