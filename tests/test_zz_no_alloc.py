"""The allocation-free decode entry point, checked against the handle API.

Some callers cannot allocate device memory once they are running (a server
whose memory arena is planned at start-up, a loop that cannot take
cudaMalloc's device-wide synchronisation). aoh_decode_step_noalloc serves
them: its scratch is a static device array inside the library and the caller
passes the KV buffer and the device lengths. This test drives it through the
C ABI for two calls in a row and compares each output with aoh_decode_step on
an identical cache, within the parity tolerance of the other GPU tests.
The file is named to be collected last."""

import pytest
import torch

from gpu_cases import MAX_ABS, MEAN_ABS, ensure_lib
from paper_2608_06849_gb300 import aoh
from paper_2608_06849_gb300.workloads import Workload, decode_inputs, randn_bf16

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("B,Hq,Hkv,D,T,S,W,labels", [
    (4, 32, 8, 128, 9000, 64, 1000, [1, 0, 0, 1, 1, 0, 0, 1]),
    (2, 8, 2, 64, 700, 16, 100, [0, 1]),
    (2, 28, 4, 128, 5000, 32, 700, [0, 1, 1, 0]),
])
def test_noalloc_decode_matches_handle_decode(B, Hq, Hkv, D, T, S, W, labels):
    ensure_lib()
    wl = Workload("noalloc", B, Hq, Hkv, D, T, 2, S, W, sum(labels), seed=3)
    cache = aoh.Cache(B, Hq, Hkv, D, T + 4, S, W, labels)
    k = randn_bf16((B, T, Hkv, D), 11, "cuda")
    v = randn_bf16((B, T, Hkv, D), 12, "cuda")
    cache.prefill(None, k, v, None)
    torch.cuda.synchronize()
    kv_copy = cache.buffer.clone()                       # identical cache for the no-alloc path
    lens = torch.full((B,), T, dtype=torch.int32, device="cuda")
    for step in range(2):
        q, kn, vn = decode_inputs(wl, step, device="cuda")
        out_ref = torch.full_like(q, float("nan"))
        out_na = torch.full_like(q, float("nan"))
        cache.decode_step(q, kn, vn, out_ref)
        aoh.aoh_decode_step_noalloc(cache.cfg, labels, kv_copy, lens, T + step, q, kn, vn, out_na)
        torch.cuda.synchronize()
        assert torch.isfinite(out_na.float()).all()
        err = (out_na.float() - out_ref.float()).abs()
        assert err.max().item() <= MAX_ABS, err.max().item()
        assert err.mean().item() <= MEAN_ABS, err.mean().item()
        assert lens.tolist() == [T + step + 1] * B
    cache.check()
    assert torch.equal(kv_copy, cache.buffer)            # the same rows were appended
    cache.close()
