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
