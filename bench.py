"""Benchmark of the AoH attention path on GB300.

One "step" is one decode step of the Llama-3-8B-shaped decode workload
(32 query / 8 KV heads, d_head 128, batch 16, every sequence at 128K cached
tokens, 4 of 8 KV heads streaming with S=128, W=4096): the headline is
decode attention us/step and its HBM GB/s. The same run times the
Qwen2.5-7B-shaped 32K prefill (28 / 4 heads, 2 streaming, S=128, W=2048) for
prefill attention TFLOP/s, reported in the "prefill" object, and, with
short timed regions, the two other workloads: two layers of the 28-layer
Qwen2.5-7B-shaped stack at 256K (per-layer prefill and decode, KV bytes;
"stack_256k") and the 12-point ragged decode sweep ("ragged_sweep").

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl native|reference]

--impl reference times the CPU float64 oracle on a bounded sample of the
same decode step (no GPU needed). Multi-GPU runs (torchrun) are independent
replicas of the per-GPU workload (weak scaling, no collective on the data
path); rank 0 prints one JSON line.
"""

import argparse
import json
import math
import os
import platform
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "decode attn µs/step & HBM GB/s @128K ctx; prefill attn TFLOP/s @32K"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
NOMINAL_HBM_GBS = 7900.0  # GB300 HBM3e, nominal (context beside the measured copy rate)


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return d, "of measured"
    return dict(FALLBACK_PEAKS), "of fallback"


# ------------------------------------------------------------------ workload

def decode_workload(batch=None, ctx=None):
    import dataclasses

    from paper_2608_06849_gb300.workloads import DECODE_128K, labels_for
    wl = DECODE_128K
    if batch or ctx:
        wl = dataclasses.replace(wl, batch=batch or wl.batch, prefill_len=ctx or wl.prefill_len,
                                 name=f"{wl.name}-small")
    return wl, labels_for(wl)


def prefill_workload(T=None):
    import dataclasses

    from paper_2608_06849_gb300.workloads import PREFILL_32K, labels_for
    wl = PREFILL_32K
    if T:
        wl = dataclasses.replace(wl, prefill_len=T, name=f"{wl.name}-small")
    return wl, labels_for(wl)


def decode_bytes(lens_before, labels, wl):
    """Algorithmic HBM bytes of one decode step: cached K/V rows read once,
    the new token's K/V read and appended, q read, output written."""
    D, g = wl.d_head, wl.g
    row = D * 2
    total = 0
    for t in lens_before:
        for lab in labels:
            rows = (t + 1) if lab == 0 else min(t + 1, wl.sink + wl.window)
            total += (rows - 1) * row * 2          # cached K and V rows
            total += row * 2 * 2                   # new K/V read + appended
        total += wl.n_q_heads * D * 2 * 2          # q read + out written
    return total


def reuse_bytes(lens_before, labels, wl, top_k):
    """Algorithmic HBM bytes of one H2Share reuse step: min(top_k, t + 1)
    borrowed K/V rows per retrieval head, the ring rows of streaming heads,
    the new token's K/V read and appended, the index lists, q and out."""
    D = wl.d_head
    row = D * 2
    total = 0
    for t in lens_before:
        for lab in labels:
            rows = min(top_k, t + 1) if lab == 0 else min(t + 1, wl.sink + wl.window)
            total += (rows - 1) * row * 2 + row * 2 * 2
            if lab == 0:
                total += min(top_k, t + 1) * 4
        total += wl.n_q_heads * D * 2 * 2
    return total


def attended_pairs(T, S, W, streaming):
    """Number of (query, key) pairs a head attends in a causal prefill of T tokens."""
    if not streaming:
        return T * (T + 1) // 2
    i = list(range(T))
    tot = 0
    for x in i:
        sinks = min(x + 1, S)
        lo = max(S, x - W + 1)
        tot += sinks + max(0, x - lo + 1)
    return tot


def attended_pairs_chunk(T, S, W, K, streaming):
    """The same under the chunk-eviction rule: a streaming row x of chunk
    c = x // K sees the sinks and keys c*K - W .. x."""
    if not streaming:
        return T * (T + 1) // 2
    tot = 0
    for x in range(T):
        sinks = min(x + 1, S)
        lo = max(S, (x // K) * K - W, 0)
        tot += sinks + max(0, x - lo + 1)
    return tot


def prefill_flops(wl, labels, T, chunk=0):
    g = wl.g
    if chunk:
        pairs = sum(attended_pairs_chunk(T, wl.sink, wl.window, chunk, lab == 1) for lab in labels) * g
    else:
        pairs = sum(attended_pairs(T, wl.sink, wl.window, lab == 1) for lab in labels) * g
    return 4.0 * wl.d_head * pairs


# ------------------------------------------------------------------- clocks

class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index):
        self.proc = None
        self.out = os.path.join("/tmp", f"aoh_clocks_{os.getpid()}.csv")
        try:
            self.f = open(self.out, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                                          "-lms", "20", "-i", str(device_index)], stdout=self.f,
                                         stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.f.close()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.out):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx.append(float(parts[2]))
            except ValueError:
                continue
            for n, val in zip(names, parts[5:9]):
                if val.lower() == "active":
                    reasons.add(n)
        os.unlink(self.out)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "samples": len(sm),
                "reasons": sorted(reasons)}


# ------------------------------------------------------------------- ranks

class Ranks:
    """One process per GPU (torchrun env). The ranks run independent replicas
    of the per-GPU workload; nothing crosses ranks on the data path. The only
    collectives are the timing barrier and the max / sum over ranks."""

    def __init__(self, backend="nccl"):
        import torch.distributed as dist
        self.dist = dist
        self.world = int(os.environ.get("WORLD_SIZE", "1"))
        self.rank = int(os.environ.get("RANK", "0"))
        self.local = int(os.environ.get("LOCAL_RANK", "0"))
        self.backend = backend
        if self.world > 1 and not dist.is_initialized():
            dist.init_process_group(backend)

    def _device(self):
        return "cuda" if self.backend == "nccl" else "cpu"

    def barrier(self):
        import torch
        if self.world > 1:
            self.dist.barrier()
        if self.backend == "nccl":
            torch.cuda.synchronize()

    def _reduce(self, x, op):
        if self.world == 1:
            return float(x)
        import torch
        t = torch.tensor([float(x)], dtype=torch.float64, device=self._device())
        self.dist.all_reduce(t, op=op)
        return float(t.item())

    def max(self, x):
        return self._reduce(x, self.dist.ReduceOp.MAX)

    def sum(self, x):
        return self._reduce(x, self.dist.ReduceOp.SUM)


def replica_seed(base, rank):
    """Each rank's replica draws its own inputs."""
    return int(base) + 1000 * int(rank)


# -------------------------------------------------------------- native arm

def run_native(args):
    import torch

    from paper_2608_06849_gb300 import aoh
    from paper_2608_06849_gb300 import build as aoh_build
    from paper_2608_06849_gb300.workloads import decode_inputs, randn_bf16

    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    ranks = Ranks("nccl")
    world, rank = ranks.world, ranks.rank
    aoh_build.build()
    aoh.load()
    peaks, peak_note = load_peaks()
    barrier = ranks.barrier
    max_over_ranks = ranks.max

    stream = torch.cuda.current_stream()
    K, W = args.steps, args.warmup

    # ---------------- decode leg (headline)
    wl, labels = decode_workload(args.decode_batch, args.decode_ctx)
    B, D, T0 = wl.batch, wl.d_head, wl.prefill_len
    KH = min(K, 16)                                   # H2Share leg steps
    total_steps = W + K + K + 2 + 2 * (W + KH)         # warmup, timed, e2e, anchor, reuse
    cache = aoh.Cache(B, wl.n_q_heads, wl.n_kv_heads, D, T0 + total_steps + 8, wl.sink, wl.window, labels)
    kfill = randn_bf16((B, T0, wl.n_kv_heads, D), replica_seed(7001, rank), "cuda")
    vfill = randn_bf16((B, T0, wl.n_kv_heads, D), replica_seed(7002, rank), "cuda")
    cache.prefill(None, kfill, vfill, None)
    torch.cuda.synchronize()
    del kfill, vfill
    torch.cuda.empty_cache()
    inputs = [decode_inputs(wl, s, device="cuda") for s in range(W + K)]
    out = torch.empty(B, wl.n_q_heads, D, dtype=torch.bfloat16, device="cuda")
    for s in range(W):
        cache.decode_step(*inputs[s], out)
    cache.check()
    lens_before = cache.lens()
    step_bytes = []
    for s in range(K):
        step_bytes.append(decode_bytes([x + s for x in lens_before], labels, wl))
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(K + 1)]
    clocks = ClockSampler(local) if rank == 0 else None
    barrier()
    ev[0].record(stream)
    for s in range(K):
        cache.decode_step(*inputs[W + s], out)
        ev[s + 1].record(stream)
    barrier()
    per_step_ms = [ev[s].elapsed_time(ev[s + 1]) for s in range(K)]
    dec_ms = max_over_ranks(sum(per_step_ms))
    cache.check()
    dec_us_step = dec_ms * 1000.0 / K
    avg_bytes = sum(step_bytes) / K
    dec_gbs = avg_bytes / (dec_us_step * 1e-6) / 1e9          # per GPU (the roofline is per GPU)
    dec_gbs_total = ranks.sum(avg_bytes) / (dec_us_step * 1e-6) / 1e9

    # e2e: the same decode step through the public API, fed from pinned host
    # buffers: every step copies its q / k_new / v_new in and its output back
    # out. The copies run on a second stream with two device buffers each, so
    # the next step's input copy and this step's output copy overlap the
    # kernels; the timed region ends when the last output copy has landed.
    hq = [t.cpu().pin_memory() for t in inputs[W]]
    hout = [torch.empty(out.shape, dtype=out.dtype).pin_memory() for _ in range(2)]
    dq = [[torch.empty_like(t) for t in inputs[W]] for _ in range(2)]
    dout = [torch.empty_like(out) for _ in range(2)]
    h2d = sum(t.numel() * t.element_size() for t in hq)
    d2h = hout[0].numel() * hout[0].element_size()
    copy = torch.cuda.Stream()
    in_ready = [torch.cuda.Event() for _ in range(2)]
    done = [torch.cuda.Event() for _ in range(2)]
    out_read = [torch.cuda.Event() for _ in range(2)]
    barrier()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    copy.wait_stream(stream)
    with torch.cuda.stream(copy):
        for dst, src in zip(dq[0], hq):
            dst.copy_(src, non_blocking=True)
        in_ready[0].record(copy)
    for s in range(K):
        i = s & 1
        if s + 1 < K:
            with torch.cuda.stream(copy):
                if s >= 1:
                    copy.wait_event(done[1 - i])  # step s - 1 has read these inputs
                for dst, src in zip(dq[1 - i], hq):
                    dst.copy_(src, non_blocking=True)
                in_ready[1 - i].record(copy)
        stream.wait_event(in_ready[i])
        if s >= 2:
            stream.wait_event(out_read[i])  # step s - 2's output has been copied out
        cache.decode_step(dq[i][0], dq[i][1], dq[i][2], dout[i])
        done[i].record(stream)
        with torch.cuda.stream(copy):
            copy.wait_event(done[i])
            hout[i].copy_(dout[i], non_blocking=True)
            out_read[i].record(copy)
    stream.wait_stream(copy)
    e1.record(stream)
    barrier()
    e2e_us = max_over_ranks(e0.elapsed_time(e1)) * 1000.0 / K

    # ---------------- H2Share leg on the same cache: anchor steps (decode +
    # scores + top-k selection), then reuse steps over the borrowed positions
    top_k = args.h2_top_k
    retr = [h for h in range(wl.n_kv_heads) if labels[h] == 0]
    idx = torch.empty((B, len(retr), top_k), dtype=torch.int32, device="cuda")
    gmap = list(range(len(retr)))
    for s_ in range(W):
        cache.decode_step_anchor(*inputs[s_], out, top_k, idx)
    barrier()
    e0.record(stream)
    for s_ in range(KH):
        cache.decode_step_anchor(*inputs[W + s_], out, top_k, idx)
    e1.record(stream)
    barrier()
    anchor_us = max_over_ranks(e0.elapsed_time(e1)) * 1000.0 / KH
    for s_ in range(W):
        cache.decode_step_reuse(*inputs[s_], out, idx, top_k, gmap)
    cache.check()
    lens_r = cache.lens()
    barrier()
    e0.record(stream)
    for s_ in range(KH):
        cache.decode_step_reuse(*inputs[W + s_], out, idx, top_k, gmap)
    e1.record(stream)
    barrier()
    reuse_us = max_over_ranks(e0.elapsed_time(e1)) * 1000.0 / KH
    cache.check()
    r_bytes = sum(reuse_bytes([x + s_ for x in lens_r], labels, wl, top_k) for s_ in range(KH)) / KH
    h2 = {"top_k": top_k, "anchor_us_per_step": round(anchor_us, 2),
          "anchor_over_decode": round(anchor_us / dec_us_step, 4),
          "reuse_us_per_step": round(reuse_us, 2), "reuse_bytes_per_step": int(r_bytes),
          "reuse_hbm_gbs": round(r_bytes / (reuse_us * 1e-6) / 1e9, 1),
          "reuse_speedup_vs_decode": round(dec_us_step / reuse_us, 2),
          "note": "same cache and inputs as the decode leg; the reuse layer borrows the anchor's positions "
                  "(identity group map); top_k is a reading (the paper gives none)"}
    cache.close()
    del cache, inputs
    torch.cuda.empty_cache()

    # ---------------- prefill leg
    pwl, plabels = prefill_workload(args.prefill_len)
    from paper_2608_06849_gb300.workloads import prefill_inputs
    q, k, v = prefill_inputs(pwl, device="cuda")
    T = pwl.prefill_len
    pcache = aoh.Cache(1, pwl.n_q_heads, pwl.n_kv_heads, pwl.d_head, T, pwl.sink, pwl.window, plabels)
    pout = torch.empty_like(q)
    Kp = max(3, min(K, args.prefill_steps))
    for _ in range(max(W, 3)):
        pcache.reset()
        pcache.prefill(q, k, v, pout)
    pcache.check()
    pev = [torch.cuda.Event(enable_timing=True) for _ in range(Kp + 1)]
    barrier()
    pev[0].record(stream)
    for s in range(Kp):
        pcache.reset()
        pcache.prefill(q, k, v, pout)
        pev[s + 1].record(stream)
    barrier()
    pre_ms = max_over_ranks(pev[0].elapsed_time(pev[Kp])) / Kp
    pcache.check()
    flops = prefill_flops(pwl, plabels, T)
    pre_tflops = flops / (pre_ms * 1e-3) / 1e12
    pre_tflops_total = ranks.sum(flops) / (pre_ms * 1e-3) / 1e12
    pcache.close()

    # ---------------- chunked prefill leg: the same 32K prefill in chunks
    n_chunks = args.prefill_chunks
    C = T // n_chunks
    chunks = [(q[:, i * C:(i + 1) * C].contiguous(), k[:, i * C:(i + 1) * C].contiguous(),
               v[:, i * C:(i + 1) * C].contiguous()) for i in range(n_chunks)]
    couts = [torch.empty_like(ch[0]) for ch in chunks]
    ccache = aoh.Cache(1, pwl.n_q_heads, pwl.n_kv_heads, pwl.d_head, T, pwl.sink, pwl.window, plabels)
    for _ in range(max(W, 3)):
        ccache.reset()
        for ch, co in zip(chunks, couts):
            ccache.prefill(ch[0], ch[1], ch[2], co)
    ccache.check()
    cev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    barrier()
    cev[0].record(stream)
    for _ in range(Kp):
        ccache.reset()
        for ch, co in zip(chunks, couts):
            ccache.prefill(ch[0], ch[1], ch[2], co)
    cev[1].record(stream)
    barrier()
    chunk_ms = max_over_ranks(cev[0].elapsed_time(cev[1])) / Kp
    ccache.check()
    ccache.close()

    # ---------------- the same chunks under the chunk-eviction rule (chunk = C):
    # streaming rows see the sinks, the W tokens before their chunk and the chunk
    ecache = aoh.Cache(1, pwl.n_q_heads, pwl.n_kv_heads, pwl.d_head, T, pwl.sink, pwl.window, plabels, chunk=C)
    for _ in range(max(W, 3)):
        ecache.reset()
        for ch, co in zip(chunks, couts):
            ecache.prefill(ch[0], ch[1], ch[2], co)
    ecache.check()
    barrier()
    cev[0].record(stream)
    for _ in range(Kp):
        ecache.reset()
        for ch, co in zip(chunks, couts):
            ecache.prefill(ch[0], ch[1], ch[2], co)
    cev[1].record(stream)
    barrier()
    evict_ms = max_over_ranks(cev[0].elapsed_time(cev[1])) / Kp
    ecache.check()
    ecache.close()
    evict_flops = prefill_flops(pwl, plabels, T, chunk=C)
    del chunks, couts

    # ---------------- the other two workloads: the 256K stack (two layers) and
    # the ragged decode sweep, with short timed regions
    hbm_peak = float(peaks.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"]))
    tf_peak = float(peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"]))
    stack = ragged = None
    if not args.no_extra_workloads:
        del q, k, v
        torch.cuda.empty_cache()
        barrier()
        stack = stack_leg(aoh, torch, args.extra_steps, W, args.stack_layers, 2, tf_peak, hbm_peak)
        barrier()
        ragged = ragged_leg(aoh, torch, args.extra_steps, W, hbm_peak)
        barrier()
    clock_info = clocks.stop() if clocks else None

    # ---------------- cpu baseline (oracle on a bounded sample), rank 0 only
    cpu = pcpu = None
    if rank == 0 and not args.no_cpu_baseline:
        cpu = oracle_decode_sample(args.cpu_seconds)
        pcpu = oracle_prefill_sample(min(10.0, args.cpu_seconds))

    if rank != 0:
        return
    line = {
        "metric": METRIC,
        "value": round(dec_us_step, 3),
        "unit": "us/step",
        "n_gpus": world,
        "steps": K,
        "warmup": W,
        "ms_per_step": round(dec_us_step / 1000.0, 6),
        "higher_is_better": False,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic",
        "config": {
            "workload": f"{wl.name}: B={B} Hq={wl.n_q_heads} Hkv={wl.n_kv_heads} d={D} ctx={T0} "
                        f"streaming={sum(labels)}/{len(labels)} S={wl.sink} W={wl.window}",
            "prefill_workload": f"{pwl.name}: T={T} Hq={pwl.n_q_heads} Hkv={pwl.n_kv_heads} d={pwl.d_head} "
                                f"streaming={sum(plabels)}/{len(plabels)} S={pwl.sink} W={pwl.window}",
            "l2": "inputs larger than L2 (decode reads a 4.4 GB cache per step; prefill q/k/v 302 MB)",
            "parallelism": f"replicas x{world}",
        },
        "decode": {"us_per_step": round(dec_us_step, 3), "hbm_gbs": round(dec_gbs, 1),
                   "hbm_gbs_all_ranks": round(dec_gbs_total, 1),
                   "bytes_per_step": int(avg_bytes), "kernel_us_median": round(statistics.median(per_step_ms) * 1000, 3)},
        "roofline": {"bound": "hbm", "achieved": round(dec_gbs, 1), "peak": hbm_peak, "unit": "GB/s",
                     "frac": round(dec_gbs / hbm_peak, 4), "traffic": traffic_for(decode_kernel_key(wl)),
                     "peak_note": f"peak = {peak_note} HBM copy bandwidth (a read+write copy; decode only reads, "
                                  f"so frac is a ratio to the measured copy rate and may pass 1); kernel: "
                                  + decode_kernel_name(wl),
                     "nominal_peak": NOMINAL_HBM_GBS,
                     "frac_of_nominal": round(dec_gbs / NOMINAL_HBM_GBS, 4)},
        "prefill": {"ms": round(pre_ms, 3), "tflops": round(pre_tflops, 2), "flops": flops, "steps": Kp,
                    "tflops_all_ranks": round(pre_tflops_total, 2),
                    "roofline": {"bound": "tensor", "achieved": round(pre_tflops, 2), "peak": tf_peak,
                                 "unit": "TFLOP/s", "frac": round(pre_tflops / tf_peak, 4),
                                 "traffic": traffic_for("prefill"),
                                 "peak_note": f"{peak_note} dense bf16 (burst); time includes the cache append"},
                    "cpu_baseline": pcpu},
        "chunked_prefill": {"chunks": n_chunks, "chunk_tokens": C, "ms": round(chunk_ms, 3),
                            "tflops": round(flops / (chunk_ms * 1e-3) / 1e12, 2),
                            "frac": round(flops / (chunk_ms * 1e-3) / 1e12 / tf_peak, 4),
                            "note": "same 32K prefill as consecutive chunks; each chunk reads the cached prefix"},
        "chunk_eviction_prefill": {"chunk": C, "ms": round(evict_ms, 3), "flops": evict_flops,
                                   "tflops": round(evict_flops / (evict_ms * 1e-3) / 1e12, 2),
                                   "frac": round(evict_flops / (evict_ms * 1e-3) / 1e12 / tf_peak, 4),
                                   "note": "the same chunks with aoh_config.chunk = C: streaming rows see the sinks, "
                                           "the W tokens before their chunk and the chunk (attended pairs counted "
                                           "under that rule)"},
        "h2share": dict(h2, reuse_frac_of_peak=round(h2["reuse_hbm_gbs"] / hbm_peak, 4)),
        "stack_256k": stack,
        "ragged_sweep": ragged,
        "e2e": {"value": round(e2e_us, 3), "unit": "us/step", "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
        "gpu_launches": K,
        "clocks": clock_info,
        "cpu_baseline": cpu,
    }
    print(json.dumps(line))


def decode_kernel_key(wl):
    """Which decode kernel serves this shape (the library's dispatch: d_head
    128 runs on the tensor cores, d_head 64 on CUDA cores)."""
    return "decode_tc" if wl.d_head == 128 else "decode"


def decode_kernel_name(wl):
    g = wl.n_q_heads // wl.n_kv_heads
    if wl.d_head == 128:
        return f"decode_tc_kernel<{g}> (tcgen05 split-KV)"
    return f"decode_kernel<DecodeCfg<64,{g}>> (CUDA-core split-KV)"


def traffic_for(kernel):
    """DRAM bytes per launch from the committed ncu summary, if it was taken
    on the current kernel source (else null)."""
    p = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(p):
        return None
    try:
        d = json.load(open(p)).get(kernel)
        if not d:
            return None
        from paper_2608_06849_gb300.build import kernel_digest
        if d.get("kernel_digest") != kernel_digest(kernel):
            return None
        return d.get("bytes_per_launch")
    except Exception:
        return None


# ---------------------------------------------------------- reference arm

class OracleDecodeSample:
    """The float64 oracle on one sequence's decode step at 128K context, for
    one retrieval and one streaming KV head group; scaled to the full step
    (16 sequences x 4 retrieval + 4 streaming groups, one pair per scale unit)."""

    def __init__(self):
        import numpy as np

        from paper_2608_06849_gb300.workloads import randn_bf16

        self.wl, self.labels = decode_workload()
        D, g, T = self.wl.d_head, self.wl.g, self.wl.prefill_len
        self.k = randn_bf16((T + 1, 2, D), 9001).float().numpy().astype(np.float64)
        self.v = randn_bf16((T + 1, 2, D), 9002).float().numpy().astype(np.float64)
        self.q = randn_bf16((2 * g, D), 9003).float().numpy().astype(np.float64)
        n_r = len(self.labels) - sum(self.labels)
        assert n_r == sum(self.labels)
        self.scale = self.wl.batch * n_r

    def step_us(self):
        from oracle import attention as oatt
        t0 = time.perf_counter()
        oatt.decode_step(self.q, self.k, self.v, [0, 1], self.wl.sink, self.wl.window)
        return (time.perf_counter() - t0) * 1e6 * self.scale

    def describe(self, reps):
        return (f"float64 oracle, 1 of {self.wl.batch} sequences x (1 retrieval + 1 streaming) of "
                f"{len(self.labels)} KV head groups at ctx {self.wl.prefill_len}, median of {reps} reps, "
                f"scaled x{self.scale}; numpy default BLAS threading")


def oracle_prefill_sample(budget_s=10.0, wl=None, labels=None):
    """The float64 oracle on seeded random query rows of a prefill (all query
    heads, the workload's labels; the 32K prefill by default), until about
    budget_s has passed, extrapolated to the whole prefill by attended
    (query, key) pairs."""
    import numpy as np

    from oracle import attention as oatt
    from paper_2608_06849_gb300.workloads import randn_bf16
    if wl is None:
        wl, labels = prefill_workload()
    T, D, S, W, g = wl.prefill_len, wl.d_head, wl.sink, wl.window, wl.g
    k = randn_bf16((T, wl.n_kv_heads, D), 9101).float().numpy().astype(np.float64)
    v = randn_bf16((T, wl.n_kv_heads, D), 9102).float().numpy().astype(np.float64)
    rng = np.random.default_rng(9103)

    def pairs(i):
        tot = 0
        for lab in labels:
            if lab == 0:
                tot += i + 1
            else:
                tot += min(i + 1, S) + max(0, i - max(S, i - W + 1) + 1)
        return tot * g

    spent, done_pairs, n_rows = 0.0, 0, 0
    while spent < budget_s:
        rows = np.sort(rng.choice(T, size=8, replace=False))
        q = randn_bf16((8, wl.n_q_heads, D), 9104 + n_rows).float().numpy().astype(np.float64)
        t0 = time.perf_counter()
        oatt.attend(q, rows, k, v, labels, S, W)
        spent += time.perf_counter() - t0
        done_pairs += sum(pairs(int(i)) for i in rows)
        n_rows += 8
    total_pairs = prefill_flops(wl, labels, T) / (4.0 * D)
    ms = spent / done_pairs * total_pairs * 1e3
    return {"value": round(ms, 1), "unit": "ms/prefill", "cores": os.cpu_count(), "kind": "oracle",
            "sample": f"float64 oracle on {n_rows} random query rows (all {wl.n_q_heads} heads) of the {T}-token "
                      f"prefill, {spent:.1f} s, extrapolated by attended (query, key) pairs "
                      f"({done_pairs} of {int(total_pairs)})", **host_cpu()}


def oracle_decode_layer(wl, labels, lens, budget_s=5.0, max_seqs=4):
    """The float64 oracle on one layer's decode step (all heads) for up to
    max_seqs of the batch's sequences at their lengths, repeated for about
    budget_s; the median scaled to the whole batch by rows attended."""
    import numpy as np

    from oracle import attention as oatt
    from paper_2608_06849_gb300.workloads import randn_bf16
    D, S, W = wl.d_head, wl.sink, wl.window

    def rows(t):
        return sum((t + 1) if lab == 0 else min(t + 1, S + W) for lab in labels)

    sample = list(lens[:max_seqs])
    data = []
    for i, t in enumerate(sample):
        k = randn_bf16((t + 1, wl.n_kv_heads, D), 9201 + 3 * i).float().numpy().astype(np.float64)
        v = randn_bf16((t + 1, wl.n_kv_heads, D), 9202 + 3 * i).float().numpy().astype(np.float64)
        q = randn_bf16((wl.n_q_heads, D), 9203 + 3 * i).float().numpy().astype(np.float64)
        data.append((q, k, v))
    vals = []
    t0 = time.perf_counter()
    while not vals or time.perf_counter() - t0 < budget_s:
        a = time.perf_counter()
        for q, k, v in data:
            oatt.decode_step(q, k, v, labels, S, W)
        vals.append(time.perf_counter() - a)
    scale = sum(rows(t) for t in lens) / sum(rows(t) for t in sample)
    return {"value": round(statistics.median(vals) * scale * 1e6, 1), "unit": "us/step", "cores": os.cpu_count(),
            "kind": "oracle", "sample": f"float64 oracle decode step on {len(sample)} of {len(lens)} sequences "
                                        f"(all heads), median of {len(vals)} reps, scaled x{scale:.2f} by rows "
                                        f"attended", **host_cpu()}


def host_cpu():
    """The host CPU as the kernel reports it, and the BLAS threads numpy may use."""
    model = platform.machine()
    try:
        with open("/proc/cpuinfo") as f:
            for line in f:
                key = line.split(":")[0].strip().lower()
                if key in ("model name", "cpu part"):
                    val = line.split(":", 1)[1].strip()
                    # Arm reports a part number; 0xd4f is the Neoverse V2 (Grace)
                    model += " " + {"0xd4f": "Neoverse-V2 (0xd4f)"}.get(val, val)
                    break
    except OSError:
        pass
    threads = os.environ.get("OMP_NUM_THREADS") or os.environ.get("OPENBLAS_NUM_THREADS") or "default (one per core)"
    return {"cpu": model, "blas_threads": threads}


def oracle_decode_sample(budget_s=15.0):
    s = OracleDecodeSample()
    s.step_us()
    vals = []
    t0 = time.perf_counter()
    while not vals or time.perf_counter() - t0 < budget_s:
        vals.append(s.step_us())
    return {"value": round(statistics.median(vals), 1), "unit": "us/step", "cores": os.cpu_count(),
            "kind": "oracle", "sample": s.describe(len(vals)), **host_cpu()}


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    s = OracleDecodeSample()
    for _ in range(args.warmup):
        s.step_us()
    vals = [s.step_us() for _ in range(args.steps)]
    value = sum(vals) / len(vals)
    wl, labels = s.wl, s.labels
    line = {
        "impl": "reference",
        "metric": METRIC,
        "value": round(value, 1),
        "unit": "us/step",
        "n_gpus": int(os.environ.get("WORLD_SIZE", "1")),
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(value / 1000.0, 3),
        "higher_is_better": False,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "f64",
        "data": "synthetic",
        "config": {"workload": f"{wl.name}: B={wl.batch} Hq={wl.n_q_heads} Hkv={wl.n_kv_heads} d={wl.d_head} "
                               f"ctx={wl.prefill_len} streaming={sum(labels)}/{len(labels)} S={wl.sink} W={wl.window}"},
        "cpu_baseline": {"value": round(value, 1), "unit": "us/step", "cores": os.cpu_count(), "kind": "oracle",
                         "sample": s.describe(len(vals)), **host_cpu()},
        "e2e": {"value": round(value, 1), "unit": "us/step", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))


# ------------------------------------------------------- other workloads

def _decode_timing(aoh, torch, cache, wl, steps, warmup):
    from paper_2608_06849_gb300.workloads import decode_inputs
    inputs = [decode_inputs(wl, s, device="cuda") for s in range(warmup + steps)]
    out = torch.empty(wl.batch, wl.n_q_heads, wl.d_head, dtype=torch.bfloat16, device="cuda")
    for s in range(warmup):
        cache.decode_step(*inputs[s], out)
    cache.check()
    before = cache.lens()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    e0.record()
    for s in range(steps):
        cache.decode_step(*inputs[warmup + s], out)
    e1.record()
    torch.cuda.synchronize()
    cache.check()
    return e0.elapsed_time(e1) * 1000.0 / steps, before


def ragged_leg(aoh, torch, steps, warmup, hbm):
    """Decode of 64 sequences with lengths uniform in [4K, 32K], S = 64, over
    the sweep of streaming fraction x window: one entry per point, with the
    HBM fraction of its algorithmic bytes."""
    import dataclasses

    from paper_2608_06849_gb300.workloads import RAGGED, labels_for, randn_bf16, seq_lens
    lens = seq_lens(RAGGED)
    T = max(lens)
    B, Hkv, D = RAGGED.batch, RAGGED.n_kv_heads, RAGGED.d_head
    kfill = randn_bf16((B, T, Hkv, D), 7101, "cuda")
    vfill = randn_bf16((B, T, Hkv, D), 7102, "cuda")
    points = []
    for frac in (0.0, 0.25, 0.5, 0.75):
        for W in (512, 2048, 8192):
            wl = dataclasses.replace(RAGGED, n_streaming=int(frac * Hkv), window=W)
            labels = labels_for(wl)
            cache = aoh.Cache(B, wl.n_q_heads, Hkv, D, T + steps + warmup + 4, wl.sink, W, labels)
            cache.prefill(None, kfill, vfill, None, seq_lens=lens)
            us, before = _decode_timing(aoh, torch, cache, wl, steps, warmup)
            nbytes = decode_bytes(before, labels, wl)
            points.append({"streaming_frac": frac, "window": W, "us_per_step": round(us, 2),
                           "bytes_per_step": nbytes, "hbm_gbs": round(nbytes / (us * 1e-6) / 1e9, 1),
                           "frac_of_peak": round(nbytes / (us * 1e-6) / 1e9 / hbm, 4)})
            cache.close()
    del kfill, vfill
    torch.cuda.empty_cache()
    return {"workload": f"{RAGGED.name}: B={B} Hq={RAGGED.n_q_heads} Hkv={Hkv} d={D} "
                        f"lens uniform [4096, 32768] seed {RAGGED.seed} S={RAGGED.sink}",
            "steps": steps, "warmup": warmup, "peak_hbm_gbs": hbm, "sweep": points,
            "frac_range": [min(p["frac_of_peak"] for p in points), max(p["frac_of_peak"] for p in points)]}


def run_ragged(args):
    """The ragged sweep alone (one JSON line), with the oracle's time on one
    sweep point."""
    import dataclasses

    import torch

    from paper_2608_06849_gb300 import aoh
    from paper_2608_06849_gb300 import build as aoh_build
    from paper_2608_06849_gb300.workloads import RAGGED, labels_for, seq_lens
    aoh_build.build()
    aoh.load()
    peaks, note = load_peaks()
    hbm = float(peaks.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"]))
    res = ragged_leg(aoh, torch, args.steps, args.warmup, hbm)
    res.update({"metric": "decode attn us/step and HBM GB/s", "peak_note": note})
    half = dataclasses.replace(RAGGED, n_streaming=RAGGED.n_kv_heads // 2, window=2048)
    res["cpu_baseline"] = None if args.no_cpu_baseline else dict(
        oracle_decode_layer(half, labels_for(half), seq_lens(RAGGED), budget_s=5.0),
        point="streaming_frac 0.5, window 2048")
    print(json.dumps(res))


def stack_leg(aoh, torch, steps, warmup, layers, prefill_reps, tf_peak, hbm, cpu=False):
    """Layers of the 28-layer Qwen2.5-7B-shaped stack at 256K (each layer its
    own labels and inputs): per layer, the 256K prefill and `steps` decode
    steps after it; the whole stack's KV bytes against the all-retrieval
    layout. Per-layer figures with their roofline fractions."""
    from paper_2608_06849_gb300.workloads import STACK_256K, labels_for, prefill_inputs
    wl = STACK_256K
    T = wl.prefill_len
    per_layer = []
    cpu_base = None
    for layer in range(layers):
        labels = labels_for(wl, layer=layer)
        q, k, v = prefill_inputs(wl, device="cuda", seed_offset=layer)
        cache = aoh.Cache(1, wl.n_q_heads, wl.n_kv_heads, wl.d_head, T + steps + warmup + 4, wl.sink, wl.window,
                          labels)
        out = torch.empty_like(q)
        cache.reset()
        cache.prefill(q, k, v, out)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        e0.record()
        for _ in range(prefill_reps):
            cache.reset()
            cache.prefill(q, k, v, out)
        e1.record()
        torch.cuda.synchronize()
        cache.check()
        pre_ms = e0.elapsed_time(e1) / prefill_reps
        flops = prefill_flops(wl, labels, T)
        del q, out, k, v
        us, before = _decode_timing(aoh, torch, cache, wl, steps, warmup)
        nbytes = decode_bytes(before, labels, wl)
        cache.close()
        torch.cuda.empty_cache()
        per_layer.append({"layer": layer, "labels": labels, "prefill_ms": round(pre_ms, 3),
                          "prefill_tflops": round(flops / (pre_ms * 1e-3) / 1e12, 1),
                          "prefill_frac_of_peak": round(flops / (pre_ms * 1e-3) / 1e12 / tf_peak, 4),
                          "decode_us_per_step": round(us, 2), "decode_bytes_per_step": nbytes,
                          "decode_hbm_gbs": round(nbytes / (us * 1e-6) / 1e9, 1),
                          "decode_frac_of_peak": round(nbytes / (us * 1e-6) / 1e9 / hbm, 4)})
        if cpu and layer == 0:
            cpu_base = {"decode": oracle_decode_layer(wl, labels, before, budget_s=5.0),
                        "prefill": oracle_prefill_sample(8.0, wl, labels)}
    cfg = aoh.make_config(1, wl.n_q_heads, wl.n_kv_heads, wl.d_head, T + wl.decode_steps, wl.sink, wl.window)
    kv_aoh = sum(aoh.aoh_cache_bytes(cfg, labels_for(wl, layer=L)) for L in range(wl.layers))
    kv_full = wl.layers * aoh.aoh_cache_bytes(cfg, [0] * wl.n_kv_heads)
    n = len(per_layer)
    pre_ms = sum(x["prefill_ms"] for x in per_layer) / n
    dec_us = sum(x["decode_us_per_step"] for x in per_layer) / n
    res = {
        "workload": f"{wl.name}: {wl.layers} layers x (Hq={wl.n_q_heads} Hkv={wl.n_kv_heads} d={wl.d_head}), "
                    f"T={T} (+{wl.decode_steps} decode), 2 of 4 KV heads streaming per layer, S={wl.sink} "
                    f"W={wl.window}; {n} layers timed",
        "layers_timed": per_layer, "prefill_reps": prefill_reps, "decode_steps": steps, "decode_warmup": warmup,
        "prefill_ms_per_layer": round(pre_ms, 3),
        "prefill_frac_of_peak": round(sum(x["prefill_frac_of_peak"] for x in per_layer) / n, 4),
        "decode_us_per_layer_step": round(dec_us, 2),
        "decode_frac_of_peak": round(sum(x["decode_frac_of_peak"] for x in per_layer) / n, 4),
        "stack_estimate": {"prefill_s": round(wl.layers * pre_ms / 1000, 3),
                           "decode_ms_per_token": round(wl.layers * dec_us / 1000, 3)},
        "kv_bytes_stack": kv_aoh, "kv_bytes_all_retrieval": kv_full, "kv_ratio": round(kv_full / kv_aoh, 4),
        "peaks": {"bf16_tflops": tf_peak, "hbm_gbs": hbm}}
    if cpu_base is not None:
        res["cpu_baseline"] = cpu_base
    return res


def run_stack(args):
    """The 256K stack alone (one JSON line), with the oracle's time on layer 0."""
    import torch

    from paper_2608_06849_gb300 import aoh
    from paper_2608_06849_gb300 import build as aoh_build
    aoh_build.build()
    aoh.load()
    peaks, note = load_peaks()
    tf_peak = float(peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"]))
    hbm = float(peaks.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"]))
    res = stack_leg(aoh, torch, args.steps, args.warmup, args.stack_layers, 3, tf_peak, hbm,
                    cpu=not args.no_cpu_baseline)
    res["peak_note"] = note
    print(json.dumps(res))


def run_graph(args):
    """Batch-1 decode latency per token through a whole Qwen2.5-7B-shaped
    model (28 layers of 28 query / 4 KV heads, d_head 128, 2 of 4 KV heads
    streaming, S=128, W=4096; one cache per layer, seeded N(0,1) bf16 K/V)
    at several context lengths, as the paper reports it. Each token runs the
    28 layers' decode steps through the allocation-free entry point, once
    launched eagerly from the host and once replayed as one CUDA graph
    captured for all 28 layers."""
    import torch

    from paper_2608_06849_gb300 import aoh
    from paper_2608_06849_gb300 import build as aoh_build
    from paper_2608_06849_gb300.workloads import STACK_256K, decode_inputs, labels_for, randn_bf16
    aoh_build.build()
    aoh.load()
    peaks, note = load_peaks()
    hbm = float(peaks.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"]))
    wl = STACK_256K
    L, B, Hq, Hkv, D = wl.layers, 1, wl.n_q_heads, wl.n_kv_heads, wl.d_head
    tokens = max(args.steps, 8)
    points = []
    for T in (4096, 32768, 131072):
        cap = T + 2 * tokens + args.warmup + 8
        caches, lens, ins, outs, labels = [], [], [], [], []
        for layer in range(L):
            lab = labels_for(wl, layer=layer)
            c = aoh.Cache(B, Hq, Hkv, D, cap, wl.sink, wl.window, lab)
            k = randn_bf16((B, T, Hkv, D), 5000 + 2 * layer, "cuda")
            v = randn_bf16((B, T, Hkv, D), 5001 + 2 * layer, "cuda")
            c.prefill(None, k, v, None)
            del k, v
            caches.append(c)
            labels.append(lab)
            lens.append(torch.full((B,), T, dtype=torch.int32, device="cuda"))
            ins.append(decode_inputs(wl, layer, device="cuda"))
            outs.append(torch.empty(B, Hq, D, dtype=torch.bfloat16, device="cuda"))
        torch.cuda.synchronize()
        bound = cap - 1  # host upper bound of every length during this run

        def token():
            for layer in range(L):
                aoh.aoh_decode_step_noalloc(caches[layer].cfg, labels[layer], caches[layer].buffer, lens[layer], bound,
                                            *ins[layer], outs[layer])

        for _ in range(max(args.warmup, 3)):
            token()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        e0.record()
        for _ in range(tokens):
            token()
        e1.record()
        torch.cuda.synchronize()
        eager_us = e0.elapsed_time(e1) * 1000 / tokens
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            token()
        graph.replay()
        torch.cuda.synchronize()
        e0.record()
        for _ in range(tokens):
            graph.replay()
        e1.record()
        torch.cuda.synchronize()
        graph_us = e0.elapsed_time(e1) * 1000 / tokens
        t_mid = T + max(args.warmup, 3) + tokens
        nbytes = sum(decode_bytes([t_mid], labels[layer], wl) for layer in range(L))
        points.append({"context": T, "eager_us_per_token": round(eager_us, 1), "graph_us_per_token": round(graph_us, 1),
                       "bytes_per_token": nbytes, "graph_hbm_gbs": round(nbytes / (graph_us * 1e-6) / 1e9, 1),
                       "graph_frac_of_peak": round(nbytes / (graph_us * 1e-6) / 1e9 / hbm, 4)})
        for c in caches:
            c.close()
        del caches, lens, ins, outs, graph
        torch.cuda.empty_cache()
    print(json.dumps({
        "workload": f"{wl.name}-decode-per-token: {L} layers x (Hq={Hq} Hkv={Hkv} d={D}), B=1, 2 of 4 KV heads "
                    f"streaming per layer, S={wl.sink} W={wl.window}; {tokens} tokens per point",
        "points": points, "peak_hbm_gbs": hbm, "peak_note": note}))


def run_classify(args):
    """Effective-rank classification of a Qwen2.5-7B-shaped model (28 layers
    of 28 query / 4 KV heads, d_head 128, d_model 3584; seeded N(0,1) bf16
    weights whose rows decay geometrically at a random rate per head): one
    layer per call and all 28 layers in one call, timed on the GPU; the
    float64 oracle on one layer on the host cores."""
    import numpy as np
    import torch

    from oracle import effective_rank as oer
    from paper_2608_06849_gb300 import aoh
    from paper_2608_06849_gb300 import build as aoh_build
    aoh_build.build()
    aoh.load()
    Hq, Hkv, dh, dm, layers = 28, 4, 128, 3584, 28
    gen = torch.Generator().manual_seed(0)
    decay = torch.logspace(0, -2, dh, dtype=torch.float64)
    wq = torch.empty(layers, Hq, dh, dm, dtype=torch.bfloat16)
    wk = torch.empty(layers, Hkv, dh, dm, dtype=torch.bfloat16)
    for l in range(layers):
        expo = torch.rand(Hq, 1, 1, generator=gen, dtype=torch.float64) * 1.5
        wq[l] = ((decay[None, :, None] ** expo) * torch.randn(Hq, dh, dm, generator=gen, dtype=torch.float64)).bfloat16()
        wk[l] = (decay[None, :, None] ** 0.5 * torch.randn(Hkv, dh, dm, generator=gen, dtype=torch.float64)).bfloat16()
    dq, dk = wq.cuda(), wk.cuda()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

    def timed(fn, reps):
        for _ in range(max(args.warmup, 3)):
            fn()
        torch.cuda.synchronize()
        e0.record()
        for _ in range(reps):
            out = fn()
        e1.record()
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / reps, out

    ms_layer, (labels0, er0) = timed(lambda: aoh.aoh_classify(dq[0], dk[0], Hkv, 50), 3)
    ms_model, (labels, ers) = timed(lambda: aoh.aoh_classify(dq, dk, Hkv, 50), 3)
    gram_flops = 2.0 * dh * dh * dm * (Hq + Hkv) * layers
    t0 = time.perf_counter()
    want = oer.head_scores(wq[0].double().numpy(), wk[0].double().numpy(), Hkv)
    cpu_s = time.perf_counter() - t0
    fp64_peak = 1250.0  # GFLOP/s, the nominal FP64 rate of this part
    print(json.dumps({
        "workload": f"qwen2.5-7b-classify: {layers} layers x (Hq={Hq} Hkv={Hkv} d_head={dh} d_model={dm}), "
                    "sparsity 50%",
        "ms_one_layer_per_call": round(ms_layer, 3), "ms_model_in_one_call": round(ms_model, 2),
        "ms_per_layer_in_model_call": round(ms_model / layers, 3),
        "labels_layer0": labels[0], "labels_layer0_single_call": labels0,
        "max_rel_err_vs_oracle_layer0": float(np.max(np.abs(np.array(ers[0]) - want) / want)),
        "roofline": {"bound": "alu", "achieved": round(gram_flops / (ms_model * 1e-3) / 1e9, 1),
                     "peak": fp64_peak, "unit": "GFLOP/s",
                     "frac": round(gram_flops / (ms_model * 1e-3) / 1e9 / fp64_peak, 4),
                     "note": "Gram flops (2 d_head^2 d_model per projection) over the whole model call; "
                             "FP64 nominal"},
        "cpu_baseline": {"value": round(cpu_s * 1e3, 1), "unit": "ms/layer", "cores": os.cpu_count(),
                         "kind": "oracle", "sample": "layer 0, float64 oracle head_scores", **host_cpu()}}))


def run_h2map(args):
    """H2Share head mapping of one Qwen2.5-7B-shaped layer pair (28 query / 4
    KV heads, d_head 128, d_model 3584; seeded N(0,1) bf16 weights, the reuse
    layer a noisy group-permuted copy of the anchor): the whole
    aoh_h2share_map call timed on the GPU, its tensor-core contractions
    against the bf16 peak; the float64 oracle on the host cores."""
    import numpy as np
    import torch

    from oracle import h2share as ohs
    from paper_2608_06849_gb300 import aoh
    from paper_2608_06849_gb300 import build as aoh_build
    aoh_build.build()
    aoh.load()
    Hq, Hkv, dh, dm = 28, 4, 128, 3584
    g = Hq // Hkv
    gen = torch.Generator().manual_seed(0)
    wqa = torch.randn(Hq, dh, dm, generator=gen, dtype=torch.float64)
    wka = torch.randn(Hkv, dh, dm, generator=gen, dtype=torch.float64)
    perm = [2, 0, 3, 1]
    wqr = torch.cat([wqa[p * g:(p + 1) * g] for p in perm]) + 0.5 * torch.randn(Hq, dh, dm, generator=gen,
                                                                               dtype=torch.float64)
    wkr = wka[perm] + 0.5 * torch.randn(Hkv, dh, dm, generator=gen, dtype=torch.float64)
    w = [x.bfloat16() for x in (wqa, wka, wqr, wkr)]
    dw = [x.cuda() for x in w]
    la = lr = [0] * Hkv
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    for _ in range(max(args.warmup, 3)):
        aoh.aoh_h2share_map(*dw, la, lr)
    reps = 10
    torch.cuda.synchronize()
    e0.record()
    for _ in range(reps):
        m, sim = aoh.aoh_h2share_map(*dw, la, lr)
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / reps
    nq, nk = Hq * dh, Hkv * dh
    tiles = lambda n: (n + 127) // 128
    flops = 2.0 * dm * (nq * nq + nk * nk + 2 * tiles(nq) * 128 * 128 + 2 * tiles(nk) * 128 * 128)
    t0 = time.perf_counter()
    want = ohs.group_similarity(*[x.double().numpy() for x in w])
    cpu_s = time.perf_counter() - t0
    peaks, note = load_peaks()
    peak = float(peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"]))
    ach = flops / (ms * 1e-3) / 1e12
    print(json.dumps({
        "workload": f"qwen2.5-7b-h2share-map: one layer pair (Hq={Hq} Hkv={Hkv} d_head={dh} d_model={dm})",
        "ms_per_layer_pair": round(ms, 4), "map": m, "map_expected_from_construction": perm,
        "max_abs_err_group_sim_vs_oracle": float(np.max(np.abs(np.array(sim) - want))),
        "roofline": {"bound": "tensor", "achieved": round(ach, 1), "peak": peak, "unit": "TFLOP/s",
                     "frac": round(ach / peak, 4),
                     "note": "bf16 contraction flops of the whole call (Q_a Q_r^T, K_r K_a^T, four diagonal-block "
                             "Grams) over the whole call's time, including the fp64 trace kernel, the map kernel "
                             "and the host copy; " + note + " burst peak"},
        "cpu_baseline": {"value": round(cpu_s * 1e3, 1), "unit": "ms/layer pair", "cores": os.cpu_count(),
                         "kind": "oracle", "sample": "the same layer pair, float64 oracle group_similarity",
                         **host_cpu()}}))


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=64)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["native", "reference"], default="native")
    ap.add_argument("--prefill-steps", type=int, default=10)
    ap.add_argument("--prefill-chunks", type=int, default=8)
    ap.add_argument("--workload", choices=["default", "ragged", "stack", "classify", "h2map", "graph"],
                    default="default",
                    help="default: the headline decode + prefill run; ragged / stack: the other two workloads; "
                         "classify: the effective-rank head classifier; h2map: the H2Share head mapping; "
                         "graph: batch-1 per-token decode through 28 layers, eager and as one CUDA graph")
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--h2-top-k", type=int, default=2048, help="positions an H2Share anchor step selects")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--decode-batch", type=int, default=None, help="smaller decode batch (profiling runs)")
    ap.add_argument("--decode-ctx", type=int, default=None, help="smaller decode context (profiling runs)")
    ap.add_argument("--prefill-len", type=int, default=None, help="shorter prefill (profiling runs)")
    ap.add_argument("--stack-layers", type=int, default=2, help="layers of the 256K stack timed")
    ap.add_argument("--extra-steps", type=int, default=16,
                    help="timed decode steps of the stack and ragged legs in the default run")
    ap.add_argument("--no-extra-workloads", action="store_true",
                    help="default run without the 256K stack and ragged sweep legs (profiling runs)")
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "native":
        args.warmup = 3
    if args.impl == "reference":
        run_reference(args)
    elif args.workload == "ragged":
        run_ragged(args)
    elif args.workload == "stack":
        run_stack(args)
    elif args.workload == "classify":
        run_classify(args)
    elif args.workload == "h2map":
        run_h2map(args)
    elif args.workload == "graph":
        run_graph(args)
    else:
        run_native(args)


if __name__ == "__main__":
    main()
