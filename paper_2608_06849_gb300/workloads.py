"""Seeded synthetic inputs shaped like the paper's workloads.

This module draws random numbers and picks head labels; it holds none of the
attention arithmetic, so both the CUDA path and the CPU oracle may be fed from
it. The paper measures on LongBench / passkey prompts through real models
(Sec. 6.1, Appendix "Additional Efficiency Results"); attention cost depends
only on shapes, lengths and the label mix, so N(0,1) bf16 tensors with the
paper's model shapes (Qwen2.5-7B: 28 query / 4 KV heads; Llama-3-8B: 32 / 8;
d_head 128) and context lengths stand in for those prompts.
"""

from dataclasses import dataclass, field

import torch


@dataclass
class Workload:
    name: str
    batch: int
    n_q_heads: int
    n_kv_heads: int
    d_head: int
    prefill_len: int          # tokens per sequence before decoding (max over the batch)
    decode_steps: int
    sink: int
    window: int
    n_streaming: int          # KV heads labelled streaming, chosen by seeded permutation
    seed: int = 0
    sink_scale: float = 1.0   # first key of every (sequence, KV head) multiplied by this
    ragged: tuple = None      # (lo, hi) inclusive range of per-sequence lengths, or None
    layers: int = 1
    extra: dict = field(default_factory=dict)

    @property
    def g(self):
        return self.n_q_heads // self.n_kv_heads


def head_labels(n_kv_heads, n_streaming, seed):
    """uint8 labels per KV head (0 retrieval, 1 streaming); the streaming ones
    are ``randperm(n_kv_heads)[:n_streaming]`` under ``seed``."""
    gen = torch.Generator().manual_seed(int(seed))
    perm = torch.randperm(n_kv_heads, generator=gen)
    labels = torch.zeros(n_kv_heads, dtype=torch.uint8)
    labels[perm[:n_streaming]] = 1
    return labels.tolist()


def seq_lens(wl):
    """Per-sequence prefill lengths: all ``prefill_len`` or seeded uniform ints."""
    if wl.ragged is None:
        return [wl.prefill_len] * wl.batch
    lo, hi = wl.ragged
    gen = torch.Generator().manual_seed(int(wl.seed))
    return torch.randint(lo, hi + 1, (wl.batch,), generator=gen).tolist()


def randn_bf16(shape, seed, device="cpu"):
    """bf16 tensor rounded from float32 N(0,1) draws of a seeded generator."""
    gen = torch.Generator(device=device).manual_seed(int(seed))
    return torch.randn(shape, generator=gen, device=device, dtype=torch.float32).to(torch.bfloat16)


def prefill_inputs(wl, device="cpu", seed_offset=0):
    """q [B,T,Hq,d], k/v [B,T,Hkv,d] in bf16. ``k[:, 0] *= sink_scale`` (a power
    of two, so exact in bf16) makes position 0 an attention sink."""
    B, T = wl.batch, wl.prefill_len
    s = wl.seed * 1000 + seed_offset
    q = randn_bf16((B, T, wl.n_q_heads, wl.d_head), s + 1, device)
    k = randn_bf16((B, T, wl.n_kv_heads, wl.d_head), s + 2, device)
    v = randn_bf16((B, T, wl.n_kv_heads, wl.d_head), s + 3, device)
    if wl.sink_scale != 1.0 and T > 0:
        k[:, 0] *= wl.sink_scale
    return q, k, v


def decode_inputs(wl, step, device="cpu"):
    """New-token q [B,Hq,d], k/v [B,Hkv,d] for decode step ``step``."""
    s = wl.seed * 1000 + 100 + 3 * int(step)
    B = wl.batch
    q = randn_bf16((B, wl.n_q_heads, wl.d_head), s + 1, device)
    k = randn_bf16((B, wl.n_kv_heads, wl.d_head), s + 2, device)
    v = randn_bf16((B, wl.n_kv_heads, wl.d_head), s + 3, device)
    return q, k, v


# The five workloads: the tiny parity case, Qwen2.5-7B-shaped prefill at 32K,
# Llama-3-8B-shaped decode at 128K, a 28-layer Qwen2.5-7B-shaped stack at 256K,
# and the ragged decode sweep.
TINY = Workload("tiny-8q2kv-d64-T1024", 1, 8, 2, 64, 1024, 32, 16, 128, 1, sink_scale=8.0,
                extra={"labels": [0, 1]})
PREFILL_32K = Workload("qwen2.5-7b-prefill-32k", 1, 28, 4, 128, 32768, 0, 128, 2048, 2, sink_scale=8.0)
DECODE_128K = Workload("llama3-8b-decode-128k-b16", 16, 32, 8, 128, 131072, 64, 128, 4096, 4)
STACK_256K = Workload("qwen2.5-7b-stack28-256k", 1, 28, 4, 128, 262144, 128, 128, 4096, 2, layers=28)
RAGGED = Workload("llama3-8b-ragged-b64", 64, 32, 8, 128, 32768, 1, 64, 2048, 4, ragged=(4096, 32768))

ALL = [TINY, PREFILL_32K, DECODE_128K, STACK_256K, RAGGED]


def labels_for(wl, layer=0):
    if "labels" in wl.extra:
        return list(wl.extra["labels"])
    return head_labels(wl.n_kv_heads, wl.n_streaming, wl.seed + layer)
