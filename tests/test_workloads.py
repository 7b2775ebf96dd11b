"""The seeded input generators shared by the oracle and the CUDA path: the
same seed gives the same tensors, labels pick exactly the requested number
of streaming heads, the sink scaling is exact, and the five workloads carry
the shapes of the paper's models."""

import torch

from paper_2608_06849_gb300 import workloads as w


def test_same_seed_same_tensors_other_seed_differs():
    a = w.randn_bf16((3, 5, 7), 11)
    assert a.dtype == torch.bfloat16
    assert torch.equal(a, w.randn_bf16((3, 5, 7), 11))
    assert not torch.equal(a, w.randn_bf16((3, 5, 7), 12))


def test_labels_count_and_seed():
    for n_kv, n_s in ((4, 2), (8, 4), (8, 0), (8, 8), (2, 1)):
        for seed in range(5):
            lab = w.head_labels(n_kv, n_s, seed)
            assert len(lab) == n_kv and sum(lab) == n_s and set(lab) <= {0, 1}
            assert lab == w.head_labels(n_kv, n_s, seed)
    # streaming heads are randperm(n)[:k] under the seed
    perm = torch.randperm(8, generator=torch.Generator().manual_seed(0))[:4].tolist()
    assert [h for h, x in enumerate(w.head_labels(8, 4, 0)) if x] == sorted(perm)


def test_sink_scaling_is_exact():
    wl = w.Workload("t", 2, 4, 2, 8, 6, 1, 2, 3, 1, seed=3, sink_scale=8.0)
    plain = w.Workload("t", 2, 4, 2, 8, 6, 1, 2, 3, 1, seed=3)
    q, k, v = w.prefill_inputs(wl)
    q0, k0, v0 = w.prefill_inputs(plain)
    assert torch.equal(q, q0) and torch.equal(v, v0)
    assert torch.equal(k[:, 1:], k0[:, 1:])
    assert torch.equal(k[:, 0].float(), k0[:, 0].float() * 8)


def test_shapes_and_decode_steps_differ():
    wl = w.TINY
    q, k, v = w.prefill_inputs(wl)
    assert q.shape == (1, 1024, 8, 64) and k.shape == v.shape == (1, 1024, 2, 64)
    d0, d1 = w.decode_inputs(wl, 0), w.decode_inputs(wl, 1)
    assert d0[0].shape == (1, 8, 64) and d0[1].shape == (1, 2, 64)
    assert not torch.equal(d0[0], d1[0])
    assert w.labels_for(wl) == [0, 1]


def test_paper_model_shapes():
    assert (w.PREFILL_32K.n_q_heads, w.PREFILL_32K.n_kv_heads, w.PREFILL_32K.d_head) == (28, 4, 128)
    assert (w.DECODE_128K.n_q_heads, w.DECODE_128K.n_kv_heads, w.DECODE_128K.batch) == (32, 8, 16)
    assert w.DECODE_128K.prefill_len == 131072 and w.PREFILL_32K.prefill_len == 32768
    assert w.STACK_256K.layers == 28 and w.STACK_256K.prefill_len == 262144
    for wl in w.ALL:
        assert sum(w.labels_for(wl)) == (1 if wl is w.TINY else wl.n_streaming)
    # per-layer labels of the stack: half streaming in every layer, seeded by layer
    per_layer = [w.labels_for(w.STACK_256K, layer) for layer in range(28)]
    assert all(sum(lab) == 2 for lab in per_layer) and len({tuple(x) for x in per_layer}) > 1


def test_ragged_lengths_in_range_and_seeded():
    lens = w.seq_lens(w.RAGGED)
    assert len(lens) == 64 and all(4096 <= x <= 32768 for x in lens)
    assert lens == w.seq_lens(w.RAGGED) and len(set(lens)) > 32
    assert w.seq_lens(w.DECODE_128K) == [131072] * 16
