"""GPU parity through the C ABI: outputs against the float64 oracle on the
same bf16 inputs (max |err| <= 1e-2, mean |err| <= 1e-3, and two bf16 ulps
elementwise); cache contents bit-exact against the oracle's slot model."""

import pytest
import torch

from gpu_cases import run_case
from paper_2608_06849_gb300.workloads import TINY, labels_for

pytestmark = pytest.mark.gpu


def test_tiny_workload_prefill_then_32_decode_steps():
    """8 query / 2 KV heads, d 64, 1024-token prefill then 32 decode steps;
    KV head 0 retrieval, KV head 1 streaming with S=16, W=128; sink key x8."""
    wl = TINY
    run_case(wl.batch, wl.n_q_heads, wl.n_kv_heads, wl.d_head, wl.prefill_len, wl.sink, wl.window,
             labels_for(wl), decode_steps=wl.decode_steps, sink_scale=wl.sink_scale, raw_name="tiny")


CASES = {
    # name: (B, Hq, Hkv, d, T, S, W, labels, seq_lens, decode_steps)
    "ragged_two_seqs": (2, 8, 2, 128, 300, 4, 37, [1, 0], [300, 123], 5),
    "T_below_S": (1, 8, 2, 128, 10, 16, 8, [1, 0], None, 12),
    "T_below_S_plus_W": (1, 8, 2, 64, 50, 16, 64, [1, 1], None, 40),
    "sink0_window1": (1, 4, 1, 128, 70, 0, 1, [1], None, 3),
    "all_retrieval": (2, 8, 2, 128, 333, 16, 32, [0, 0], None, 3),
    "all_streaming": (1, 16, 4, 128, 517, 7, 100, [1, 1, 1, 1], None, 3),
    "group7_d128": (1, 14, 2, 128, 257, 8, 100, [0, 1], None, 4),
    "group2_d128": (1, 4, 2, 128, 150, 3, 20, [1, 0], None, 3),
    "group8_d64": (1, 16, 2, 64, 200, 5, 33, [0, 1], None, 3),
    "group7_d64": (1, 7, 1, 64, 129, 2, 50, [1], None, 3),
    "group2_d64": (1, 4, 2, 64, 150, 3, 20, [0, 1], None, 3),
    "ring_wraps_many_times": (1, 8, 2, 128, 40, 3, 5, [1, 0], None, 30),
    "single_token_prefill": (3, 8, 2, 128, 1, 4, 4, [0, 1], None, 6),
    "tile_edges": (1, 8, 2, 128, 65, 1, 63, [1, 0], None, 70),
    "mha_group1_d128": (1, 2, 2, 128, 140, 4, 30, [0, 1], None, 3),
    "mha_group1_d64": (2, 3, 3, 64, 90, 0, 7, [1, 0, 1], [90, 41], 3),
    "prefill_multi_tile_ragged": (3, 8, 2, 128, 777, 16, 200, [1, 0], [777, 129, 640], 2),
    # group sizes 7 and 8 at d 128 decode on the tensor cores: tiles of 128 keys
    # with tails of 1 and 127 rows, a ring that wraps, several items per CTA
    "group7_d128_tile_edges": (1, 14, 2, 128, 127, 1, 126, [0, 1], None, 70),
    "group7_d128_ring_wraps": (1, 7, 1, 128, 40, 3, 5, [1], None, 30),
    "group8_d128_ragged": (3, 16, 2, 128, 600, 8, 129, [1, 0], [600, 255, 1], 5),
    "group8_d128_four_heads": (2, 32, 4, 128, 1000, 16, 32, [0, 1, 0, 0], None, 3),
    "group3_d128": (1, 6, 2, 128, 300, 4, 50, [1, 0], None, 3),
    "group5_d128": (2, 10, 2, 128, 260, 4, 50, [0, 1], [260, 131], 3),
    "group6_d128": (1, 12, 2, 128, 129, 2, 64, [1, 0], None, 3),
    "group16_d128": (1, 32, 2, 128, 400, 8, 100, [0, 1], None, 3),
    # short decode steps charge each item's start in the CTA split: items of
    # one to a few rows next to long ones, so CTA ranges cover several item
    # starts and sometimes no row of an item
    "tiny_items_with_item_charge": (12, 16, 4, 128, 3000, 4, 64, [0, 1, 0, 1],
                                    [3000, 1, 2, 3, 700, 1, 1, 2500, 5, 1, 64, 129], 4),
}


@pytest.mark.parametrize("name", sorted(CASES))
def test_small_case(name):
    B, Hq, Hkv, d, T, S, W, labels, lens, steps = CASES[name]
    run_case(B, Hq, Hkv, d, T, S, W, labels, seq_lens=lens, decode_steps=steps)


def test_peaky_keys_relative_error():
    """Keys scaled x4 make the softmax sharp, so a dropped or misplaced term
    cannot hide behind a near-uniform average. A sharp softmax puts weights
    near 1 on single keys, where bf16 rounding of P and of the output alone
    reach ~1.6e-2 for |v| ~ 4, so this case is held to the elementwise bound
    derived from that arithmetic (not the workloads' absolute 1e-2)."""
    run_case(1, 8, 2, 128, 400, 16, 64, [0, 1], decode_steps=4, peaky=4.0, sink_scale=1.0, abs_bounds=False)


def test_long_decode_split_path():
    """Long enough that decode uses many split-KV CTAs and the fused combine."""
    run_case(2, 8, 2, 128, 20000, 64, 1000, [0, 1], decode_steps=3, check_prefill_out=True,
             rows=[0, 1, 63, 64, 1063, 1064, 9999, 19999])


def test_long_decode_split_path_group7():
    """The same at group size 7: each item's rows span more than 16 CTAs, so
    the split partials merge in two levels."""
    run_case(2, 14, 2, 128, 20000, 64, 1000, [0, 1], decode_steps=3, check_prefill_out=False)


def test_decode_past_capacity_is_refused():
    from paper_2608_06849_gb300 import aoh
    from gpu_cases import ensure_lib
    ensure_lib()
    cache = aoh.Cache(1, 8, 2, 64, 4, 2, 2, [0, 1])
    k = torch.randn(1, 4, 2, 64, device="cuda").to(torch.bfloat16)
    cache.prefill(k.repeat(1, 1, 4, 1), k, k)
    q1 = torch.zeros(1, 8, 64, device="cuda", dtype=torch.bfloat16)
    k1 = torch.zeros(1, 2, 64, device="cuda", dtype=torch.bfloat16)
    with pytest.raises(aoh.AohError) as e:
        cache.decode_step(q1, k1, k1, torch.empty_like(q1))
    assert e.value.status == 2
    with pytest.raises(aoh.AohError) as e:            # a further chunk would pass max_seq
        cache.prefill(k.repeat(1, 1, 4, 1), k, k)
    assert e.value.status == 2
    cache.reset()
    cache.prefill(k.repeat(1, 1, 4, 1), k, k)
    assert cache.lens() == [4]
    cache.close()
