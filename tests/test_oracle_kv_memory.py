"""The KV-cache byte formula reproduces the memory numbers the paper prints."""

import os

import pytest

from oracle import kv_memory as kvm

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _rows(name):
    out = []
    for line in open(os.path.join(GOLDEN, name)):
        line = line.strip()
        if line and not line.startswith("#"):
            out.append(line.split())
    return out


@pytest.mark.parametrize("row", _rows("kv_memory_32k_table.txt"), ids=lambda r: f"{r[0]}-sp{r[5]}")
def test_32k_kv_memory_table(row):
    model, L, G, d, ctx, sp, S, W, printed, dec = row
    nbytes = kvm.model_kv_bytes(int(L), int(G), int(sp), int(ctx), int(S), int(W), int(d))
    assert kvm.round_half_up(kvm.gib(nbytes), int(dec)) == float(printed)


@pytest.mark.parametrize("row", _rows("kv_memory_prefill_efficiency_tables.txt"),
                         ids=lambda r: f"{r[0]}-{r[4]}-sp{r[5]}")
def test_efficiency_tables_prefill_memory(row):
    model, L, G, d, ctx, sp, S, W, printed = row
    nbytes = kvm.model_kv_bytes(int(L), int(G), int(sp), int(ctx), int(S), int(W), int(d))
    assert kvm.round_half_up(kvm.gb(nbytes), 3) == float(printed)


def test_384_not_512_token_streaming_budget():
    """The appendix text says 512 tokens, the printed 0.885 GiB needs 384."""
    at384 = kvm.model_kv_bytes(28, 4, 50, 32768, 128, 256, 128)
    at512 = kvm.model_kv_bytes(28, 4, 50, 32768, 128, 384, 128)
    assert kvm.round_half_up(kvm.gib(at384), 3) == 0.885
    assert kvm.round_half_up(kvm.gib(at512), 3) != 0.885


def test_single_layer_formula():
    # B * (n_R * max_seq + n_S * (S + W)) * d * 2 (K,V) * 2 (bf16)
    assert kvm.kv_cache_bytes(2, 3, 1, 100, 4, 6, 64) == 2 * (300 + 10) * 64 * 4
    assert kvm.kv_cache_bytes(1, 0, 0, 100, 4, 6, 64) == 0


def test_budget_rounds_up():
    """k = ceil((1 - s) G): 7 groups at 50 % keep 4, 3 groups at 10 % keep 3."""
    assert kvm.retrieval_groups(7, 50) == 4
    assert kvm.retrieval_groups(3, 10) == 3
    assert kvm.retrieval_groups(4, 50) == 2
