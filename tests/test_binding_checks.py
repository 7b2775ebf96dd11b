"""The Python binding refuses tensors too small for the cache's configuration
before any pointer reaches the library (the C ABI gets bare pointers and
cannot check sizes). Runs on the CPU: a Cache object is assembled without a
device buffer, and correctly sized CPU tensors get past the size checks only
to be refused as non-CUDA tensors."""

import pytest
import torch

from paper_2608_06849_gb300 import aoh


def _cache(B=2, Hq=8, Hkv=2, D=64, labels=(0, 1)):
    c = object.__new__(aoh.Cache)
    c.batch, c.n_q_heads, c.n_kv_heads, c.d_head = B, Hq, Hkv, D
    c.labels = list(labels)
    c.handle = None
    return c


def _bf16(*shape):
    return torch.zeros(*shape, dtype=torch.bfloat16)


def _needs_cuda(excinfo):
    return "CUDA tensor" in str(excinfo.value)


def test_prefill_sizes():
    c = _cache()
    q, kv = _bf16(2, 10, 8, 64), _bf16(2, 10, 2, 64)
    with pytest.raises(ValueError) as e:
        c.prefill(q, kv, kv, _bf16(2, 10, 8, 64))
    assert _needs_cuda(e)
    for args, name in (((_bf16(2, 9, 8, 64), kv, kv, None), "q"),
                       ((q, kv, _bf16(2, 10, 1, 64), None), "v"),
                       ((q, kv, kv, _bf16(1, 10, 8, 64)), "out"),
                       ((None, _bf16(1, 10, 2, 64), kv, None), "k")):
        with pytest.raises(ValueError, match=f"^{name} holds"):
            c.prefill(*args)
    with pytest.raises(ValueError, match="seq_lens"):
        c.prefill(q, kv, kv, None, seq_lens=[10])


def test_decode_sizes():
    c = _cache()
    q, kv = _bf16(2, 8, 64), _bf16(2, 2, 64)
    with pytest.raises(ValueError) as e:
        c.decode_step(q, kv, kv, _bf16(2, 8, 64))
    assert _needs_cuda(e)
    with pytest.raises(ValueError, match="^out holds"):
        c.decode_step(q, kv, kv, _bf16(2, 7, 64))
    with pytest.raises(ValueError, match="^k_new holds"):
        c.decode_step(q, _bf16(2, 1, 64), kv, q)


def test_h2share_index_sizes():
    c = _cache(labels=(0, 0))
    q, kv = _bf16(2, 8, 64), _bf16(2, 2, 64)
    idx = torch.zeros(2, 2, 16, dtype=torch.int32)
    with pytest.raises(ValueError) as e:
        c.decode_step_anchor(q, kv, kv, q, 16, idx)
    assert _needs_cuda(e)
    with pytest.raises(ValueError, match="^indices holds"):
        c.decode_step_anchor(q, kv, kv, q, 17, idx)
    with pytest.raises(ValueError, match="^indices holds"):
        c.decode_step_reuse(q, kv, kv, q, idx, 17, [0, 1])
    with pytest.raises(ValueError, match="batch, n_anchor_groups, top_k"):
        c.decode_step_reuse(q, kv, kv, q, idx.view(4, 16), 16, [0, 1])
    with pytest.raises(ValueError) as e:
        c.decode_step_reuse(q, kv, kv, q, idx, 16, [0, 1])
    assert _needs_cuda(e)


def test_reuse_group_map_slots():
    # anchor retrieval groups 1 and 3 hold index-list slots 0 and 1
    anchor = [1, 0, 1, 0]
    reuse = [0, 1, 0, 0]
    head_map = [3, -1, 1, 3]
    assert aoh.reuse_group_map(head_map, anchor, reuse) == [1, 0, 1]
    assert aoh.reuse_group_map([0, 0], [1, 1], [1, 1]) == []
    with pytest.raises(ValueError, match="not an anchor retrieval group"):
        aoh.reuse_group_map([0, 1, 1, 3], anchor, reuse)


def test_missing_library_fails_loudly(monkeypatch, tmp_path):
    """No fallback: without the built library every call raises."""
    monkeypatch.setattr(aoh, "_lib", None)
    monkeypatch.setattr(aoh, "LIB_PATH", str(tmp_path / "libaoh.so"))
    with pytest.raises(RuntimeError, match="is missing"):
        aoh.aoh_version()
    with pytest.raises(RuntimeError, match="is missing"):
        aoh.aoh_cache_bytes(aoh.make_config(1, 8, 2, 64, 16, 2, 4), [0, 1])


def test_h2share_map_shapes():
    wq, wk = _bf16(8, 64, 96), _bf16(2, 64, 96)
    with pytest.raises(ValueError, match="^w_q_reuse has shape"):
        aoh.aoh_h2share_map(wq, wk, _bf16(8, 64, 95), wk, [0, 0], [0, 0])
    with pytest.raises(ValueError, match="^w_k_anchor has shape"):
        aoh.aoh_h2share_map(wq, _bf16(2, 64, 95), wq, _bf16(2, 64, 95), [0, 0], [0, 0])
    with pytest.raises(ValueError, match="entries"):
        aoh.aoh_h2share_map(wq, wk, wq, wk, [0, 0, 0], [0, 0])
    with pytest.raises(ValueError) as e:
        aoh.aoh_h2share_map(wq, wk, wq, wk, [0, 0], [0, 0])
    assert _needs_cuda(e)


def test_noalloc_sizes():
    cfg = aoh.make_config(2, 8, 2, 64, 100, 4, 16)
    labels = [0, 1]
    kv_bytes = 2 * (100 + 20) * 64 * 4
    kv = torch.zeros(kv_bytes, dtype=torch.uint8)
    lens = torch.zeros(2, dtype=torch.int32)
    q, k1 = _bf16(2, 8, 64), _bf16(2, 2, 64)
    with pytest.raises(ValueError, match="^kv_buffer holds"):
        aoh.aoh_decode_step_noalloc(cfg, labels, kv[:-1], lens, 10, q, k1, k1, q)
    with pytest.raises(ValueError, match="^lens holds"):
        aoh.aoh_decode_step_noalloc(cfg, labels, kv, lens[:1], 10, q, k1, k1, q)
    with pytest.raises(ValueError, match="^v_new holds"):
        aoh.aoh_decode_step_noalloc(cfg, labels, kv, lens, 10, q, k1, k1[:1], q)
    with pytest.raises(ValueError, match="entries"):
        aoh.aoh_decode_step_noalloc(cfg, [0], kv, lens, 10, q, k1, k1, q)
    with pytest.raises(ValueError, match="CUDA tensor"):
        aoh.aoh_decode_step_noalloc(cfg, labels, kv, lens, 10, q, k1, k1, q)
