"""The C-ABI library loads and exports every symbol include/aoh.h declares;
host-only calls (byte count, argument validation) behave as documented.
No compute call is made here, so these run without a GPU."""

import ctypes
import os
import re

import pytest

from oracle import kv_memory as kvm
from paper_2608_06849_gb300 import aoh
from paper_2608_06849_gb300 import build as aoh_build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "aoh.h")


@pytest.fixture(scope="module")
def lib():
    aoh_build.build()
    return aoh.load()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    names = re.findall(r"\b(aoh_[a-z0-9_]+)\s*\(", text)
    return sorted(set(names))


def test_header_declares_the_boundary():
    names = declared_functions()
    for n in ["aoh_cache_bytes", "aoh_cache_init", "aoh_prefill", "aoh_decode_step"]:
        assert n in names


def test_every_declared_symbol_is_exported(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name
    assert set(declared_functions()) <= set(aoh.EXPORTS) | set(declared_functions())
    assert sorted(aoh.EXPORTS) == declared_functions()


def test_noalloc_rejects_bad_arguments_on_host(lib):
    cfg = aoh.make_config(1, 8, 2, 64, 64, 4, 8)
    labels = (ctypes.c_uint8 * 2)(0, 1)
    fake = ctypes.c_void_p(1 << 20)
    assert lib.aoh_decode_step_noalloc(ctypes.byref(cfg), labels, None, None, 0, fake, fake, fake, fake, None) == 1
    big = aoh.make_config(4096, 8, 8, 64, 64, 4, 8)  # 32768 (b, head) items > 16320
    labels8 = (ctypes.c_uint8 * 8)(*([0] * 8))
    lens = ctypes.cast(fake, ctypes.POINTER(ctypes.c_int32))
    assert lib.aoh_decode_step_noalloc(ctypes.byref(big), labels8, fake, lens, 0, fake, fake, fake, fake, None) == 2
    assert "16320" in lib.aoh_last_error().decode()


def test_version(lib):
    assert aoh.aoh_version() == 102


@pytest.mark.parametrize("B,Hq,Hkv,d,max_seq,S,W,labels", [
    (1, 8, 2, 64, 1056, 16, 128, [0, 1]),
    (1, 28, 4, 128, 32768, 128, 2048, [1, 1, 0, 0]),
    (16, 32, 8, 128, 131136, 128, 4096, [1, 0, 0, 1, 1, 0, 0, 1]),
    (3, 4, 4, 64, 100, 0, 1, [1, 1, 1, 1]),
    (2, 4, 2, 128, 7, 5, 9, [0, 0]),
])
def test_cache_bytes_matches_formula(lib, B, Hq, Hkv, d, max_seq, S, W, labels):
    cfg = aoh.make_config(B, Hq, Hkv, d, max_seq, S, W)
    n_s = sum(labels)
    want = kvm.kv_cache_bytes(B, Hkv - n_s, n_s, max_seq, S, W, d)
    assert aoh.aoh_cache_bytes(cfg, labels) == want


def test_qwen25_stack_bytes(lib):
    """28 layers of the Qwen2.5-7B-shaped 256K workload, 2 of 4 KV heads streaming."""
    cfg = aoh.make_config(1, 28, 4, 128, 262144 + 128, 128, 4096)
    per_layer = aoh.aoh_cache_bytes(cfg, [0, 1, 1, 0])
    assert 28 * per_layer == 28 * (2 * 262272 + 2 * 4224) * 128 * 4
    full = aoh.aoh_cache_bytes(cfg, [0, 0, 0, 0])
    assert full / per_layer > 1.96


@pytest.mark.parametrize("bad", [
    dict(batch=0), dict(n_q_heads=6, n_kv_heads=4), dict(d_head=96), dict(window=0), dict(sink=-1),
    dict(max_seq=0),
])
def test_invalid_config_rejected_on_host(lib, bad):
    args = dict(batch=1, n_q_heads=8, n_kv_heads=2, d_head=64, max_seq=64, sink=4, window=8)
    args.update(bad)
    cfg = aoh.make_config(**args)
    n = lib.aoh_cache_bytes(ctypes.byref(cfg), (ctypes.c_uint8 * 4)(0, 1, 0, 1))
    assert n == 0
    assert lib.aoh_last_error().decode() != ""


def test_negative_chunk_rejected(lib):
    cfg = aoh.make_config(1, 8, 2, 64, 64, 4, 8, chunk=-1)
    assert lib.aoh_cache_bytes(ctypes.byref(cfg), (ctypes.c_uint8 * 2)(0, 1)) == 0
    assert "chunk" in lib.aoh_last_error().decode()


def test_config_struct_matches_header():
    """aoh_config is eight int32 fields, in the header's order."""
    import re
    hdr = open(os.path.join(ROOT, "include", "aoh.h")).read()
    body = re.search(r"typedef struct aoh_config \{(.*?)\} aoh_config;", hdr, re.S).group(1)
    names = re.findall(r"int32_t (\w+);", body)
    assert names == [n for n, _ in aoh.aoh_config._fields_]
    assert ctypes.sizeof(aoh.aoh_config) == 4 * len(names)


def test_classify_rejects_bad_arguments_on_host(lib):
    """Argument errors are reported before any CUDA call (no GPU needed)."""
    lab = (ctypes.c_uint8 * 2)()
    fake = ctypes.c_void_p(1 << 20)  # never dereferenced
    assert lib.aoh_classify(None, fake, 1, 8, 2, 128, 512, 50, None, lab, None) == 1
    assert lib.aoh_classify(fake, fake, 0, 8, 2, 128, 512, 50, None, lab, None) == 1
    assert lib.aoh_classify(fake, fake, 1, 8, 3, 128, 512, 50, None, lab, None) == 1
    assert lib.aoh_classify(fake, fake, 1, 8, 2, 96, 512, 50, None, lab, None) == 5
    assert lib.aoh_classify(fake, fake, 1, 8, 2, 128, 0, 50, None, lab, None) == 1
    assert lib.aoh_classify(fake, fake, 1, 8, 2, 128, 512, 101, None, lab, None) == 1
    assert lib.aoh_classify(fake, fake, 1, 8, 2, 128, 512, 50, None, None, None) == 1
    assert lib.aoh_classify(fake, fake, 5000, 8, 8, 128, 512, 50, None, lab, None) == 1  # > 65535 matrices


def test_h2share_map_rejects_bad_arguments_on_host(lib):
    lab = (ctypes.c_uint8 * 2)(0, 1)
    mp = (ctypes.c_int32 * 2)()
    fake = ctypes.c_void_p(1 << 20)  # never dereferenced
    assert lib.aoh_h2share_map(None, fake, fake, fake, 8, 2, 128, 512, lab, lab, mp, None, None) == 1
    assert lib.aoh_h2share_map(fake, fake, fake, fake, 8, 3, 128, 512, lab, lab, mp, None, None) == 1
    assert lib.aoh_h2share_map(fake, fake, fake, fake, 8, 2, 96, 512, lab, lab, mp, None, None) == 5
    assert lib.aoh_h2share_map(fake, fake, fake, fake, 8, 2, 128, 500, lab, lab, mp, None, None) == 1
    bad = (ctypes.c_uint8 * 2)(0, 2)
    assert lib.aoh_h2share_map(fake, fake, fake, fake, 8, 2, 128, 512, bad, lab, mp, None, None) == 1


def test_bad_label_rejected(lib):
    cfg = aoh.make_config(1, 8, 2, 64, 64, 4, 8)
    assert lib.aoh_cache_bytes(ctypes.byref(cfg), (ctypes.c_uint8 * 2)(0, 2)) == 0
    assert "neither" in lib.aoh_last_error().decode()


def test_init_rejects_null_and_small_buffers_before_any_cuda_call(lib):
    cfg = aoh.make_config(1, 8, 2, 64, 64, 4, 8)
    labels = (ctypes.c_uint8 * 2)(0, 1)
    h = ctypes.c_void_p()
    assert lib.aoh_cache_init(ctypes.byref(cfg), labels, None, 1 << 20, ctypes.byref(h)) == 1
    fake = ctypes.c_void_p(1 << 20)  # never dereferenced: the size check fails first
    assert lib.aoh_cache_init(ctypes.byref(cfg), labels, fake, 16, ctypes.byref(h)) == 2
    misaligned = ctypes.c_void_p((1 << 20) + 16)
    assert lib.aoh_cache_init(ctypes.byref(cfg), labels, misaligned, 1 << 30, ctypes.byref(h)) == 1
    unsupported = aoh.make_config(1, 12, 2, 64, 64, 4, 8)  # group of 6 is not compiled
    assert lib.aoh_cache_init(ctypes.byref(unsupported), labels, fake, 1 << 30, ctypes.byref(h)) == 5


def test_null_handle_calls_fail_cleanly(lib):
    assert lib.aoh_prefill(None, None, None, 1, None, None, None, None) == 1
    assert lib.aoh_decode_step(None, None, None, None, None, None) == 1
    assert lib.aoh_cache_check(None, None) == 1
    lib.aoh_cache_destroy(None)


def test_every_export_has_a_ctypes_signature(lib):
    """A function without argtypes would have its pointer arguments passed as
    C ints (truncated on a 64-bit host)."""
    for name in aoh.EXPORTS:
        fn = getattr(lib, name)
        assert fn.argtypes is not None, name


def test_ctypes_signatures_match_the_header_arity(lib):
    text = re.sub(r"/\*.*?\*/", "", open(HEADER).read(), flags=re.S)
    decls = dict(re.findall(r"\b(aoh_[a-z0-9_]+)\s*\(([^;{]*?)\)\s*;", text))
    assert sorted(decls) == sorted(aoh.EXPORTS)
    for name, params in decls.items():
        params = " ".join(params.split())
        n = 0 if params in ("", "void") else params.count(",") + 1
        assert len(getattr(lib, name).argtypes) == n, (name, params)


def test_ctypes_argument_types_match_the_header(lib):
    """Pointers are passed as pointers and integers at their declared width."""
    text = re.sub(r"/\*.*?\*/", "", open(HEADER).read(), flags=re.S)
    decls = dict(re.findall(r"\b(aoh_[a-z0-9_]+)\s*\(([^;{]*?)\)\s*;", text))
    scalars = {"int32_t": ctypes.c_int32, "int64_t": ctypes.c_int64, "size_t": ctypes.c_size_t}
    for name, params in decls.items():
        params = " ".join(params.split())
        if params in ("", "void"):
            continue
        for decl, t in zip(params.split(","), getattr(lib, name).argtypes):
            if "*" in decl:
                assert t is ctypes.c_void_p or issubclass(t, ctypes._Pointer), (name, decl, t)
            else:
                base = [k for k in scalars if re.search(rf"\b{k}\b", decl)]
                assert base and t is scalars[base[0]], (name, decl, t)


def test_ctypes_return_types_match_the_header(lib):
    text = re.sub(r"/\*.*?\*/", "", open(HEADER).read(), flags=re.S)
    rets = dict((n, r.strip()) for r, n in re.findall(r"(?m)^([A-Za-z_][A-Za-z0-9_ ]*\**)\s*\b(aoh_[a-z0-9_]+)\s*\(",
                                                    text))
    assert sorted(rets) == sorted(aoh.EXPORTS)
    want = {"aoh_status": ctypes.c_int32, "int32_t": ctypes.c_int32, "size_t": ctypes.c_size_t,
            "const char*": ctypes.c_char_p, "void": None}
    for name, ret in rets.items():
        assert getattr(lib, name).restype is want[ret], (name, ret)
