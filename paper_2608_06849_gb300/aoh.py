"""ctypes binding of ``libaoh.so`` (the C ABI in ``include/aoh.h``).

Argument marshalling only: every step of the attention path runs in the
library's CUDA kernels. The functions carry the C names; torch tensors are
passed as raw device pointers plus the current CUDA stream. There is no
fallback: if the library is missing or fails to load, every call raises.

``Cache`` is a small convenience owner of a KV buffer (a torch uint8 device
tensor) and its handle. Its methods, ``aoh_decode_step_noalloc``,
``aoh_classify`` and ``aoh_h2share_map`` check tensor sizes against the
configuration; the handle-level functions (``aoh_prefill``,
``aoh_decode_step`` ...) pass the pointers on unchecked, as the C ABI does.
"""

import ctypes
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libaoh.so")

AOH_OK = 0
STATUS_NAMES = {0: "OK", 1: "INVALID", 2: "CAPACITY", 3: "CUDA", 4: "TIMEOUT", 5: "UNSUPPORTED", 6: "STATE"}
RETRIEVAL = 0
STREAMING = 1

EXPORTS = [
    "aoh_cache_bytes",
    "aoh_cache_init",
    "aoh_prefill",
    "aoh_decode_step",
    "aoh_cache_lens",
    "aoh_cache_region",
    "aoh_cache_reset",
    "aoh_cache_reserve",
    "aoh_cache_check",
    "aoh_cache_destroy",
    "aoh_last_error",
    "aoh_version",
    "aoh_decode_step_noalloc",
    "aoh_decode_step_noalloc_status",
    "aoh_decode_step_noalloc_selftest",
    "aoh_classify",
    "aoh_decode_step_anchor",
    "aoh_decode_step_reuse",
    "aoh_cache_selftest_wait",
    "aoh_h2share_map",
]


class AohError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__(f"aoh status {STATUS_NAMES.get(status, status)}: {msg}")
        self.status = status


class aoh_config(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in
                ("batch", "n_q_heads", "n_kv_heads", "d_head", "max_seq", "sink", "window", "chunk")]


_lib = None


def load():
    """Load ``libaoh.so`` once; raise if it is absent (no CPU fallback)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing: build it with paper_2608_06849_gb300.build.build()")
    lib = ctypes.CDLL(LIB_PATH)
    P = ctypes.c_void_p
    i32 = ctypes.c_int32
    cfgp = ctypes.POINTER(aoh_config)
    u8p = ctypes.POINTER(ctypes.c_uint8)
    i32p = ctypes.POINTER(ctypes.c_int32)
    szp = ctypes.POINTER(ctypes.c_size_t)
    sig = {
        "aoh_cache_bytes": (ctypes.c_size_t, [cfgp, u8p]),
        "aoh_cache_init": (i32, [cfgp, u8p, P, ctypes.c_size_t, ctypes.POINTER(P)]),
        "aoh_prefill": (i32, [P, P, P, i32, i32p, P, P, P]),
        "aoh_decode_step": (i32, [P, P, P, P, P, P]),
        "aoh_decode_step_anchor": (i32, [P, P, P, P, P, i32, P, P]),
        "aoh_decode_step_reuse": (i32, [P, P, P, P, P, P, i32, i32, i32p, P]),
        "aoh_cache_lens": (i32, [P, i32p]),
        "aoh_cache_region": (i32, [P, i32, i32, szp, szp, i32p]),
        "aoh_cache_reset": (i32, [P, P]),
        "aoh_cache_reserve": (i32, [P, i32, i32]),
        "aoh_cache_check": (i32, [P, P]),
        "aoh_h2share_map": (i32, [P, P, P, P, i32, i32, i32, i32, u8p, u8p, i32p,
                                  ctypes.POINTER(ctypes.c_double), P]),
        "aoh_cache_selftest_wait": (i32, [P, ctypes.c_int64, ctypes.POINTER(ctypes.c_int64), P]),
        "aoh_cache_destroy": (None, [P]),
        "aoh_last_error": (ctypes.c_char_p, []),
        "aoh_version": (i32, []),
        "aoh_decode_step_noalloc": (i32, [cfgp, u8p, P, i32p, i32, P, P, P, P, P]),
        "aoh_decode_step_noalloc_status": (i32, [ctypes.POINTER(ctypes.c_uint32), P]),
        "aoh_decode_step_noalloc_selftest": (i32, [cfgp, u8p, P, i32p, i32, P, P, P, P, P]),
        "aoh_classify": (i32, [P, P, i32, i32, i32, i32, i32, i32, ctypes.POINTER(ctypes.c_double), u8p, P]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib


def _check(status):
    if status != AOH_OK:
        raise AohError(status, load().aoh_last_error().decode())


def _labels_arr(labels):
    return (ctypes.c_uint8 * len(labels))(*[int(x) for x in labels])


def make_config(batch, n_q_heads, n_kv_heads, d_head, max_seq, sink, window, chunk=0):
    """chunk = 0: per-token streaming window; K > 0: streaming prefill rows
    evict after each K-token chunk (aoh_config.chunk)."""
    return aoh_config(batch, n_q_heads, n_kv_heads, d_head, max_seq, sink, window, chunk)


def _stream_ptr(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _ptr(t, name, dtype=torch.bfloat16):
    if t is None:
        return None
    if not t.is_cuda or t.dtype != dtype or not t.is_contiguous():
        raise ValueError(f"{name} must be a contiguous {dtype} CUDA tensor")
    return ctypes.c_void_p(t.data_ptr())


# ----------------------------------------------------------------- C names

def aoh_version():
    return load().aoh_version()


def aoh_cache_bytes(cfg, labels):
    n = load().aoh_cache_bytes(ctypes.byref(cfg), _labels_arr(labels))
    if n == 0:
        raise AohError(1, load().aoh_last_error().decode())
    return n


def aoh_cache_init(cfg, labels, kv_buffer):
    """kv_buffer: a CUDA uint8 tensor of at least aoh_cache_bytes() bytes."""
    h = ctypes.c_void_p()
    _check(load().aoh_cache_init(ctypes.byref(cfg), _labels_arr(labels), _ptr(kv_buffer, "kv_buffer", torch.uint8),
                                 kv_buffer.numel(), ctypes.byref(h)))
    return h


def aoh_prefill(q, k, v, T, seq_lens, cache, out, stream=None):
    lens = None if seq_lens is None else (ctypes.c_int32 * len(seq_lens))(*[int(x) for x in seq_lens])
    _check(load().aoh_prefill(_ptr(q, "q"), _ptr(k, "k"), _ptr(v, "v"), int(T), lens, cache,
                              _ptr(out, "out"), _stream_ptr(stream)))


def aoh_decode_step(q, k_new, v_new, cache, out, stream=None):
    _check(load().aoh_decode_step(_ptr(q, "q"), _ptr(k_new, "k_new"), _ptr(v_new, "v_new"), cache,
                                  _ptr(out, "out"), _stream_ptr(stream)))


def aoh_decode_step_anchor(q, k_new, v_new, cache, out, top_k, indices, stream=None):
    """H2Share anchor step; indices: contiguous int32 CUDA tensor [B, n_r, top_k]."""
    _check(load().aoh_decode_step_anchor(_ptr(q, "q"), _ptr(k_new, "k_new"), _ptr(v_new, "v_new"), cache,
                                         _ptr(out, "out"), int(top_k), _ptr(indices, "indices", torch.int32),
                                         _stream_ptr(stream)))


def aoh_decode_step_reuse(q, k_new, v_new, cache, out, indices, top_k, group_map, stream=None):
    """H2Share reuse step; indices [B, n_anchor_groups, top_k] int32 CUDA tensor
    from the anchor step (None when the layer has no retrieval head);
    group_map: host list, one anchor group per retrieval KV head of this
    layer."""
    gm = (ctypes.c_int32 * max(1, len(group_map)))(*[int(x) for x in group_map])
    n_anchor = int(indices.shape[1]) if indices is not None else 1
    _check(load().aoh_decode_step_reuse(_ptr(q, "q"), _ptr(k_new, "k_new"), _ptr(v_new, "v_new"), cache,
                                        _ptr(out, "out"), _ptr(indices, "indices", torch.int32),
                                        n_anchor, int(top_k), gm, _stream_ptr(stream)))


def aoh_decode_step_noalloc(cfg, labels, kv_buffer, lens, max_len, q, k_new, v_new, out, stream=None,
                            _selftest=False):
    """The allocation-free decode step: ``kv_buffer`` (CUDA uint8) and ``lens``
    (CUDA int32 [B], advanced by one on the device) belong to the caller.
    ``_selftest`` calls aoh_decode_step_noalloc_selftest instead."""
    if len(labels) != cfg.n_kv_heads:
        raise ValueError(f"labels need {cfg.n_kv_heads} entries (one per KV head)")
    n_s = sum(1 for x in labels if int(x) == STREAMING)
    n_r = len(labels) - n_s
    _need(kv_buffer, "kv_buffer", cfg.batch * (n_r * cfg.max_seq + n_s * (cfg.sink + cfg.window)) * cfg.d_head * 4)
    _need(lens, "lens", cfg.batch)
    nq, nkv = cfg.batch * cfg.n_q_heads * cfg.d_head, cfg.batch * cfg.n_kv_heads * cfg.d_head
    for t, name, n in ((q, "q", nq), (k_new, "k_new", nkv), (v_new, "v_new", nkv), (out, "out", nq)):
        _need(t, name, n)
    if not lens.is_cuda or lens.dtype != torch.int32 or not lens.is_contiguous():
        raise ValueError("lens must be a contiguous int32 CUDA tensor")
    fn = load().aoh_decode_step_noalloc_selftest if _selftest else load().aoh_decode_step_noalloc
    _check(fn(
        ctypes.byref(cfg), _labels_arr(labels), _ptr(kv_buffer, "kv_buffer", torch.uint8),
        ctypes.cast(ctypes.c_void_p(lens.data_ptr()), ctypes.POINTER(ctypes.c_int32)), int(max_len),
        _ptr(q, "q"), _ptr(k_new, "k_new"), _ptr(v_new, "v_new"), _ptr(out, "out"), _stream_ptr(stream)))


def aoh_decode_step_noalloc_status(stream=None):
    """Read and clear the allocation-free decode's sticky status word on the
    current device (after synchronising ``stream``). Returns
    ``(status, flags)``: status is AOH_OK, 4 (TIMEOUT) or 2 (CAPACITY);
    flags holds bit 1 (a bounded wait ran out) and bit 2 (a step found a
    sequence already holding max_seq tokens). Does not raise on those."""
    flags = ctypes.c_uint32(0)
    st = load().aoh_decode_step_noalloc_status(ctypes.byref(flags), _stream_ptr(stream))
    if st not in (AOH_OK, 2, 4):
        _check(st)
    return st, flags.value


def aoh_classify(w_q, w_k, n_kv_heads, sparsity_pct, stream=None):
    """Effective-rank labels. w_q [L, Hq, d_head, d_model] and w_k
    [L, Hkv, d_head, d_model] (or one layer without the leading L) are
    contiguous bf16 CUDA tensors. Returns (labels, er): per layer a list of
    n_kv_heads labels and a list of n_q_heads ER values (one layer: the
    lists themselves)."""
    single = w_q.dim() == 3
    if single:
        w_q, w_k = w_q.unsqueeze(0), w_k.unsqueeze(0)
    L, Hq, dh, dm = w_q.shape
    if tuple(w_k.shape) != (L, n_kv_heads, dh, dm):
        raise ValueError("w_k must be [layers, n_kv_heads, d_head, d_model] like w_q")
    er = (ctypes.c_double * (L * Hq))()
    lab = (ctypes.c_uint8 * (L * n_kv_heads))()
    _check(load().aoh_classify(_ptr(w_q, "w_q"), _ptr(w_k, "w_k"), L, Hq, n_kv_heads, dh, dm, int(sparsity_pct),
                               er, lab, _stream_ptr(stream)))
    labels = [list(lab[l * n_kv_heads:(l + 1) * n_kv_heads]) for l in range(L)]
    ers = [list(er[l * Hq:(l + 1) * Hq]) for l in range(L)]
    return (labels[0], ers[0]) if single else (labels, ers)


def aoh_h2share_map(w_q_anchor, w_k_anchor, w_q_reuse, w_k_reuse, anchor_labels, reuse_labels, stream=None):
    """Group mapping of a reuse layer onto an anchor layer. Weights: bf16 CUDA
    tensors [Hq, d_head, d_model] / [Hkv, d_head, d_model]. Returns (map, sim):
    map[r] = anchor group of reuse group r (-1 if streaming), sim [Hkv][Hkv]
    anchor-major group similarities."""
    Hq, dh, dm = w_q_anchor.shape
    Hkv = w_k_anchor.shape[0]
    for t, name, shape in ((w_k_anchor, "w_k_anchor", (Hkv, dh, dm)), (w_q_reuse, "w_q_reuse", (Hq, dh, dm)),
                           (w_k_reuse, "w_k_reuse", (Hkv, dh, dm))):
        if tuple(t.shape) != shape:
            raise ValueError(f"{name} has shape {tuple(t.shape)}; expected {shape}")
    if len(anchor_labels) != Hkv or len(reuse_labels) != Hkv:
        raise ValueError(f"anchor_labels and reuse_labels need {Hkv} entries (one per KV head)")
    mp = (ctypes.c_int32 * Hkv)()
    sim = (ctypes.c_double * (Hkv * Hkv))()
    _check(load().aoh_h2share_map(_ptr(w_q_anchor, "w_q_anchor"), _ptr(w_k_anchor, "w_k_anchor"),
                                  _ptr(w_q_reuse, "w_q_reuse"), _ptr(w_k_reuse, "w_k_reuse"), Hq, Hkv, dh, dm,
                                  _labels_arr(anchor_labels), _labels_arr(reuse_labels), mp, sim,
                                  _stream_ptr(stream)))
    return list(mp), [list(sim[a * Hkv:(a + 1) * Hkv]) for a in range(Hkv)]


def reuse_group_map(head_map, anchor_labels, reuse_labels):
    """The group_map of aoh_decode_step_reuse from a mapping head_map[r] =
    anchor KV group (aoh_h2share_map): for each reuse retrieval group in
    increasing order, the slot of its anchor group among the anchor's
    retrieval groups (the order of the anchor step's index lists)."""
    slots = {a: i for i, a in enumerate(h for h, l in enumerate(anchor_labels) if int(l) == 0)}
    out = []
    for r, l in enumerate(reuse_labels):
        if int(l) != 0:
            continue
        a = int(head_map[r])
        if a not in slots:
            raise ValueError(f"reuse retrieval group {r} maps to {a}, not an anchor retrieval group")
        out.append(slots[a])
    return out


def aoh_cache_lens(cache, batch):
    arr = (ctypes.c_int32 * batch)()
    _check(load().aoh_cache_lens(cache, arr))
    return list(arr)


def aoh_cache_region(cache, b, kv_head):
    ko, vo, cap = ctypes.c_size_t(), ctypes.c_size_t(), ctypes.c_int32()
    _check(load().aoh_cache_region(cache, int(b), int(kv_head), ctypes.byref(ko), ctypes.byref(vo),
                                   ctypes.byref(cap)))
    return ko.value, vo.value, cap.value


def aoh_cache_reset(cache, stream=None):
    _check(load().aoh_cache_reset(cache, _stream_ptr(stream)))


def aoh_cache_reserve(cache, max_tokens, anchor_workspace=False):
    """Allocate the prefill work list for chunks of up to max_tokens tokens
    and, optionally, the H2Share anchor workspace, so later calls within
    those limits allocate nothing."""
    _check(load().aoh_cache_reserve(cache, int(max_tokens), 1 if anchor_workspace else 0))


def aoh_cache_check(cache, stream=None):
    _check(load().aoh_cache_check(cache, _stream_ptr(stream)))


def aoh_cache_selftest_wait(cache, limit_ns, stream=None):
    """Run the bounded-wait self-test; returns the wait's duration in ns."""
    el = ctypes.c_int64()
    _check(load().aoh_cache_selftest_wait(cache, int(limit_ns), ctypes.byref(el), _stream_ptr(stream)))
    return el.value


def aoh_cache_destroy(cache):
    load().aoh_cache_destroy(cache)


# ------------------------------------------------------------- convenience

def _need(t, name, n):
    """The kernels read or write the first ``n`` elements behind a pointer;
    a smaller tensor would send them past its end, so it is refused here
    (the C ABI receives bare pointers and cannot check sizes)."""
    if t is not None and t.numel() < n:
        raise ValueError(f"{name} holds {t.numel()} elements; this call needs {n}")


class Cache:
    """A KV buffer on the current CUDA device plus its library handle.

    Its methods check every tensor's element count against the cache's
    configuration before calling the library."""

    def __init__(self, batch, n_q_heads, n_kv_heads, d_head, max_seq, sink, window, labels, device=None, chunk=0):
        self.cfg = make_config(batch, n_q_heads, n_kv_heads, d_head, max_seq, sink, window, chunk)
        self.labels = [int(x) for x in labels]
        self.nbytes = aoh_cache_bytes(self.cfg, self.labels)
        self.buffer = torch.empty(self.nbytes, dtype=torch.uint8, device=device or "cuda")
        self.handle = aoh_cache_init(self.cfg, self.labels, self.buffer)
        self.batch, self.n_q_heads, self.n_kv_heads, self.d_head = batch, n_q_heads, n_kv_heads, d_head
        self.max_seq, self.sink, self.window, self.chunk = max_seq, sink, window, chunk

    def _check_step(self, q, k_new, v_new, out):
        nq = self.batch * self.n_q_heads * self.d_head
        nkv = self.batch * self.n_kv_heads * self.d_head
        for t, name, n in ((q, "q", nq), (k_new, "k_new", nkv), (v_new, "v_new", nkv), (out, "out", nq)):
            _need(t, name, n)

    def prefill(self, q, k, v, out=None, seq_lens=None, stream=None):
        """q, out [B, T, Hq, d] (both may be None: append only); k, v [B, T, Hkv, d]."""
        T = k.shape[1]
        nq = self.batch * T * self.n_q_heads * self.d_head
        nkv = self.batch * T * self.n_kv_heads * self.d_head
        for t, name, n in ((q, "q", nq), (k, "k", nkv), (v, "v", nkv), (out, "out", nq)):
            _need(t, name, n)
        if seq_lens is not None and len(seq_lens) != self.batch:
            raise ValueError(f"seq_lens has {len(seq_lens)} entries; the cache holds {self.batch} sequences")
        aoh_prefill(q, k, v, T, seq_lens, self.handle, out, stream)

    def decode_step(self, q, k_new, v_new, out, stream=None):
        """q, out [B, Hq, d]; k_new, v_new [B, Hkv, d]."""
        self._check_step(q, k_new, v_new, out)
        aoh_decode_step(q, k_new, v_new, self.handle, out, stream)

    def decode_step_anchor(self, q, k_new, v_new, out, top_k, indices, stream=None):
        """As decode_step; indices [B, n_retrieval, top_k] receives the selection."""
        self._check_step(q, k_new, v_new, out)
        n_r = sum(1 for x in self.labels if x == RETRIEVAL)
        _need(indices, "indices", self.batch * n_r * max(0, int(top_k)))
        aoh_decode_step_anchor(q, k_new, v_new, self.handle, out, top_k, indices, stream)

    def decode_step_reuse(self, q, k_new, v_new, out, indices, top_k, group_map, stream=None):
        """As decode_step; indices [B, n_anchor_groups, top_k] from an anchor step."""
        self._check_step(q, k_new, v_new, out)
        if indices is not None:
            if indices.dim() != 3 or indices.shape[0] != self.batch:
                raise ValueError("indices must be [batch, n_anchor_groups, top_k]")
            _need(indices, "indices", self.batch * int(indices.shape[1]) * max(0, int(top_k)))
        aoh_decode_step_reuse(q, k_new, v_new, self.handle, out, indices, top_k, group_map, stream)

    def lens(self):
        return aoh_cache_lens(self.handle, self.batch)

    def region(self, b, kv_head):
        """(K rows, V rows) of (b, kv_head) as bf16 views [capacity, d_head] of the buffer."""
        ko, vo, cap = aoh_cache_region(self.handle, b, kv_head)
        nb = cap * self.d_head * 2
        kr = self.buffer[ko:ko + nb].view(torch.bfloat16).view(cap, self.d_head)
        vr = self.buffer[vo:vo + nb].view(torch.bfloat16).view(cap, self.d_head)
        return kr, vr

    def reset(self, stream=None):
        aoh_cache_reset(self.handle, stream)

    def reserve(self, max_tokens, anchor_workspace=False):
        aoh_cache_reserve(self.handle, max_tokens, anchor_workspace)

    def check(self, stream=None):
        aoh_cache_check(self.handle, stream)

    def close(self):
        if getattr(self, "handle", None):
            aoh_cache_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
