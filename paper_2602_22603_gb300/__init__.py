"""Python binding of libsq: the GB300 hot path of SideQuest's KV-cache
management (paged GQA decode attention over copy-on-write prefix pages, and
span eviction by in-place compaction).

Argument marshalling only: every step runs in the CUDA library
(_build/libsq.so, built by `build.build_all()`).  There is no CPU fallback:
if the library is missing, importing the binding's functions raises.

Functions carry the C names of include/sq.h.  Device buffers may be given as
torch CUDA tensors or raw integer addresses; streams as torch.cuda.Stream,
raw cudaStream_t integers, or None (torch's current stream).
"""
from __future__ import annotations

import ctypes
import os
import threading
from typing import Iterable, List, Optional, Sequence, Tuple

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "libsq.so")

SQ_OK = 0
SQ_ERR_INVALID_ARG = -1
SQ_ERR_BAD_HANDLE = -2
SQ_ERR_NO_PAGES = -3
SQ_ERR_CAPACITY = -4
SQ_ERR_CUDA = -5
SQ_ERR_DEVICE = -6
SQ_ERR_DEVICE_TIMEOUT = -7
SQ_ERR_UNSUPPORTED = -8
SQ_ERR_NO_MEMORY = -9
SQ_OUT_BF16 = 0
SQ_OUT_F32 = 1
SQ_DEBUG_DROP_DECODE_STAGE = 1


class sq_config(ctypes.Structure):
    _fields_ = [
        ("num_layers", ctypes.c_int32),
        ("num_q_heads", ctypes.c_int32),
        ("num_kv_heads", ctypes.c_int32),
        ("head_dim", ctypes.c_int32),
        ("page_size", ctypes.c_int32),
        ("num_pages", ctypes.c_int32),
        ("max_seqs", ctypes.c_int32),
        ("max_pages_per_seq", ctypes.c_int32),
        ("kv_pool", ctypes.c_void_p),
        ("decode_ctas", ctypes.c_int32),
    ]


class sq_span(ctypes.Structure):
    _fields_ = [("start", ctypes.c_int32), ("end", ctypes.c_int32)]


class sq_stats_t(ctypes.Structure):
    _fields_ = [(name, ctypes.c_int64) for name in (
        "live_pages", "peak_live_pages", "decode_calls", "decode_logical_bytes",
        "decode_unique_bytes", "evict_calls", "evicted_tokens", "evict_moved_rows",
        "evict_bytes", "appended_tokens", "cow_pages", "prefill_calls", "prefill_pairs",
        "decode_early_calls", "decode_early_held", "decode_plans_built")]

    def as_dict(self):
        return {name: int(getattr(self, name)) for name, _ in self._fields_}


class SqError(RuntimeError):
    def __init__(self, code: int, call: str):
        self.code = code
        super().__init__(f"{call} failed: {strerror(code)} ({code})")


_lib = None
_lock = threading.Lock()

_P = ctypes.c_void_p
_I32 = ctypes.c_int32
_I32P = ctypes.POINTER(ctypes.c_int32)
_SIGS = {
    "sq_pool_bytes": (ctypes.c_size_t, [ctypes.POINTER(sq_config)]),
    "sq_cache_create": (ctypes.c_int, [ctypes.POINTER(sq_config), ctypes.POINTER(_P)]),
    "sq_cache_destroy": (ctypes.c_int, [_P]),
    "sq_seq_new": (ctypes.c_int, [_P, _I32P]),
    "sq_append_kv": (ctypes.c_int, [_P, _I32, _I32, _P, _P, _P]),
    "sq_fork_aux": (ctypes.c_int, [_P, _I32, _I32P]),
    "sq_append_kv_batch": (ctypes.c_int, [_P, _I32P, _I32, _P, _P, _P]),
    "sq_decode_attention": (ctypes.c_int, [_P, _I32P, _I32, _I32, _P, _P, _I32, ctypes.c_float, _P]),
    "sq_evict_spans": (ctypes.c_int, [_P, _I32, ctypes.POINTER(sq_span), _I32, _P]),
    "sq_evict_spans_ragged": (ctypes.c_int, [_P, _I32, ctypes.POINTER(sq_span), _I32, _P]),
    "sq_prefill_attention": (ctypes.c_int, [_P, _I32, _I32, _I32, _P, _P, _I32, _P, ctypes.c_float,
                                            ctypes.POINTER(sq_span), _I32, _P]),
    "sq_release": (ctypes.c_int, [_P, _I32, _P]),
    "sq_seq_info": (ctypes.c_int, [_P, _I32, _I32P, _I32P]),
    "sq_seq_next_pos": (ctypes.c_int, [_P, _I32, ctypes.POINTER(ctypes.c_int64)]),
    "sq_get_page_table": (ctypes.c_int, [_P, _I32, _I32P, _I32, _I32P]),
    "sq_get_page_fill": (ctypes.c_int, [_P, _I32, _I32P, _I32, _I32P]),
    "sq_page_refcount": (ctypes.c_int, [_P, _I32, _I32P]),
    "sq_free_pages": (ctypes.c_int, [_P, _I32P]),
    "sq_pool_ptr": (ctypes.c_int, [_P, ctypes.POINTER(_P)]),
    "sq_stats": (ctypes.c_int, [_P, ctypes.POINTER(sq_stats_t)]),
    "sq_sync_status": (ctypes.c_int, [_P, _P]),
    "sq_strerror": (ctypes.c_char_p, [ctypes.c_int]),
    "sq_probe_read": (ctypes.c_int, [_P, _P, ctypes.c_size_t, _P]),
    "sq_debug_set": (ctypes.c_int, [_P, _I32]),
    "sq_decode_attention_noalloc": (ctypes.c_int, [_P, _I32P, _I32, _I32, _P, _P, _I32,
                                                   ctypes.c_float, _P]),
}


def lib() -> ctypes.CDLL:
    """The loaded libsq.so.  Raises if it has not been built."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIB_PATH):
                raise RuntimeError(
                    f"libsq.so not found at {LIB_PATH}: build it with "
                    "`python -m paper_2602_22603_gb300.build` (needs nvcc)")
            L = ctypes.CDLL(LIB_PATH)
            for name, (res, args) in _SIGS.items():
                f = getattr(L, name)
                f.restype = res
                f.argtypes = args
            _lib = L
    return _lib


def strerror(code: int) -> str:
    return lib().sq_strerror(int(code)).decode()


sq_strerror = strerror


def _check(rc: int, call: str) -> None:
    if rc != SQ_OK:
        raise SqError(rc, call)


def _ptr(x) -> Optional[int]:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return int(x.data_ptr())


def _stream(s) -> Optional[int]:
    if s is None:
        import torch
        return int(torch.cuda.current_stream().cuda_stream)
    if isinstance(s, int):
        return s
    return int(s.cuda_stream)


# ---- the C calls ------------------------------------------------------------
def make_config(num_layers, num_q_heads, num_kv_heads, head_dim, page_size, num_pages,
                max_seqs=64, max_pages_per_seq=None, kv_pool=None, decode_ctas=0) -> sq_config:
    return sq_config(num_layers, num_q_heads, num_kv_heads, head_dim, page_size, num_pages,
                     max_seqs, max_pages_per_seq or num_pages, _ptr(kv_pool), decode_ctas)


def sq_pool_bytes(cfg: sq_config) -> int:
    return int(lib().sq_pool_bytes(ctypes.byref(cfg)))


def sq_cache_create(cfg: sq_config) -> int:
    out = _P()
    _check(lib().sq_cache_create(ctypes.byref(cfg), ctypes.byref(out)), "sq_cache_create")
    return out.value


def sq_cache_destroy(cache: int) -> None:
    _check(lib().sq_cache_destroy(cache), "sq_cache_destroy")


def sq_seq_new(cache: int) -> int:
    h = _I32()
    _check(lib().sq_seq_new(cache, ctypes.byref(h)), "sq_seq_new")
    return h.value


def sq_append_kv(cache: int, seq: int, n_tokens: int, k, v, stream=None) -> None:
    _check(lib().sq_append_kv(cache, seq, n_tokens, _ptr(k), _ptr(v), _stream(stream)),
           "sq_append_kv")


def sq_append_kv_batch(cache: int, seqs, k, v, stream=None) -> None:
    arr = seqs if isinstance(seqs, ctypes.Array) else (ctypes.c_int32 * len(seqs))(*seqs)
    _check(lib().sq_append_kv_batch(cache, arr, len(seqs), _ptr(k), _ptr(v), _stream(stream)),
           "sq_append_kv_batch")


def sq_fork_aux(cache: int, parent: int) -> int:
    h = _I32()
    _check(lib().sq_fork_aux(cache, parent, ctypes.byref(h)), "sq_fork_aux")
    return h.value


def sq_decode_attention(cache: int, seqs: Sequence[int], layer: int, q, out,
                        out_dtype: int = SQ_OUT_BF16, sm_scale: float = 1.0,
                        stream=None) -> None:
    arr = seqs if isinstance(seqs, ctypes.Array) else (ctypes.c_int32 * len(seqs))(*seqs)
    _check(lib().sq_decode_attention(cache, arr, len(seqs), layer, _ptr(q), _ptr(out),
                                     out_dtype, float(sm_scale), _stream(stream)),
           "sq_decode_attention")


def sq_decode_attention_noalloc(cache: int, seqs: Sequence[int], layer: int, q, out,
                                out_dtype: int = SQ_OUT_BF16, sm_scale: float = 1.0,
                                stream=None) -> None:
    """sq_decode_attention without any device allocation (fixed library
    scratch; see include/sq.h for the limits and the sharing rule)."""
    arr = (ctypes.c_int32 * len(seqs))(*seqs)
    _check(lib().sq_decode_attention_noalloc(cache, arr, len(seqs), layer, _ptr(q), _ptr(out),
                                             out_dtype, float(sm_scale), _stream(stream)),
           "sq_decode_attention_noalloc")


def sq_evict_spans(cache: int, seq: int, spans: Sequence[Tuple[int, int]], stream=None) -> None:
    arr = (sq_span * max(1, len(spans)))(*[sq_span(int(a), int(b)) for a, b in spans])
    _check(lib().sq_evict_spans(cache, seq, arr, len(spans), _stream(stream)), "sq_evict_spans")


def sq_evict_spans_ragged(cache: int, seq: int, spans: Sequence[Tuple[int, int]],
                          stream=None) -> None:
    arr = (sq_span * max(1, len(spans)))(*[sq_span(int(a), int(b)) for a, b in spans])
    _check(lib().sq_evict_spans_ragged(cache, seq, arr, len(spans), _stream(stream)),
           "sq_evict_spans_ragged")


def sq_prefill_attention(cache: int, seq: int, layer: int, n_q: int, q, out,
                         out_dtype: int = SQ_OUT_BF16, lse=None, sm_scale: float = 1.0,
                         spans: Sequence[Tuple[int, int]] = (), stream=None) -> None:
    arr = (sq_span * max(1, len(spans)))(*[sq_span(int(a), int(b)) for a, b in spans])
    _check(lib().sq_prefill_attention(cache, seq, layer, n_q, _ptr(q), _ptr(out), out_dtype,
                                      _ptr(lse), float(sm_scale), arr, len(spans),
                                      _stream(stream)),
           "sq_prefill_attention")


def sq_release(cache: int, seq: int, stream=None) -> None:
    _check(lib().sq_release(cache, seq, _stream(stream)), "sq_release")


def sq_seq_info(cache: int, seq: int) -> Tuple[int, int]:
    n, p = _I32(), _I32()
    _check(lib().sq_seq_info(cache, seq, ctypes.byref(n), ctypes.byref(p)), "sq_seq_info")
    return n.value, p.value


def sq_seq_next_pos(cache: int, seq: int) -> int:
    """Position of the sequence's next token (tokens ever appended; eviction
    does not lower it)."""
    x = ctypes.c_int64()
    _check(lib().sq_seq_next_pos(cache, seq, ctypes.byref(x)), "sq_seq_next_pos")
    return x.value


def sq_get_page_table(cache: int, seq: int) -> List[int]:
    _, npages = sq_seq_info(cache, seq)
    buf = (ctypes.c_int32 * max(1, npages))()
    n = _I32()
    _check(lib().sq_get_page_table(cache, seq, buf, npages, ctypes.byref(n)), "sq_get_page_table")
    return list(buf[: n.value])


def sq_get_page_fill(cache: int, seq: int) -> List[int]:
    _, npages = sq_seq_info(cache, seq)
    buf = (ctypes.c_int32 * max(1, npages))()
    n = _I32()
    _check(lib().sq_get_page_fill(cache, seq, buf, npages, ctypes.byref(n)), "sq_get_page_fill")
    return list(buf[: n.value])


def sq_page_refcount(cache: int, page: int) -> int:
    out = _I32()
    _check(lib().sq_page_refcount(cache, page, ctypes.byref(out)), "sq_page_refcount")
    return out.value


def sq_free_pages(cache: int) -> int:
    out = _I32()
    _check(lib().sq_free_pages(cache, ctypes.byref(out)), "sq_free_pages")
    return out.value


def sq_pool_ptr(cache: int) -> int:
    out = _P()
    _check(lib().sq_pool_ptr(cache, ctypes.byref(out)), "sq_pool_ptr")
    return out.value


def sq_stats(cache: int) -> dict:
    st = sq_stats_t()
    _check(lib().sq_stats(cache, ctypes.byref(st)), "sq_stats")
    return st.as_dict()


def sq_probe_read(cache: int, buf, nbytes: int, stream=None) -> None:
    _check(lib().sq_probe_read(cache, _ptr(buf), nbytes, _stream(stream)), "sq_probe_read")


def sq_debug_set(cache: int, flags: int) -> None:
    _check(lib().sq_debug_set(cache, flags), "sq_debug_set")


def sq_sync_status(cache: int, stream=None) -> int:
    """Synchronise the stream and return the device status code (no raise)."""
    return int(lib().sq_sync_status(cache, _stream(stream)))


# ---- a small object wrapper --------------------------------------------------
class Cache:
    """Owns one sq_cache.  Methods are the C calls with the cache bound."""

    def __init__(self, num_layers, num_q_heads, num_kv_heads, head_dim, page_size, num_pages,
                 max_seqs=64, max_pages_per_seq=None, kv_pool=None, decode_ctas=0):
        self.cfg = make_config(num_layers, num_q_heads, num_kv_heads, head_dim, page_size,
                               num_pages, max_seqs, max_pages_per_seq, kv_pool, decode_ctas)
        self._keep = kv_pool
        self.handle = sq_cache_create(self.cfg)
        self.L, self.Hq, self.Hkv = num_layers, num_q_heads, num_kv_heads
        self.D, self.P, self.num_pages = head_dim, page_size, num_pages

    def close(self):
        if self.handle:
            sq_cache_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def pool_view(self):
        """The pool as a torch bf16 tensor [L, num_pages, 2, Hkv, P, D]
        (a zero-copy view of library memory)."""
        import torch

        class _Arr:
            pass

        a = _Arr()
        shape = (self.L, self.num_pages, 2, self.Hkv, self.P, self.D)
        a.__cuda_array_interface__ = {
            "shape": shape, "typestr": "<i2", "data": (sq_pool_ptr(self.handle), False),
            "version": 3, "strides": None}
        return torch.as_tensor(a, device="cuda").view(torch.bfloat16)

    seq_new = lambda self: sq_seq_new(self.handle)
    append_kv = lambda self, seq, n, k, v, stream=None: sq_append_kv(self.handle, seq, n, k, v, stream)
    fork_aux = lambda self, parent: sq_fork_aux(self.handle, parent)
    append_kv_batch = lambda self, seqs, k, v, stream=None: sq_append_kv_batch(self.handle, seqs, k, v, stream)
    decode_attention = (lambda self, seqs, layer, q, out, out_dtype=SQ_OUT_BF16, sm_scale=1.0,
                        stream=None: sq_decode_attention(self.handle, seqs, layer, q, out,
                                                         out_dtype, sm_scale, stream))
    evict_spans = lambda self, seq, spans, stream=None: sq_evict_spans(self.handle, seq, spans, stream)
    evict_spans_ragged = (lambda self, seq, spans, stream=None:
                          sq_evict_spans_ragged(self.handle, seq, spans, stream))
    prefill_attention = (lambda self, seq, layer, n_q, q, out, out_dtype=SQ_OUT_BF16, lse=None,
                         sm_scale=1.0, spans=(), stream=None:
                         sq_prefill_attention(self.handle, seq, layer, n_q, q, out, out_dtype, lse,
                                              sm_scale, spans, stream))
    release = lambda self, seq, stream=None: sq_release(self.handle, seq, stream)
    seq_info = lambda self, seq: sq_seq_info(self.handle, seq)
    next_pos = lambda self, seq: sq_seq_next_pos(self.handle, seq)
    page_table = lambda self, seq: sq_get_page_table(self.handle, seq)
    page_fills = lambda self, seq: sq_get_page_fill(self.handle, seq)
    page_refcount = lambda self, page: sq_page_refcount(self.handle, page)
    free_pages = lambda self: sq_free_pages(self.handle)
    stats = lambda self: sq_stats(self.handle)
    sync_status = lambda self, stream=None: sq_sync_status(self.handle, stream)
