"""ctypes binding of libkvg (include/kvg.h): same names, argument marshalling only.

Every function here forwards to the C ABI; all GPU work runs in the library's
CUDA kernels.  There is no fallback: if libkvg.so has not been built the
import raises.  Tensors are passed as raw pointers (``tensor.data_ptr()``)
and streams as ``torch.cuda.Stream.cuda_stream`` integers (0 = legacy
default stream).  A non-OK status raises :class:`KvgError`.
"""
from __future__ import annotations

import ctypes
import os
import re

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "_build", "libkvg.so")
HEADER = os.path.join(os.path.dirname(_PKG), "include", "kvg.h")

KVG_OK = 0
KVG_ERR_ARG, KVG_ERR_OOM, KVG_ERR_CUDA, KVG_ERR_NOT_FOUND = -1, -2, -3, -4
KVG_ERR_CAPACITY, KVG_ERR_POSITION, KVG_ERR_DIGEST, KVG_ERR_FORMAT = -5, -6, -7, -8
KVG_ERR_TIMEOUT, KVG_ERR_DEVICE_CHECK = -9, -10
KVG_RESIDENCY_HBM, KVG_RESIDENCY_PINNED_HOST, KVG_RESIDENCY_CACHE_POOL = 0, 1, 2
KVG_ROPE_HALF, KVG_ROPE_INTERLEAVED = 0, 1
KVG_GRAFT_VERIFY, KVG_GRAFT_SYNC = 1, 2
KVG_SHA256_PLAIN, KVG_SHA256_PAGED = 0, 1
KVG_DECODE_MERGE = 1
KVG_KV_BF16, KVG_KV_E4M3 = 0, 1
KVG_REPORT_MAX_PAGES = 64


class KvgError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"kvg status {status}: {message}")
        self.status = status


class kvg_dims(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int32), ("n_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("page_size", ctypes.c_int32),
                ("rope_theta", ctypes.c_double), ("rope_style", ctypes.c_int32),
                ("kv_dtype", ctypes.c_int32), ("k_scale", ctypes.c_float), ("v_scale", ctypes.c_float)]


class kvg_block_info(ctypes.Structure):
    _fields_ = [("n_tokens", ctypes.c_int64), ("n_pages", ctypes.c_int64),
                ("residency", ctypes.c_int32), ("reserved", ctypes.c_int32),
                ("bytes", ctypes.c_void_p), ("total_bytes", ctypes.c_uint64),
                ("positions_offset", ctypes.c_uint64), ("digests_offset", ctypes.c_uint64),
                ("pages_offset", ctypes.c_uint64), ("block_digest", ctypes.c_uint8 * 32)]


class kvg_cache_view(ctypes.Structure):
    _fields_ = [("pool", ctypes.c_void_p), ("page_table", ctypes.c_void_p),
                ("page_fill", ctypes.c_void_p), ("positions", ctypes.c_void_p),
                ("pool_bytes", ctypes.c_uint64), ("page_bytes", ctypes.c_uint64),
                ("n_pages", ctypes.c_int32), ("max_seqs", ctypes.c_int32),
                ("max_slots", ctypes.c_int32), ("max_pages", ctypes.c_int32)]


class kvg_graft_report(ctypes.Structure):
    _fields_ = [("seq", ctypes.c_int32), ("n_pages_checked", ctypes.c_int32),
                ("n_mismatch", ctypes.c_int32), ("n_listed", ctypes.c_int32),
                ("mismatch_pages", ctypes.c_int32 * KVG_REPORT_MAX_PAGES)]


_vp, _i32, _i64, _u32, _u64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_uint32, ctypes.c_uint64
_P = ctypes.POINTER

_SIGNATURES = {
    "kvg_store_create": ([_P(kvg_dims), _i32, _u64, _i32, _P(_vp)], _i32),
    "kvg_store_destroy": ([_vp], None),
    "kvg_store_create_in_cache": ([_vp, _u64, _P(_vp)], _i32),
    "kvg_store_block_info": ([_vp, _u64, _P(kvg_block_info)], _i32),
    "kvg_store_import": ([_vp, _vp, _u64, _u32, _P(_u64)], _i32),
    "kvg_store_export": ([_vp, _u64, _vp, _u64], _i32),
    "kvg_store_save": ([_vp, _u64, ctypes.c_char_p], _i32),
    "kvg_store_load": ([_vp, ctypes.c_char_p, _u32, _P(_u64)], _i32),
    "kvg_store_prefetch": ([_vp, _u64, _vp], _i32),
    "kvg_cache_create": ([_P(kvg_dims), _i32, _i32, _i32, _i32, _P(_vp)], _i32),
    "kvg_cache_destroy": ([_vp], None),
    "kvg_cache_set_free_order": ([_vp, _vp, _i32], _i32),
    "kvg_cache_set_layer_windows": ([_vp, _vp, _i32], _i32),
    "kvg_graft_batch": ([_vp, _vp, _vp, _vp, _vp, _i32, _u32, _vp, _vp], _i32),
    "kvg_cache_view_get": ([_vp, _P(kvg_cache_view)], _i32),
    "kvg_cache_seq_info": ([_vp, _i32, _P(_i32), _P(_i32)], _i32),
    "kvg_cache_append": ([_vp, _i32, _vp, _vp, _vp, _i32, _vp], _i32),
    "kvg_cache_append_batch": ([_vp, _vp, _i32, _vp, _vp, _vp, _vp], _i32),
    "kvg_cache_release": ([_vp, _i32, _vp], _i32),
    "kvg_deposit": ([_vp, _vp, _i32, _i32, _i32, _vp, _P(_u64)], _i32),
    "kvg_graft": ([_vp, _u64, _vp, _i32, _i32, _i64, _u32, _vp, _P(kvg_graft_report)], _i32),
    "kvg_graft_chunked": ([_vp, _u64, _vp, _i32, _i32, _i64, _u32, _vp, _P(kvg_graft_report), _P(_vp), _i32,
                           _P(_i32), _P(_i32)], _i32),
    "kvg_verify": ([_vp, _u64, _vp, _i32, _i32, _u32, _vp, _P(kvg_graft_report)], _i32),
    "kvg_decode_attention": ([_vp, _i32, _vp, _i32, _vp, _i32, _vp, ctypes.c_float, _vp], _i32),
    "kvg_decode_attention_noalloc": ([_vp, _i32, _vp, _i32, _vp, _i32, _vp, ctypes.c_float, _vp], _i32),
    "kvg_decode_attention_range": ([_vp, _i32, _vp, _i32, _vp, _i32, ctypes.c_float, _i32, _i32, _u32, _vp, _vp],
                                   _i32),
    "kvg_decode_state_finish": ([_vp, _i64, _i32, _vp, _vp], _i32),
    "kvg_digest": ([_vp, _u64, _i32, _u64, _vp, _vp], _i32),
    "kvg_sync": ([_vp, _vp, ctypes.c_double, _P(kvg_graft_report)], _i32),
    "kvg_selftest_bounded_wait": ([_vp, _u64, _vp], _i32),
    "kvg_status_string": ([_i32], ctypes.c_char_p),
    "kvg_last_error": ([], ctypes.c_char_p),
    "kvg_version": ([], _u32),
    "kvg_launch_count": ([], _u64),
}

_lib = None


def header_functions() -> list[str]:
    """Names of the functions include/kvg.h declares."""
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(kvg_[a-z0-9_]+)\s*\(", text)))


def lib() -> ctypes.CDLL:
    """Loads the in-tree libkvg.so (raises if it was not built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"libkvg.so is not built ({LIB_PATH}); run __graft_entry__.build()")
        L = ctypes.CDLL(LIB_PATH)
        for name, (args, res) in _SIGNATURES.items():
            f = getattr(L, name)
            f.argtypes = args
            f.restype = res
        _lib = L
    return _lib


def _check(status: int):
    if status != KVG_OK:
        msg = lib().kvg_last_error().decode(errors="replace")
        raise KvgError(status, msg or lib().kvg_status_string(status).decode())


def _stream(stream) -> int:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    return int(getattr(stream, "cuda_stream", stream))


def make_dims(n_layers, n_kv_heads, head_dim, page_size, rope_theta=10000.0, rope_style=0,
              kv_dtype=KVG_KV_BF16, k_scale=1.0, v_scale=1.0) -> kvg_dims:
    return kvg_dims(n_layers, n_kv_heads, head_dim, page_size, float(rope_theta), rope_style, kv_dtype,
                    float(k_scale), float(v_scale))


# ---- thin wrappers, same names as the C ABI ---------------------------------

def kvg_store_create(dims: kvg_dims, residency: int, capacity_bytes: int, device: int = 0):
    h = _vp()
    _check(lib().kvg_store_create(ctypes.byref(dims), residency, capacity_bytes, device, ctypes.byref(h)))
    return h


def kvg_store_create_in_cache(cache, capacity_bytes: int):
    h = _vp()
    _check(lib().kvg_store_create_in_cache(cache, capacity_bytes, ctypes.byref(h)))
    return h


def kvg_store_destroy(store):
    lib().kvg_store_destroy(store)


def kvg_store_block_info(store, block_id: int) -> kvg_block_info:
    info = kvg_block_info()
    _check(lib().kvg_store_block_info(store, block_id, ctypes.byref(info)))
    return info


def kvg_store_import(store, data: bytes, flags: int = 0) -> int:
    buf = ctypes.create_string_buffer(bytes(data), len(data))
    out = _u64()
    _check(lib().kvg_store_import(store, buf, len(data), flags, ctypes.byref(out)))
    return out.value


def kvg_store_export(store, block_id: int) -> bytes:
    info = kvg_store_block_info(store, block_id)
    buf = ctypes.create_string_buffer(info.total_bytes)
    _check(lib().kvg_store_export(store, block_id, buf, info.total_bytes))
    return buf.raw


def kvg_store_save(store, block_id: int, path: str):
    _check(lib().kvg_store_save(store, block_id, os.fsencode(path)))


def kvg_store_load(store, path: str, flags: int = 0) -> int:
    out = _u64()
    _check(lib().kvg_store_load(store, os.fsencode(path), flags, ctypes.byref(out)))
    return out.value


def kvg_store_prefetch(store, block_id: int, stream=None):
    _check(lib().kvg_store_prefetch(store, block_id, _stream(stream)))


def kvg_cache_create(dims: kvg_dims, n_pages: int, max_seqs: int, max_slots: int, device: int = 0):
    h = _vp()
    _check(lib().kvg_cache_create(ctypes.byref(dims), n_pages, max_seqs, max_slots, device, ctypes.byref(h)))
    return h


def kvg_cache_destroy(cache):
    lib().kvg_cache_destroy(cache)


def kvg_cache_set_free_order(cache, order):
    arr = (ctypes.c_int32 * len(order))(*[int(x) for x in order])
    _check(lib().kvg_cache_set_free_order(cache, arr, len(order)))


def kvg_cache_set_layer_windows(cache, windows):
    """windows: one int per layer (0 = global attention), or [] to reset."""
    arr = (ctypes.c_int32 * max(len(windows), 1))(*[int(x) for x in windows])
    _check(lib().kvg_cache_set_layer_windows(cache, arr, len(windows)))


def kvg_cache_view_get(cache) -> kvg_cache_view:
    v = kvg_cache_view()
    _check(lib().kvg_cache_view_get(cache, ctypes.byref(v)))
    return v


def kvg_cache_seq_info(cache, seq: int):
    a, b = _i32(), _i32()
    _check(lib().kvg_cache_seq_info(cache, seq, ctypes.byref(a), ctypes.byref(b)))
    return a.value, b.value


def kvg_cache_append(cache, seq: int, k_ptr: int, v_ptr: int, pos_ptr: int, n: int, stream=None):
    _check(lib().kvg_cache_append(cache, seq, k_ptr, v_ptr, pos_ptr, n, _stream(stream)))


def kvg_cache_append_batch(cache, seq_ids, k_ptr: int, v_ptr: int, pos_ptr: int, stream=None):
    ids = (ctypes.c_int32 * len(seq_ids))(*[int(x) for x in seq_ids])
    _check(lib().kvg_cache_append_batch(cache, ids, len(seq_ids), k_ptr, v_ptr, pos_ptr, _stream(stream)))


def kvg_cache_release(cache, seq: int, stream=None):
    _check(lib().kvg_cache_release(cache, seq, _stream(stream)))


def kvg_deposit(store, cache, seq: int, slot0: int, n: int, stream=None) -> int:
    out = _u64()
    _check(lib().kvg_deposit(store, cache, seq, slot0, n, _stream(stream), ctypes.byref(out)))
    return out.value


def kvg_graft(store, block_id: int, cache, seq: int, dst_slot: int = -1, delta: int = 0, flags: int = 0,
              stream=None, report: kvg_graft_report | None = None):
    _check(lib().kvg_graft(store, block_id, cache, seq, dst_slot, delta, flags, _stream(stream),
                           ctypes.byref(report) if report is not None else None))


def kvg_graft_chunked(store, block_id: int, cache, seq: int, events, dst_slot: int = -1, delta: int = 0,
                      flags: int = 0, stream=None, report: kvg_graft_report | None = None):
    """kvg_graft with a completion event per chunk.  events: a list of CUDA
    event handles (ints, e.g. torch.cuda.Event().cuda_event after a record,
    or from cudaEventCreate).  Returns [chunk_end_slot[j] for j < n_chunks]:
    events[j] covers the rows of slots [dst_slot, chunk_end_slot[j])."""
    n = len(events)
    if n < 1:
        raise ValueError("at least one event")
    ev = (_vp * n)(*[int(e) for e in events])
    ends = (ctypes.c_int32 * n)()
    nc = ctypes.c_int32(0)
    _check(lib().kvg_graft_chunked(store, block_id, cache, seq, dst_slot, delta, flags, _stream(stream),
                                   ctypes.byref(report) if report is not None else None, ev, n, ends,
                                   ctypes.byref(nc)))
    return [int(ends[j]) for j in range(nc.value)]


def kvg_graft_batch(store, block_ids, cache, seq_ids, flags: int = 0, stream=None,
                    report: kvg_graft_report | None = None, deltas=None):
    """deltas: None (every graft at its own position) or one int per graft."""
    n = len(block_ids)
    if len(seq_ids) != n or (deltas is not None and len(deltas) != n):
        raise ValueError("block_ids, seq_ids and deltas differ in length")
    ids = (ctypes.c_uint64 * max(n, 1))(*[int(b) for b in block_ids])
    seqs = (ctypes.c_int32 * max(n, 1))(*[int(x) for x in seq_ids])
    ds = None if deltas is None else (ctypes.c_int64 * max(n, 1))(*[int(d) for d in deltas])
    _check(lib().kvg_graft_batch(store, ids, cache, seqs, ds, n, flags, _stream(stream),
                                 ctypes.byref(report) if report is not None else None))


def kvg_verify(store, block_id: int, cache, seq: int, slot0: int = 0, flags: int = 0, stream=None,
               report: kvg_graft_report | None = None):
    _check(lib().kvg_verify(store, block_id, cache, seq, slot0, flags, _stream(stream),
                            ctypes.byref(report) if report is not None else None))


def kvg_decode_attention(cache, layer: int, seq_ids, q_ptr: int, n_q_heads: int, out_ptr: int,
                         scale: float, stream=None):
    ids = (ctypes.c_int32 * len(seq_ids))(*[int(x) for x in seq_ids])
    _check(lib().kvg_decode_attention(cache, layer, ids, len(seq_ids), q_ptr, n_q_heads, out_ptr,
                                      float(scale), _stream(stream)))


def kvg_decode_attention_noalloc(cache, layer: int, seq_ids, q_ptr: int, n_q_heads: int, out_ptr: int,
                                 scale: float, stream=None):
    """kvg_decode_attention without any GPU allocation (static scratch; see kvg.h)."""
    ids = (ctypes.c_int32 * len(seq_ids))(*[int(x) for x in seq_ids])
    _check(lib().kvg_decode_attention_noalloc(cache, layer, ids, len(seq_ids), q_ptr, n_q_heads, out_ptr,
                                              float(scale), _stream(stream)))


def kvg_decode_attention_range(cache, layer: int, seq_ids, q_ptr: int, n_q_heads: int, scale: float,
                               slot_begin: int, slot_end: int, flags: int, state_ptr: int, stream=None):
    """Split decode over slots [slot_begin, slot_end): writes (flags 0) or merges
    (KVG_DECODE_MERGE) the fp32 softmax state [Lrun][B][Hq][D + 4] (see kvg.h)."""
    ids = (ctypes.c_int32 * len(seq_ids))(*[int(x) for x in seq_ids])
    _check(lib().kvg_decode_attention_range(cache, layer, ids, len(seq_ids), q_ptr, n_q_heads, float(scale),
                                            int(slot_begin), int(slot_end), int(flags), state_ptr, _stream(stream)))


def kvg_decode_state_finish(state_ptr: int, n_rows: int, head_dim: int, out_ptr: int, stream=None):
    """bf16 output o / l of a split decode's state rows."""
    _check(lib().kvg_decode_state_finish(state_ptr, int(n_rows), int(head_dim), out_ptr, _stream(stream)))


def kvg_digest(ptr: int, n: int, mode: int, page_bytes: int, out_ptr: int, stream=None):
    _check(lib().kvg_digest(ptr, n, mode, page_bytes, out_ptr, _stream(stream)))


def kvg_sync(cache, stream=None, timeout_s: float = 10.0, report: kvg_graft_report | None = None):
    _check(lib().kvg_sync(cache, _stream(stream), timeout_s,
                          ctypes.byref(report) if report is not None else None))


def kvg_selftest_bounded_wait(cache, limit_ns: int, stream=None):
    _check(lib().kvg_selftest_bounded_wait(cache, limit_ns, _stream(stream)))


def kvg_status_string(status: int) -> str:
    return lib().kvg_status_string(status).decode()


def kvg_last_error() -> str:
    return lib().kvg_last_error().decode()


def kvg_version() -> int:
    return lib().kvg_version()


def kvg_launch_count() -> int:
    return lib().kvg_launch_count()


# ---- owning handles ---------------------------------------------------------

class Store:
    def __init__(self, dims: kvg_dims, residency: int, capacity_bytes: int, device: int = 0):
        self.dims = dims
        self.h = kvg_store_create(dims, residency, capacity_bytes, device)

    def close(self):
        if self.h:
            kvg_store_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class PoolStore(Store):
    """A store whose blocks live in `cache`'s page pool (zero-copy graft)."""

    def __init__(self, cache: "Cache", capacity_bytes: int):
        self.dims = cache.dims
        self.h = kvg_store_create_in_cache(cache.h, capacity_bytes)


class Cache:
    def __init__(self, dims: kvg_dims, n_pages: int, max_seqs: int, max_slots: int, device: int = 0):
        self.dims = dims
        self.h = kvg_cache_create(dims, n_pages, max_seqs, max_slots, device)
        self.view = kvg_cache_view_get(self.h)

    def close(self):
        if self.h:
            kvg_cache_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
