"""CPU oracle for the KV-state graft hot path (arxiv 2607.14431).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this package.  The product library
(``paper_2607_14431_gb300``) never imports, loads or calls it, and this package
imports nothing from the product: the two share no code.

What it computes, and where the paper defines it:

* SHA-256 and the two-level page digest (``kvg_oracle.c``): the byte-exactness
  gate of Sec. 3.2 (SHA-256 of raw bytes) and the per-block digests that are
  compared across machines in Sec. 4.11.
* bf16 round-to-nearest-even, RoPE rotation by an offset (Sec. 4.2) and fp64
  grouped-query decode attention (``kvg_oracle.c``).
* ``OracleCache`` / ``OracleStore`` below: the paged KV cache and the block
  store, modelled byte for byte.  A deposit captures a sequence's KV rows and
  position tags into a block with per-page digests (Sec. 3.1, Sec. 3.3 deposit
  step); a graft installs a block at its own positions [0, N) of a fresh
  sequence (Sec. 3.2, "position consistency"), or, optionally, re-based by an
  offset with the keys re-rotated (Sec. 4.2); an append writes freshly computed
  rows (the "fresh" arm that a graft must reproduce, Sec. 3.2).

The paper keeps the block layout, the page size and the hashing scheme
closed (Sec. 3.1); the readings taken here are stated beside each function.

numpy is used only to move bytes (slicing, copying); every arithmetic step is
in the C file or written out below.
"""
from __future__ import annotations

import ctypes
import os
import struct
import subprocess
import sys
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "kvg_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_SO = os.path.join(_BUILD, "libkvg_oracle.so")
_lock = threading.Lock()
_lib = None

LEAF_BYTES = 4096          # leaf size of the two-level page digest
BLOCK_MAGIC = b"KVGBLK01"  # serialized block header magic
BLOCK_VERSION = 1
HEADER_BYTES = 256


def build(force: bool = False) -> str:
    """Compiles the C oracle with gcc (plain C11, OpenMP over independent units)."""
    os.makedirs(_BUILD, exist_ok=True)
    if not force and os.path.exists(_SO) and os.path.getmtime(_SO) >= os.path.getmtime(_SRC):
        return _SO
    tmp = _SO + f".{os.getpid()}.tmp"
    cmd = ["gcc", "-std=gnu11", "-O2", "-fPIC", "-shared", "-fopenmp", "-fno-fast-math",
           "-ffp-contract=off", _SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _SO)
    return _SO


def lib():
    global _lib
    with _lock:
        if _lib is None:
            _lib = ctypes.CDLL(build())
            L = _lib
            u8p = ctypes.POINTER(ctypes.c_uint8)
            L.ora_sha256.argtypes = [ctypes.c_void_p, ctypes.c_uint64, ctypes.c_void_p]
            L.ora_sha256.restype = None
            L.ora_sha256_constants.argtypes = [ctypes.c_void_p, ctypes.c_void_p]
            L.ora_page_digest.argtypes = [ctypes.c_void_p, ctypes.c_uint64, ctypes.c_uint64,
                                          ctypes.c_void_p]
            L.ora_page_digests.argtypes = [ctypes.c_void_p, ctypes.c_uint64, ctypes.c_uint64,
                                           ctypes.c_uint64, ctypes.c_void_p]
            L.ora_bf16_rne.argtypes = [ctypes.c_double]
            L.ora_bf16_rne.restype = ctypes.c_uint16
            L.ora_bf16_rne_array.argtypes = [ctypes.c_void_p, ctypes.c_uint64, ctypes.c_void_p]
            L.ora_bf16_to_f64.argtypes = [ctypes.c_uint16]
            L.ora_bf16_to_f64.restype = ctypes.c_double
            L.ora_rope_rotate_row.argtypes = [ctypes.c_void_p, ctypes.c_int, ctypes.c_double,
                                              ctypes.c_double, ctypes.c_int, ctypes.c_void_p]
            L.ora_rope_rotate_row_f64.argtypes = [ctypes.c_void_p, ctypes.c_int, ctypes.c_double,
                                                  ctypes.c_double, ctypes.c_int, ctypes.c_void_p]
            L.ora_rope_rotate_rows_bf16.argtypes = [ctypes.c_void_p, ctypes.c_uint64, ctypes.c_int,
                                                    ctypes.c_double, ctypes.c_double,
                                                    ctypes.c_int, ctypes.c_void_p]
            L.ora_attention_head.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
                                             ctypes.c_uint64, ctypes.c_uint64, ctypes.c_int,
                                             ctypes.c_double, ctypes.c_void_p]
            L.ora_attention_head.restype = None
            L.ora_gqa_decode.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
                                         ctypes.c_uint64, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                         ctypes.c_double, ctypes.c_void_p]
            L.ora_omp_threads.restype = ctypes.c_int
            L.ora_e4m3_to_f64.argtypes = [ctypes.c_uint8]
            L.ora_e4m3_to_f64.restype = ctypes.c_double
            L.ora_e4m3_rne_sat.argtypes = [ctypes.c_double]
            L.ora_e4m3_rne_sat.restype = ctypes.c_uint8
            L.ora_e4m3_quantize_bf16.argtypes = [ctypes.c_void_p, ctypes.c_uint64, ctypes.c_float,
                                                 ctypes.c_void_p]
            L.ora_e4m3_quantize_bf16.restype = None
            L.ora_e4m3_dequant.argtypes = [ctypes.c_void_p, ctypes.c_uint64, ctypes.c_float, ctypes.c_void_p]
            L.ora_e4m3_dequant.restype = None
            L.ora_gqa_decode_f64kv.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
                                               ctypes.c_uint64, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                               ctypes.c_double, ctypes.c_void_p]
            del u8p
        return _lib


def _ptr(a: np.ndarray) -> int:
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data


def omp_threads() -> int:
    return int(lib().ora_omp_threads())


# --------------------------------------------------------------------------
# SHA-256 and page digests
# --------------------------------------------------------------------------

def sha256(data) -> bytes:
    """FIPS 180-4 SHA-256 of a bytes-like object or a contiguous numpy array."""
    a = np.ascontiguousarray(np.frombuffer(bytes(data), np.uint8) if not isinstance(data, np.ndarray)
                             else data.reshape(-1).view(np.uint8))
    out = np.zeros(32, np.uint8)
    lib().ora_sha256(_ptr(a) if a.size else None, a.size, _ptr(out))
    return out.tobytes()


def sha256_constants():
    k = np.zeros(64, np.uint32)
    h = np.zeros(8, np.uint32)
    lib().ora_sha256_constants(_ptr(k), _ptr(h))
    return k, h


def page_digest(page, leaf_bytes: int = LEAF_BYTES) -> bytes:
    """Two-level page digest: SHA-256 over the SHA-256 digests of the page's
    consecutive leaf_bytes slices (last slice may be short)."""
    a = np.ascontiguousarray(np.asarray(page).reshape(-1).view(np.uint8))
    out = np.zeros(32, np.uint8)
    rc = lib().ora_page_digest(_ptr(a), a.size, leaf_bytes, _ptr(out))
    if rc:
        raise ValueError("page_digest: bad sizes")
    return out.tobytes()


def page_digests(pages: np.ndarray, page_bytes: int, leaf_bytes: int = LEAF_BYTES) -> np.ndarray:
    """Digests of consecutive pages of `pages` (flat bytes) -> uint8 [n_pages][32]."""
    a = np.ascontiguousarray(pages.reshape(-1).view(np.uint8))
    if a.size % page_bytes:
        raise ValueError("page_digests: size not a multiple of page_bytes")
    n = a.size // page_bytes
    out = np.zeros((n, 32), np.uint8)
    if n:
        rc = lib().ora_page_digests(_ptr(a), n, page_bytes, leaf_bytes, _ptr(out))
        if rc:
            raise ValueError("page_digests failed")
    return out


# --------------------------------------------------------------------------
# bf16, RoPE, attention
# --------------------------------------------------------------------------

def bf16_rne(x) -> np.ndarray:
    """Correctly rounded fp64 -> bf16 (ties to even); returns uint16 bits."""
    a = np.ascontiguousarray(np.asarray(x, np.float64))
    out = np.zeros(a.shape, np.uint16)
    lib().ora_bf16_rne_array(_ptr(a), a.size, _ptr(out))
    return out


def bf16_to_f64(b) -> np.ndarray:
    """bf16 bits -> exact fp64 value.

    Signalling-NaN patterns become quiet NaNs in the widening cast; numpy
    reports that as an invalid-value warning, which is expected here.
    """
    b = np.asarray(b, np.uint16)
    with np.errstate(invalid="ignore"):
        return (b.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def rope_rotate_rows(x: np.ndarray, delta: float, theta: float, style: int = 0) -> np.ndarray:
    """Rotates bf16 rows x[..., D] by `delta` positions (Sec. 4.2); fp64 result."""
    x = np.ascontiguousarray(x, np.uint16)
    D = x.shape[-1]
    flat = x.reshape(-1, D)
    out = np.zeros(flat.shape, np.float64)
    L = lib()
    for r in range(flat.shape[0]):
        rc = L.ora_rope_rotate_row(_ptr(flat[r]), D, float(delta), float(theta), style,
                                   _ptr(out[r]))
        if rc:
            raise ValueError("rope: bad D")
    return out.reshape(x.shape)


def rope_rotate_rows_f64(x: np.ndarray, delta: float, theta: float, style: int = 0) -> np.ndarray:
    x = np.ascontiguousarray(x, np.float64)
    D = x.shape[-1]
    flat = x.reshape(-1, D)
    out = np.zeros(flat.shape, np.float64)
    L = lib()
    for r in range(flat.shape[0]):
        L.ora_rope_rotate_row_f64(_ptr(flat[r]), D, float(delta), float(theta), style,
                                  _ptr(out[r]))
    return out.reshape(x.shape)


def rope_rotate_rows_bf16(x: np.ndarray, delta: float, theta: float, style: int = 0) -> np.ndarray:
    """fp64 rotation of bf16 rows, each result rounded to bf16 (RNE)."""
    x = np.ascontiguousarray(x, np.uint16)
    D = x.shape[-1]
    out = np.zeros(x.shape, np.uint16)
    rc = lib().ora_rope_rotate_rows_bf16(_ptr(x), x.size // D, D, float(delta), float(theta),
                                         style, _ptr(out))
    if rc:
        raise ValueError("rope: bad D")
    return out


def attention_head(q: np.ndarray, k: np.ndarray, v: np.ndarray, scale: float) -> np.ndarray:
    """One query head q[D] over rows k[n][D], v[n][D] (bf16 bits) -> fp64 o[D]."""
    q = np.ascontiguousarray(q, np.uint16)
    k = np.ascontiguousarray(k, np.uint16)
    v = np.ascontiguousarray(v, np.uint16)
    D = q.shape[-1]
    n = k.shape[0]
    o = np.zeros(D, np.float64)
    lib().ora_attention_head(_ptr(q), _ptr(k) if n else None, _ptr(v) if n else None, n, D, D,
                             float(scale), _ptr(o))
    return o


def e4m3_to_f64(c) -> np.ndarray:
    """Values of E4M3 codes (uint8) in fp64."""
    c = np.ascontiguousarray(c, np.uint8)
    out = np.zeros(c.shape, np.float64)
    lib().ora_e4m3_dequant(_ptr(c), c.size, 1.0, _ptr(out))
    return out


def e4m3_rne(x) -> np.ndarray:
    """fp64 values -> E4M3 codes, ties to even, saturating at +-448."""
    x = np.asarray(x, np.float64)
    return np.array([lib().ora_e4m3_rne_sat(float(v)) for v in x.reshape(-1)], np.uint8).reshape(x.shape)


def e4m3_quantize(x_bf16: np.ndarray, scale: float) -> np.ndarray:
    """bf16 bits -> E4M3 codes of fp32 value * fp32(1 / scale), the product in fp32."""
    x = np.ascontiguousarray(x_bf16, np.uint16)
    out = np.zeros(x.shape, np.uint8)
    lib().ora_e4m3_quantize_bf16(_ptr(x), x.size, float(scale), _ptr(out))
    return out


def e4m3_dequant(c: np.ndarray, scale: float) -> np.ndarray:
    """E4M3 codes -> code value * scale in fp64."""
    c = np.ascontiguousarray(c, np.uint8)
    out = np.zeros(c.shape, np.float64)
    lib().ora_e4m3_dequant(_ptr(c), c.size, float(scale), _ptr(out))
    return out


def gqa_decode_f64kv(q: np.ndarray, k: np.ndarray, v: np.ndarray, scale: float) -> np.ndarray:
    """gqa_decode with k/v given as fp64 values [n][Hkv][D] (dequantized rows)."""
    q = np.ascontiguousarray(q, np.uint16)
    k = np.ascontiguousarray(k, np.float64)
    v = np.ascontiguousarray(v, np.float64)
    Hq, D = q.shape
    n, Hkv, D2 = k.shape
    assert D2 == D and v.shape == k.shape
    o = np.zeros((Hq, D), np.float64)
    rc = lib().ora_gqa_decode_f64kv(_ptr(q), _ptr(k) if n else None, _ptr(v) if n else None, n, Hq, Hkv, D,
                                    float(scale), _ptr(o))
    if rc:
        raise ValueError("gqa_decode: Hq must be a multiple of Hkv")
    return o


def gqa_decode(q: np.ndarray, k: np.ndarray, v: np.ndarray, scale: float) -> np.ndarray:
    """Decode attention of one query token: q[Hq][D], k/v[n][Hkv][D] (bf16 bits,
    logical token order) -> fp64 o[Hq][D].  Query head h reads KV head
    h // (Hq // Hkv)."""
    q = np.ascontiguousarray(q, np.uint16)
    k = np.ascontiguousarray(k, np.uint16)
    v = np.ascontiguousarray(v, np.uint16)
    Hq, D = q.shape
    n, Hkv, D2 = k.shape
    assert D2 == D and v.shape == k.shape
    o = np.zeros((Hq, D), np.float64)
    rc = lib().ora_gqa_decode(_ptr(q), _ptr(k) if n else None, _ptr(v) if n else None, n, Hq,
                              Hkv, D, float(scale), _ptr(o))
    if rc:
        raise ValueError("gqa_decode: Hq must be a multiple of Hkv")
    return o


# --------------------------------------------------------------------------
# Block store and paged cache, modelled byte for byte
# --------------------------------------------------------------------------

def _round_up(x: int, m: int) -> int:
    return (x + m - 1) // m * m


KV_BF16, KV_E4M3 = 0, 1  # cache element types (dims); block header dtype codes 1, 2


class Dims:
    """KV geometry: L layers, Hkv KV heads, D head dim, P tokens per page, and
    the element type: bf16, or fp8 E4M3 codes with per-tensor scales (a K
    element is code value * k_scale, a V element code value * v_scale)."""

    def __init__(self, n_layers, n_kv_heads, head_dim, page_size, rope_theta=10000.0,
                 rope_style=0, kv_dtype=KV_BF16, k_scale=1.0, v_scale=1.0):
        self.L, self.Hkv, self.D, self.P = int(n_layers), int(n_kv_heads), int(head_dim), int(page_size)
        self.rope_theta = float(rope_theta)
        self.rope_style = int(rope_style)
        self.kv_dtype = int(kv_dtype)
        # the scales are fp32 values
        self.k_scale = float(np.float32(k_scale))
        self.v_scale = float(np.float32(v_scale))

    @property
    def fp8(self):
        return self.kv_dtype == KV_E4M3

    @property
    def code_dtype(self):
        return np.uint8 if self.fp8 else np.uint16

    @property
    def page_elems(self):
        return self.Hkv * self.P * self.D

    @property
    def page_bytes(self):
        return (1 if self.fp8 else 2) * self.page_elems

    def same(self, o) -> bool:
        return ((self.L, self.Hkv, self.D, self.P, self.kv_dtype) == (o.L, o.Hkv, o.D, o.P, o.kv_dtype)
                and (not self.fp8 or (self.k_scale, self.v_scale) == (o.k_scale, o.v_scale)))

    def codes(self, k_bf16: np.ndarray, v_bf16: np.ndarray):
        """Rows as the cache stores them: bf16 bits, or E4M3 codes."""
        if not self.fp8:
            return k_bf16, v_bf16
        return e4m3_quantize(k_bf16, self.k_scale), e4m3_quantize(v_bf16, self.v_scale)


class Block:
    """A deposited KV block (the paper's persistent artifact, Sec. 3.3).

    Reading of the closed layout: pages[l][kv][j] is laid out exactly like a
    cache page, [Hkv][P][D] bf16, holding tokens [j*P, (j+1)*P) of the block;
    rows past n_tokens in the last page are zero.  digests[l][kv][j] is the
    two-level page digest of that page; the block digest is SHA-256 over the
    little-endian int32 position tags followed by every page digest in
    [l][kv][j] order."""

    def __init__(self, dims: Dims, positions: np.ndarray, pages: np.ndarray):
        self.dims = dims
        self.positions = np.ascontiguousarray(positions, np.int32)
        self.n_tokens = int(self.positions.size)
        self.n_pages = pages.shape[2]
        self.pages = pages  # [L][2][n_pages][Hkv][P][D] bf16 bits or E4M3 codes
        d = dims
        self.digests = page_digests(pages.reshape(-1), d.page_bytes).reshape(
            d.L, 2, self.n_pages, 32)
        self.block_digest = sha256(self.positions.astype("<i4").tobytes() + self.digests.tobytes())

    def serialize(self) -> bytes:
        """Serialized block: a 256-byte header, the int32 position tags, the
        page digests and the pages, each section 256-byte (pages: 4096-byte)
        aligned.  Header fields (little-endian): magic[8], u32 version,
        u32 header_bytes, i32 L, Hkv, D, P, i64 n_tokens, i64 n_pages,
        f64 rope_theta, i32 rope_style, i32 dtype (1 = bf16), u64 offsets of
        positions / digests / pages, u64 total bytes, 32-byte block digest."""
        d = self.dims
        pos_off = HEADER_BYTES
        dig_off = _round_up(pos_off + 4 * self.n_tokens, 256)
        pages_off = _round_up(dig_off + self.digests.size, 4096)
        total = pages_off + self.pages.size * (1 if d.fp8 else 2)
        hdr = bytearray(HEADER_BYTES)
        struct.pack_into("<8sIIiiiiqqdiiQQQQ", hdr, 0, BLOCK_MAGIC, BLOCK_VERSION, HEADER_BYTES,
                         d.L, d.Hkv, d.D, d.P, self.n_tokens, self.n_pages, d.rope_theta,
                         d.rope_style, 2 if d.fp8 else 1, pos_off, dig_off, pages_off, total)
        hdr[96:128] = self.block_digest
        if d.fp8:  # the per-tensor scales, fp32 at bytes 128 (K) and 132 (V)
            struct.pack_into("<ff", hdr, 128, d.k_scale, d.v_scale)
        out = bytearray(total)
        out[:HEADER_BYTES] = hdr
        out[pos_off:pos_off + 4 * self.n_tokens] = self.positions.astype("<i4").tobytes()
        out[dig_off:dig_off + self.digests.size] = self.digests.tobytes()
        out[pages_off:] = self.pages.astype("u1" if d.fp8 else "<u2").tobytes()
        return bytes(out)

    @staticmethod
    def header_size_fields(n_tokens: int, n_pages: int, dims: Dims):
        pos_off = HEADER_BYTES
        dig_off = _round_up(pos_off + 4 * n_tokens, 256)
        pages_off = _round_up(dig_off + dims.L * 2 * n_pages * 32, 4096)
        total = pages_off + dims.L * 2 * n_pages * dims.page_bytes
        return pos_off, dig_off, pages_off, total


class BlockMeta:
    """A block's bookkeeping only (length, pages, position tags), for
    modelling page tables at sizes where the pool bytes are not modelled."""

    def __init__(self, dims: Dims, positions: np.ndarray):
        self.dims = dims
        self.positions = np.ascontiguousarray(positions, np.int32)
        self.n_tokens = int(self.positions.size)
        self.n_pages = (self.n_tokens + dims.P - 1) // dims.P
        self.pages = None


def block_from_kv(dims: Dims, k: np.ndarray, v: np.ndarray, positions: np.ndarray) -> Block:
    """Deposit of logical rows: k, v [L][n][Hkv][D] bf16 bits (quantized to the
    cache's element type), positions[n]."""
    d = dims
    k, v = d.codes(k, v)
    n = int(positions.size)
    npb = (n + d.P - 1) // d.P
    pages = np.zeros((d.L, 2, npb, d.Hkv, d.P, d.D), d.code_dtype)
    for t in range(n):
        j, r = divmod(t, d.P)
        pages[:, 0, j, :, r, :] = k[:, t, :, :]
        pages[:, 1, j, :, r, :] = v[:, t, :, :]
    return Block(d, positions, pages)


class OracleStore:
    """Ordered list of blocks; block id = deposit order."""

    def __init__(self, dims: Dims):
        self.dims = dims
        self.blocks: list[Block] = []

    def add(self, block: Block) -> int:
        self.blocks.append(block)
        return len(self.blocks) - 1


class KvgError(Exception):
    pass


class PinnedBlock:
    """A block whose pages live in the cache's own pool (zero-copy graft):
    pids[j] holds block page j of every layer and K/V."""

    def __init__(self, pids, block: Block):
        self.pids = list(pids)
        self.block = block


class OracleCache:
    """Paged KV cache.

    pool[l][kv][page][h][row][d] bf16 bits, kv 0 = K, 1 = V.  One page id names
    the same row range in every layer.  Per sequence: page_table[j] (page id of
    the sequence's j-th page, -1 if none), page_fill[j] (valid rows, a prefix
    of the page), positions[slot] (position tag, -1 if unwritten) and n_slots
    (slot high-water mark: the next append goes to slot n_slots).

    Page allocation: pages are taken from the front of an ordered free list
    (initially 0..n_pages-1, or a permutation set while every page is free);
    a released sequence's pages go to the back in page-table order.
    """

    def __init__(self, dims: Dims, n_pages: int, max_seqs: int, max_slots: int, fill=None,
                 with_pool: bool = True):
        """with_pool=False models page tables, fills and position tags only
        (the pool bytes are not kept), for full-size workloads."""
        d = self.dims = dims
        self.n_pages = n_pages
        self.max_seqs = max_seqs
        self.max_slots = max_slots
        self.max_pages = (max_slots + d.P - 1) // d.P
        self.pool = np.zeros((d.L, 2, n_pages, d.Hkv, d.P, d.D), d.code_dtype) if with_pool else None
        if fill is not None and self.pool is not None:
            self.pool[...] = fill
        self.free = list(range(n_pages))
        self.pinned = set()
        self.page_table = np.full((max_seqs, self.max_pages), -1, np.int32)
        self.page_fill = np.zeros((max_seqs, self.max_pages), np.int32)
        self.positions = np.full((max_seqs, max_slots), -1, np.int32)
        self.n_slots = np.zeros(max_seqs, np.int32)
        self.windows = [0] * d.L  # per layer: 0 = global attention, W > 0 = last W valid rows

    def set_free_order(self, order):
        if len(self.free) != self.n_pages:
            raise KvgError("free order can only be set while every page is free")
        order = [int(x) for x in order]
        if sorted(order) != list(range(self.n_pages)):
            raise KvgError("not a permutation")
        self.free = order

    def _take(self, n):
        if n > len(self.free):
            raise KvgError("capacity")
        got, self.free = self.free[:n], self.free[n:]
        return got

    def append(self, seq: int, k: np.ndarray, v: np.ndarray, positions: np.ndarray):
        """Fresh write of n rows (k, v [L][n][Hkv][D] bf16 bits, quantized to the
        cache's element type) at slots n_slots.. (Sec. 3.2 fresh arm)."""
        d = self.dims
        k, v = d.codes(k, v)
        n = int(positions.size)
        s0 = int(self.n_slots[seq])
        if s0 + n > self.max_slots:
            raise KvgError("capacity")
        first_new = (s0 + d.P - 1) // d.P
        last = (s0 + n + d.P - 1) // d.P
        need = max(0, last - first_new)
        pids = self._take(need)
        for i, j in enumerate(range(first_new, last)):
            self.page_table[seq, j] = pids[i]
        for t in range(n):
            s = s0 + t
            j, r = divmod(s, d.P)
            pid = self.page_table[seq, j]
            if self.pool is not None:
                self.pool[:, 0, pid, :, r, :] = k[:, t, :, :]
                self.pool[:, 1, pid, :, r, :] = v[:, t, :, :]
            self.positions[seq, s] = positions[t]
            self.page_fill[seq, j] = r + 1
        self.n_slots[seq] = s0 + n

    def graft(self, seq: int, block: Block, dst_slot: int = -1, delta: int = 0):
        """Own-position graft (delta = 0, Sec. 3.2): the block's pages are
        installed whole at page-aligned slot dst_slot = the sequence's next page
        boundary; position tags are the block's own.  With delta != 0 the block
        is re-based (Sec. 4.2): position tags += delta and the valid key rows
        are rotated by delta positions (fp64, rounded to bf16); value rows and
        padding rows are copied unchanged."""
        d = self.dims
        bd = block.dims
        if not bd.same(d):
            raise KvgError("dims")
        if delta != 0 and d.fp8:
            raise KvgError("relocation needs bf16 keys")
        boundary = _round_up(int(self.n_slots[seq]), d.P)
        if dst_slot < 0:
            dst_slot = boundary
        if dst_slot != boundary:
            raise KvgError("dst_slot must be the next page boundary")
        n = block.n_tokens
        if dst_slot + n > self.max_slots:
            raise KvgError("capacity")
        newpos = block.positions.astype(np.int64) + int(delta)
        if n and (newpos.min() < 0 or newpos.max() >= 2 ** 31):
            raise KvgError("position")
        pids = self._take(block.n_pages)
        j0 = dst_slot // d.P
        for j, pid in enumerate(pids):
            self.page_table[seq, j0 + j] = pid
            self.page_fill[seq, j0 + j] = min(d.P, n - j * d.P)
            if self.pool is None:
                continue
            self.pool[:, :, pid] = block.pages[:, :, j]
            if delta != 0:
                valid = min(d.P, n - j * d.P)
                for l in range(d.L):
                    rows = block.pages[l, 0, j, :, :valid, :]
                    self.pool[l, 0, pid, :, :valid, :] = rope_rotate_rows_bf16(
                        rows, delta, d.rope_theta, d.rope_style)
        self.positions[seq, dst_slot:dst_slot + n] = newpos.astype(np.int32)
        self.n_slots[seq] = dst_slot + n

    def append_batch(self, seq_ids, k: np.ndarray, v: np.ndarray, positions: np.ndarray):
        """Decode-step append: row b of k, v [L][B][Hkv][D] is appended to
        sequence seq_ids[b] (one fresh row each, in batch order)."""
        if len(set(int(x) for x in seq_ids)) != len(seq_ids):
            raise KvgError("repeated sequence")
        for b, sq in enumerate(seq_ids):
            self.append(int(sq), k[:, b:b + 1], v[:, b:b + 1], positions[b:b + 1])

    def pin_block(self, seq: int, slot0: int, n: int) -> PinnedBlock:
        """Deposit into the pool: the block's pages (as deposit() builds them)
        are copied into pages taken from the free list for good."""
        blk = self.deposit(seq, slot0, n)
        pids = self._take(blk.n_pages)
        self.pinned |= set(pids)
        for j, pid in enumerate(pids):
            self.pool[:, :, pid] = blk.pages[:, :, j]
        return PinnedBlock(pids, blk)

    def graft_pinned(self, seq: int, pb: PinnedBlock, dst_slot: int = -1):
        """Own-position graft by aliasing: the sequence's page table points at
        the block's pages; a partially filled last page is copied into a page
        of the sequence (its appends fill that page)."""
        d = self.dims
        boundary = _round_up(int(self.n_slots[seq]), d.P)
        if dst_slot < 0:
            dst_slot = boundary
        if dst_slot != boundary:
            raise KvgError("dst_slot must be the next page boundary")
        n = pb.block.n_tokens
        if dst_slot + n > self.max_slots:
            raise KvgError("capacity")
        pages = list(pb.pids)
        if n % d.P:
            pages[-1] = self._take(1)[0]
            self.pool[:, :, pages[-1]] = self.pool[:, :, pb.pids[-1]]
        j0 = dst_slot // d.P
        for j, pid in enumerate(pages):
            self.page_table[seq, j0 + j] = pid
            self.page_fill[seq, j0 + j] = min(d.P, n - j * d.P)
        self.positions[seq, dst_slot:dst_slot + n] = pb.block.positions
        self.n_slots[seq] = dst_slot + n

    def release(self, seq: int):
        used = [int(p) for p in self.page_table[seq] if p >= 0 and int(p) not in self.pinned]
        self.free.extend(used)
        self.page_table[seq] = -1
        self.page_fill[seq] = 0
        self.positions[seq] = -1
        self.n_slots[seq] = 0

    def deposit(self, seq: int, slot0: int, n: int) -> Block:
        """Captures rows [slot0, slot0+n) of a sequence (slot0 page-aligned) with
        their position tags into a block (Sec. 3.3 deposit)."""
        d = self.dims
        if slot0 % d.P or slot0 + n > int(self.n_slots[seq]) or n <= 0:
            raise KvgError("range")
        npb = (n + d.P - 1) // d.P
        pages = np.zeros((d.L, 2, npb, d.Hkv, d.P, d.D), d.code_dtype)
        for j in range(npb):
            pid = self.page_table[seq, slot0 // d.P + j]
            valid = min(d.P, n - j * d.P)
            pages[:, :, j, :, :valid, :] = self.pool[:, :, pid, :, :valid, :]
        return Block(d, self.positions[seq, slot0:slot0 + n].copy(), pages)

    def logical_kv(self, seq: int, layer: int):
        """The sequence's valid rows in logical order: pages j = 0.. in order,
        rows [0, page_fill[j]) of each -> k, v [n][Hkv][D], positions [n]."""
        d = self.dims
        ks, vs, ps = [], [], []
        npg = (int(self.n_slots[seq]) + d.P - 1) // d.P
        for j in range(npg):
            pid = self.page_table[seq, j]
            f = int(self.page_fill[seq, j])
            if pid < 0 or f == 0:
                continue
            ks.append(np.transpose(self.pool[layer, 0, pid, :, :f, :], (1, 0, 2)))
            vs.append(np.transpose(self.pool[layer, 1, pid, :, :f, :], (1, 0, 2)))
            ps.append(self.positions[seq, j * d.P:j * d.P + f])
        if not ks:
            z = np.zeros((0, d.Hkv, d.D), d.code_dtype)
            return z, z.copy(), np.zeros(0, np.int32)
        return (np.ascontiguousarray(np.concatenate(ks)), np.ascontiguousarray(np.concatenate(vs)),
                np.concatenate(ps))

    def set_layer_windows(self, windows):
        """Per-layer sliding windows (0 = global) over the full-size cache
        (Sec. 4.3: windowed layers keep full-size KV so a restored block
        resumes exactly); [] resets every layer to global."""
        w = [int(x) for x in windows] or [0] * self.dims.L
        if len(w) != self.dims.L or min(w) < 0:
            raise KvgError("need one window >= 0 per layer")
        self.windows = w

    def decode_range(self, seq: int, layer: int, q: np.ndarray, scale: float, slot_begin: int,
                     slot_end: int) -> np.ndarray:
        """fp64 decode attention of q[Hq][D] over the valid rows whose slots lie
        in [slot_begin, slot_end) and, on a windowed layer, among the layer's
        last W valid rows of the whole sequence: the part of the decode step
        (Sec. 3.2) that a split decode computes over already-resident rows."""
        d = self.dims
        slots = []
        npg = (int(self.n_slots[seq]) + d.P - 1) // d.P
        for j in range(npg):
            for r in range(int(self.page_fill[seq, j]) if self.page_table[seq, j] >= 0 else 0):
                slots.append(j * d.P + r)
        W = self.windows[layer]
        if W > 0:
            slots = slots[-W:]
        keep = [s for s in slots if slot_begin <= s < slot_end]
        k = np.zeros((len(keep), d.Hkv, d.D), d.code_dtype)
        v = np.zeros((len(keep), d.Hkv, d.D), d.code_dtype)
        for i, s in enumerate(keep):
            j, r = divmod(s, d.P)
            pid = self.page_table[seq, j]
            k[i] = self.pool[layer, 0, pid, :, r, :]
            v[i] = self.pool[layer, 1, pid, :, r, :]
        if d.fp8:
            return gqa_decode_f64kv(q, e4m3_dequant(k, d.k_scale), e4m3_dequant(v, d.v_scale), scale)
        return gqa_decode(q, k, v, scale)

    def decode(self, seq: int, layer: int, q: np.ndarray, scale: float) -> np.ndarray:
        """fp64 decode attention of q[Hq][D] over the sequence's valid rows,
        or over the last W of them when the layer has a window W > 0."""
        k, v, _ = self.logical_kv(seq, layer)
        W = self.windows[layer]
        if W > 0:
            k, v = k[-W:], v[-W:]
        d = self.dims
        if d.fp8:
            return gqa_decode_f64kv(q, e4m3_dequant(k, d.k_scale), e4m3_dequant(v, d.v_scale), scale)
        return gqa_decode(q, k, v, scale)
