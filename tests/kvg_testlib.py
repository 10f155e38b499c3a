"""Helpers shared by the GPU tests: device views of library-owned memory,
small geometries, and the two sides of a parity check (the CUDA library via
its C ABI, the oracle on the CPU), each fed the same seeded bytes."""
from __future__ import annotations

import math

import numpy as np
import pytest
import torch

import kvg_synth as syn

CANARY = 0x7FBF  # a bf16 NaN pattern the method never produces


def need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_14431_gb300 import build
    build.build()
    from paper_2607_14431_gb300 import kvg
    return kvg


class _Iface:
    def __init__(self, ptr, n, typestr):
        self.__cuda_array_interface__ = {"shape": (n,), "typestr": typestr, "data": (int(ptr), False),
                                         "version": 3, "strides": None}


def dev_view(ptr: int, nbytes: int, dtype=torch.uint8) -> torch.Tensor:
    """A torch tensor aliasing library-owned device memory (no copy)."""
    typestr = {torch.uint8: "|u1", torch.int32: "<i4", torch.int16: "<i2"}[dtype]
    itemsize = torch.tensor([], dtype=dtype).element_size()
    return torch.as_tensor(_Iface(ptr, nbytes // itemsize, typestr), device="cuda")


def geometry(name):
    """Small geometries that still span several tiles and a ragged tail."""
    if name == "tiny":
        return syn.TINY
    if name == "d128":
        return syn.Workload("d128", 3, 8, 4, 128, 64, 1e6, 0x51)
    if name == "d256":
        return syn.Workload("d256", 2, 4, 2, 256, 64, 10000.0, 0x52)
    if name == "g4":
        return syn.Workload("g4", 2, 8, 2, 128, 32, 10000.0, 0x53)
    raise KeyError(name)


def dims_for(kvg, w, style=0):
    return kvg.make_dims(w.n_layers, w.n_kv_heads, w.head_dim, w.page_size, w.rope_theta, style)


def oracle_dims(oracle, w, style=0):
    return oracle.Dims(w.n_layers, w.n_kv_heads, w.head_dim, w.page_size, w.rope_theta, style)


def to_dev(a: np.ndarray) -> torch.Tensor:
    if a.dtype == np.uint16:
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).cuda()
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def u16(t: torch.Tensor) -> np.ndarray:
    return t.detach().contiguous().cpu().numpy().view(np.uint16)


def fill_canary(cache):
    v = cache.view
    dev_view(v.pool, v.pool_bytes, torch.int16).fill_(np.int16(np.uint16(CANARY).view(np.int16)))
    torch.cuda.synchronize()


def pool_u16(cache, w) -> np.ndarray:
    v = cache.view
    a = u16(dev_view(v.pool, v.pool_bytes, torch.int16))
    return a.reshape(w.n_layers, 2, v.n_pages, w.n_kv_heads, w.page_size, w.head_dim)


def tables(cache):
    v = cache.view
    pt = dev_view(v.page_table, v.max_seqs * v.max_pages * 4, torch.int32).cpu().numpy()
    pf = dev_view(v.page_fill, v.max_seqs * v.max_pages * 4, torch.int32).cpu().numpy()
    ps = dev_view(v.positions, v.max_seqs * v.max_slots * 4, torch.int32).cpu().numpy()
    return (pt.reshape(v.max_seqs, v.max_pages), pf.reshape(v.max_seqs, v.max_pages),
            ps.reshape(v.max_seqs, v.max_slots))


def append(kvg, cache, seq, k: np.ndarray, v: np.ndarray, pos: np.ndarray):
    """Fresh write through the C ABI; k, v [L][n][Hkv][D] bf16 bits."""
    kd, vd, pd = to_dev(k), to_dev(v), to_dev(pos.astype(np.int32))
    kvg.kvg_cache_append(cache.h, seq, kd.data_ptr(), vd.data_ptr(), pd.data_ptr(), pos.size)
    torch.cuda.synchronize()


def decode(kvg, cache, w, seq_ids, q: np.ndarray, layer=-1) -> np.ndarray:
    """q [Lrun][B][Hq][D] bf16 bits -> out bf16 bits, same shape."""
    qd = to_dev(q)
    out = torch.empty_like(qd)
    kvg.kvg_decode_attention(cache.h, layer, seq_ids, qd.data_ptr(), w.n_q_heads, out.data_ptr(),
                             1.0 / math.sqrt(w.head_dim))
    torch.cuda.synchronize()
    return u16(out)


def compare_decode(oracle, o_gpu_bits: np.ndarray, o_ref: np.ndarray, tol=1e-2):
    got = oracle.bf16_to_f64(o_gpu_bits)
    err = np.abs(got - o_ref).max() if got.size else 0.0
    rne = oracle.bf16_rne(o_ref)
    match = float((rne == o_gpu_bits).mean()) if got.size else 1.0
    assert err <= tol, f"max-abs error {err} > {tol}"
    return err, match
