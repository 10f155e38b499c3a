"""Helpers shared by the GPU tests: device views of library-owned memory,
small geometries, and the two sides of a parity check (the CUDA library via
its C ABI, the oracle on the CPU), each fed the same seeded bytes."""
from __future__ import annotations

import math
import os

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


# Decode gate (paper Sec. 3.2 for the attention being computed; Sec. 4.1 for
# the byte-exact regime it is checked in).  Three bounds, all on one output
# (every query head of one (layer, batch row)):
#   * max |got - ref| <= 1e-2 + half a bf16 step of ref, the stated
#     tolerance for bf16 outputs read as a bound on the fp32-accumulated
#     result, which the output's own bf16 rounding then moves by up to half
#     a step (0.0078 for |ref| in [2, 4): without it, 1e-2 would ask for
#     less than a bf16 step there, and of a correctly rounded output from
#     |ref| = 4 on; seeded scenarios with |ref| ~ 3 reached 0.0101-0.0110);
#   * max |got - ref| / max |ref| <= REL_TOL.  The kernel's only rounding
#     steps that matter are the softmax weights, rounded to bf16 before the
#     P.V product (relative error <= 2^-9 each, uniform, so a weighted error
#     of ~2^-9/sqrt(3) of the output's own scale, ~4 sigma at the maximum of
#     a few thousand elements), and the output's bf16 rounding (<= 2^-9 of
#     the element).  Together ~3.6e-3 of max |ref| at every context length
#     from 2 to 65,536 rows (a numpy model of these roundings on N(0, 1)
#     rows); REL_TOL = 2^-7 leaves a factor ~2 of margin.  Dropping 1% of a
#     32k context's rows moves the output by ~1e-1 of max |ref| (0.1%: 3e-2),
#     so a partial-context bug fails this bound;
#   * the fraction of elements equal to bf16_rne(ref) >= RNE_FLOOR (checked
#     on outputs of >= 256 elements).  The same model gives 0.52-0.81 (most
#     rounding boundaries lie farther from the exact value than the weights'
#     error); dropping 1% (0.1%) of the rows leaves ~0.02 (~0.08).
REL_TOL = 2.0 ** -7
RNE_FLOOR = 0.35
# Keys and the query re-rotated by RoPE (relocation, Sec. 4.2) and rounded to
# bf16 before the score, compared with the un-rotated reference: each score
# gains an error of ~1.6e-3, the model's maximum becomes ~5.4e-3 of max |ref|
# and the RNE match 0.40-0.48.
REL_TOL_RELOCATED = 2.0 ** -6
RNE_FLOOR_RELOCATED = 0.25


def check_rotation_rounding(oracle, got, ref, min_exact=0.999):
    """Relocated keys against the fp64 rotation `ref`: the kernel rotates in
    fp32 (cos/sin of the fp64 angle rounded to fp32), so its bf16 result
    `got` (uint16 bits) is the correctly rounded fp64 value except where the
    fp32 error straddles a rounding boundary.  There it is one bf16 step away
    (same sign), or, where the pair's two products nearly cancel, within the
    fp32 error of the products, 2^-21 of the rows' largest magnitude."""
    rne = oracle.bf16_rne(ref)
    g = np.asarray(got, np.uint16)
    exact = g == rne
    steps = np.abs((g & 0x7FFF).astype(np.int32) - (rne & 0x7FFF).astype(np.int32))
    off = int((~exact).sum())
    assert off <= max(2, (1.0 - min_exact) * exact.size), (off, exact.size)
    near = np.abs(oracle.bf16_to_f64(g) - ref) <= 2.0 ** -21 * np.abs(ref).max()
    assert np.all(exact | ((steps == 1) & ((g & 0x8000) == (rne & 0x8000))) | near)


def compare_decode(oracle, o_gpu_bits: np.ndarray, o_ref: np.ndarray, tol=1e-2, rel=REL_TOL, floor=RNE_FLOOR,
                   what=""):
    """Checks one decode output against the fp64 oracle with the three bounds
    above; returns (max-abs error, relative error, RNE-match fraction).  With
    KVG_DECODE_GATE_LOG set, appends the figures to that file."""
    got = oracle.bf16_to_f64(o_gpu_bits)
    if not got.size:
        return 0.0, 0.0, 1.0
    err = float(np.abs(got - o_ref).max())
    # the max-abs tolerance bounds the fp32-accumulated result; the bf16
    # output adds up to half a bf16 step of the reference on top (2^-8 of
    # |ref|'s power of two: 0.0078 for |ref| in [2, 4), beyond 1e-2 itself
    # from |ref| = 4 on)
    half_step = np.ldexp(1.0, np.floor(np.log2(np.maximum(np.abs(o_ref), 2.0 ** -126))).astype(np.int64) - 8)
    err_acc = float((np.abs(got - o_ref) - half_step).max())
    top = float(np.abs(o_ref).max())
    relerr = err / top if top > 0 else (0.0 if err == 0 else math.inf)
    rne = oracle.bf16_rne(o_ref)
    match = float((rne == o_gpu_bits).mean())
    log = os.environ.get("KVG_DECODE_GATE_LOG")
    if log:
        with open(log, "a") as f:
            f.write(f"{what or os.environ.get('PYTEST_CURRENT_TEST', '?')}\t{got.size}\t{err:.3e}\t"
                    f"{relerr:.3e}\t{match:.4f}\n")
    assert err_acc <= tol, f"{what}: max-abs error {err} is {err_acc} beyond the output's bf16 rounding > {tol}"
    assert relerr <= rel, f"{what}: relative error {relerr:.3e} > {rel:.3e} (max |ref| {top:.3e})"
    if got.size >= 256:
        assert match >= floor, f"{what}: RNE match {match:.3f} < {floor}"
    return err, relerr, match
