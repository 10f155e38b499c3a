"""A planted needle in every 16-row group of a long context (Sec. 4.4's
planted-needle check, applied to the decode kernel's tiles).

Row group j (rows 16j ... 16j + 15, the finest tile height any decode
instance uses) holds one needle row whose key points along its own random
direction u_j (|k| = 160) and whose value is that row's N(0, 1) draw; every
other key is an N(0, 1) row scaled by 1/4.  Batch row b of one decode call
queries the same sequence with q = (sqrt(D) / 4) u_b in every head, so the
needle of group b scores 40 (natural-log units), any other needle about
40 u_b.u_j (|u_b.u_j| ~ 1/sqrt(D), at most ~11 here) and any other row
about N(0, 1/16): the softmax puts all but ~1e-10 of its weight on needle b,
and the output is that needle's value row to within far less than a bf16
step.  So each batch row's output must equal its own group's value row (bit
for bit, or within 1e-6 where the value is that close to zero): a kernel
that skipped, repeated or misplaced any tile, page or group returns another
row or a mixture.  The first rows come from a graft and the rest from a
fresh write, so the tiles span both writers and a ragged last page.  Sampled
batch rows are also compared with the fp64 oracle through the decode gate."""
import math

import numpy as np
import pytest
import torch

import kvg_synth as syn
from kvg_testlib import append, compare_decode, decode, dims_for, geometry, need_gpu

pytestmark = pytest.mark.gpu

GROUP = 16


def _needle_case(w, n, seed, key_mag=160.0):
    """K, V (uint16 [L][n][Hkv][D]), the needle rows and the queries
    (uint16 [L][T][Hq][D]) of the construction above; |needle key| = key_mag
    and |q| = 40 sqrt(D) / key_mag, so a needle scores 40 for its own query."""
    g = torch.Generator().manual_seed(seed)
    k, v = syn.kv_rows(w, n, seed)
    k = (k.float() * 0.25).to(torch.bfloat16)
    T = -(-n // GROUP)
    rows = np.array([min(j * GROUP + (j * 5) % GROUP, n - 1) for j in range(T)])
    u = torch.randn((w.n_layers, T, w.n_kv_heads, w.head_dim), generator=g, dtype=torch.float64)
    u = u / u.norm(dim=-1, keepdim=True)
    k[:, torch.from_numpy(rows)] = (key_mag * u).to(torch.bfloat16)
    q = (40.0 * math.sqrt(w.head_dim) / key_mag * u).repeat_interleave(w.group, dim=2).to(torch.bfloat16)
    return syn.as_u16(k), syn.as_u16(v), rows, syn.as_u16(q)


def _check_needles(oracle, o, want_bits, T):
    same = o == want_bits
    near = np.abs(oracle.bf16_to_f64(o) - oracle.bf16_to_f64(want_bits)) <= 1e-6
    bad = np.argwhere(~(same | near))
    assert bad.size == 0, f"{len(bad)} elements off their needle's value, first (layer, group, head, d): {bad[:4]}"
    assert same.mean() > 0.999
    # the outputs really move: every group's output differs from the next one's
    assert all(not np.array_equal(o[:, b], o[:, b + 1]) for b in range(T - 1))


@pytest.mark.parametrize("geo,n_block,n_fresh", [("d256", 4096, 4133), ("d128", 2048, 3000), ("tiny", 256, 77)])
def test_a_needle_in_every_row_group_moves_the_output(oracle, geo, n_block, n_fresh):
    kvg = need_gpu()
    w = geometry(geo)
    n = n_block + n_fresh
    k, v, rows, q = _needle_case(w, n, 0x6E65 + n)
    P = w.page_size
    max_slots = (-(-n // P) + 1) * P
    dims = dims_for(kvg, w)
    src = kvg.Cache(dims, max_slots // P + 1, 1, max_slots)
    append(kvg, src, 0, np.ascontiguousarray(k[:, :n_block]), np.ascontiguousarray(v[:, :n_block]),
           syn.positions(0, n_block))
    store = kvg.Store(dims, kvg.KVG_RESIDENCY_HBM, 1 << 30)
    bid = kvg.kvg_deposit(store.h, src.h, 0, 0, n_block)
    dst = kvg.Cache(dims, 2 * (max_slots // P) + 2, 2, max_slots)
    kvg.kvg_cache_set_free_order(dst.h, syn.permutation(2 * (max_slots // P) + 2, n))
    kvg.kvg_graft(store.h, bid, dst.h, 1, -1, 0, kvg.KVG_GRAFT_VERIFY | kvg.KVG_GRAFT_SYNC)
    append(kvg, dst, 1, np.ascontiguousarray(k[:, n_block:]), np.ascontiguousarray(v[:, n_block:]),
           syn.positions(n_block, n_fresh))
    T = len(rows)
    o = decode(kvg, dst, w, [1] * T, q)  # [L][T][Hq][D]
    # needle b's value row in every head of its group
    _check_needles(oracle, o, v[:, rows].repeat(w.group, axis=2), T)
    # sampled batch rows against the fp64 oracle
    scale = 1.0 / math.sqrt(w.head_dim)
    for b in (0, T // 2, T - 1):
        for l in range(w.n_layers):
            ref = oracle.gqa_decode(q[l, b], k[l], v[l], scale)
            compare_decode(oracle, o[l, b], ref, what=f"needle {geo} group {b} layer {l}")
    kvg.kvg_sync(dst.h)


@pytest.mark.parametrize("geo,n", [("d128", 3001), ("d256", 2100)])
def test_a_needle_in_every_row_group_fp8(oracle, geo, n):
    """The same construction in an fp8 E4M3 cache (scales 1/16; needle keys
    of norm 80 so their codes stay within the E4M3 range): each output is its
    needle's dequantized value row (E4M3 code x 1/16, exact in bf16)."""
    kvg = need_gpu()
    w = geometry(geo)
    ks = vs = 0.0625
    k, v, rows, q = _needle_case(w, n, 0x6E66 + n, key_mag=80.0)
    P = w.page_size
    max_slots = (-(-n // P) + 1) * P
    dims = kvg.make_dims(w.n_layers, w.n_kv_heads, w.head_dim, P, w.rope_theta, 0, kv_dtype=kvg.KVG_KV_E4M3,
                         k_scale=ks, v_scale=vs)
    c = kvg.Cache(dims, max_slots // P + 1, 1, max_slots)
    append(kvg, c, 0, k, v, syn.positions(0, n))
    T = len(rows)
    o = decode(kvg, c, w, [0] * T, q)
    kd = oracle.e4m3_dequant(oracle.e4m3_quantize(k, ks), ks)
    vd = oracle.e4m3_dequant(oracle.e4m3_quantize(v, vs), vs)
    _check_needles(oracle, o, oracle.bf16_rne(vd[:, rows]).repeat(w.group, axis=2), T)
    scale = 1.0 / math.sqrt(w.head_dim)
    for b in (0, T // 2, T - 1):
        for l in range(w.n_layers):
            ref = oracle.gqa_decode_f64kv(q[l, b], kd[l], vd[l], scale)
            compare_decode(oracle, o[l, b], ref, what=f"needle fp8 {geo} group {b} layer {l}")
    kvg.kvg_sync(c.h)
