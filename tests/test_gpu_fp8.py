"""Quantized KV blocks on the GPU: fp8 E4M3 caches with per-tensor scales,
against the oracle.  Appends must produce the oracle's codes bit for bit (the
fp32 product with the fp32 reciprocal of the scale, then nearest-even E4M3
with saturation, on both sides); deposits, grafts and digests are byte operations on the smaller pages
and must match bit for bit; decode attention (the codes expanded to fp16, fp16
tensor-core MMAs, fp32 accumulation) within 1e-2 of the fp64 oracle over the
dequantized rows; grafted rows decode bit-identically to the same rows
written fresh."""
import hashlib
import math

import numpy as np
import pytest
import torch

import kvg_synth as syn
from kvg_testlib import compare_decode, dev_view, geometry, need_gpu, tables, to_dev, u16

pytestmark = pytest.mark.gpu

HBM_CAP = 1 << 28
CANARY8 = 0x7F  # the E4M3 NaN code: never produced by a saturating quantizer

# geometry, k_scale, v_scale: power-of-two and general scales; scale 1.0 puts
# many N(0,1) values on the subnormal grid
CASES = [("d128", 0.0625, 0.125), ("d256", 0.037, 0.29), ("g4", 1.0, 0.5)]


def _dims(kvg, w, ks, vs):
    return kvg.make_dims(w.n_layers, w.n_kv_heads, w.head_dim, w.page_size, w.rope_theta, 0,
                         kv_dtype=kvg.KVG_KV_E4M3, k_scale=ks, v_scale=vs)


def _odims(oracle, w, ks, vs):
    return oracle.Dims(w.n_layers, w.n_kv_heads, w.head_dim, w.page_size, w.rope_theta, 0, oracle.KV_E4M3, ks, vs)


def _kv(w, n, seed):
    k, v = syn.kv_rows(w, n, seed)
    return syn.as_u16(k), syn.as_u16(v)


def _append(kvg, cache, seq, k, v, pos):
    kd, vd, pd = to_dev(k), to_dev(v), to_dev(pos.astype(np.int32))
    kvg.kvg_cache_append(cache.h, seq, kd.data_ptr(), vd.data_ptr(), pd.data_ptr(), pos.size)
    torch.cuda.synchronize()


def _pool8(cache, w):
    v = cache.view
    a = dev_view(v.pool, v.pool_bytes, torch.uint8).cpu().numpy()
    return a.reshape(w.n_layers, 2, v.n_pages, w.n_kv_heads, w.page_size, w.head_dim)


def _fill(cache):
    v = cache.view
    dev_view(v.pool, v.pool_bytes, torch.uint8).fill_(CANARY8)
    torch.cuda.synchronize()


def _decode(kvg, cache, w, seq_ids, q, layer=-1):
    qd = to_dev(q)
    out = torch.empty_like(qd)
    kvg.kvg_decode_attention(cache.h, layer, seq_ids, qd.data_ptr(), w.n_q_heads, out.data_ptr(),
                             1.0 / math.sqrt(w.head_dim))
    torch.cuda.synchronize()
    return u16(out)


@pytest.mark.parametrize("geo,ks,vs", CASES)
def test_fp8_appends_quantize_bit_exact(oracle, geo, ks, vs):
    kvg = need_gpu()
    w = geometry(geo)
    P = w.page_size
    sizes = [1, P - 1, P, P + 1, 3 * P + 5]
    k, v = _kv(w, sum(sizes) + 2 * P, 101)
    max_slots = 8 * P + 64
    n_pages = 24
    c = kvg.Cache(_dims(kvg, w, ks, vs), n_pages, 6, max_slots)
    _fill(c)
    kvg.kvg_cache_set_free_order(c.h, syn.permutation(n_pages, 102))
    oc = oracle.OracleCache(_odims(oracle, w, ks, vs), n_pages, 6, max_slots, fill=CANARY8)
    oc.set_free_order(syn.permutation(n_pages, 102))
    t = 0
    for n in sizes:
        pos = syn.positions(t, n)
        _append(kvg, c, 0, k[:, t:t + n], v[:, t:t + n], pos)
        oc.append(0, k[:, t:t + n], v[:, t:t + n], pos)
        t += n
    # decode-step appends, one row per sequence
    for i, n in enumerate([5, P, 1]):
        kk, vv = _kv(w, n, 110 + i)
        _append(kvg, c, 1 + i, kk, vv, syn.positions(0, n))
        oc.append(1 + i, kk, vv, syn.positions(0, n))
    seqs = [3, 1, 2]
    for step in range(2):
        kk, vv = _kv(w, len(seqs), 120 + step)
        pos = np.array([500 + 10 * step + b for b in range(len(seqs))], np.int32)
        kd, vd, pd = to_dev(kk), to_dev(vv), to_dev(pos)
        kvg.kvg_cache_append_batch(c.h, seqs, kd.data_ptr(), vd.data_ptr(), pd.data_ptr())
        torch.cuda.synchronize()
        oc.append_batch(seqs, kk, vv, pos)
    assert np.array_equal(_pool8(c, w), oc.pool)
    pt, pf, ps = tables(c)
    assert np.array_equal(pt, oc.page_table) and np.array_equal(pf, oc.page_fill)
    assert np.array_equal(ps, oc.positions)
    kvg.kvg_sync(c.h)


@pytest.mark.parametrize("geo,ks,vs", CASES)
def test_fp8_deposit_graft_verify_bit_exact(oracle, geo, ks, vs):
    kvg = need_gpu()
    w = geometry(geo)
    P = w.page_size
    nb = 4 * P + 7
    k, v = _kv(w, nb, 131)
    dims = _dims(kvg, w, ks, vs)
    od = _odims(oracle, w, ks, vs)
    max_slots = 8 * P
    n_pages = 40
    src = kvg.Cache(dims, n_pages, 1, max_slots)
    _append(kvg, src, 0, k, v, syn.positions(0, nb))
    oblk = oracle.block_from_kv(od, k, v, syn.positions(0, nb))
    for residency in (kvg.KVG_RESIDENCY_HBM, kvg.KVG_RESIDENCY_PINNED_HOST):
        store = kvg.Store(dims, residency, HBM_CAP)
        bid = kvg.kvg_deposit(store.h, src.h, 0, 0, nb)
        blob = kvg.kvg_store_export(store.h, bid)
        assert blob == oblk.serialize()
        dst = kvg.Cache(dims, n_pages, 3, max_slots)
        _fill(dst)
        oc = oracle.OracleCache(od, n_pages, 3, max_slots, fill=CANARY8)
        rep = kvg.kvg_graft_report()
        kvg.kvg_graft(store.h, bid, dst.h, 0, -1, 0, kvg.KVG_GRAFT_VERIFY | kvg.KVG_GRAFT_SYNC, report=rep)
        assert rep.n_mismatch == 0 and rep.n_pages_checked == w.n_layers * 2 * oblk.n_pages
        oc.graft(0, oblk)
        kvg.kvg_verify(store.h, bid, dst.h, 0, 0, kvg.KVG_GRAFT_SYNC)
        assert np.array_equal(_pool8(dst, w), oc.pool)
        # a flipped byte is found on its page
        bad = bytearray(blob)
        info = kvg.kvg_store_block_info(store.h, bid)
        bad_page = 3 * oblk.n_pages + 1 if w.n_layers > 1 else oblk.n_pages + 1
        bad[info.pages_offset + bad_page * od.page_bytes + 5] ^= 0x01
        bid2 = kvg.kvg_store_import(store.h, bytes(bad), 0)
        rep2 = kvg.kvg_graft_report()
        with pytest.raises(kvg.KvgError) as e:
            kvg.kvg_graft(store.h, bid2, dst.h, 1, -1, 0, kvg.KVG_GRAFT_VERIFY | kvg.KVG_GRAFT_SYNC, report=rep2)
        assert e.value.status == kvg.KVG_ERR_DIGEST and rep2.mismatch_pages[0] == bad_page
        # relocation needs bf16 keys, in a single graft and in a batch (which
        # then grafts nothing)
        with pytest.raises(kvg.KvgError) as e:
            kvg.kvg_graft(store.h, bid, dst.h, 2, -1, 5, 0)
        assert e.value.status == kvg.KVG_ERR_ARG
        with pytest.raises(kvg.KvgError) as e:
            kvg.kvg_graft_batch(store.h, [bid], dst.h, [2], deltas=[5])
        assert e.value.status == kvg.KVG_ERR_ARG
        assert kvg.kvg_cache_seq_info(dst.h, 2)[0] == 0
        kvg.kvg_sync(dst.h)
    # element type and scales are part of the geometry
    bf16 = kvg.make_dims(w.n_layers, w.n_kv_heads, w.head_dim, w.page_size, w.rope_theta, 0)
    other = _dims(kvg, w, ks * 2, vs)
    for d2, status in ((bf16, kvg.KVG_ERR_FORMAT), (other, kvg.KVG_ERR_FORMAT)):
        s2 = kvg.Store(d2, kvg.KVG_RESIDENCY_HBM, 1 << 28)
        with pytest.raises(kvg.KvgError) as e:
            kvg.kvg_store_import(s2.h, blob, 0)
        assert e.value.status == status
    c16 = kvg.Cache(bf16, n_pages, 1, max_slots)
    with pytest.raises(kvg.KvgError) as e:
        kvg.kvg_graft(store.h, bid, c16.h, 0, -1, 0, 0)
    assert e.value.status == kvg.KVG_ERR_ARG


@pytest.mark.parametrize("geo,ks,vs", CASES)
def test_fp8_decode_matches_oracle_and_grafted_equals_fresh(oracle, geo, ks, vs):
    kvg = need_gpu()
    w = geometry(geo)
    P = w.page_size
    nb, nf = 3 * P + 9, 2 * P + 3
    k, v = _kv(w, nb + nf, 141)
    dims = _dims(kvg, w, ks, vs)
    od = _odims(oracle, w, ks, vs)
    max_slots = 8 * P
    n_pages = 48
    src = kvg.Cache(dims, n_pages, 1, max_slots)
    _append(kvg, src, 0, k[:, :nb], v[:, :nb], syn.positions(0, nb))
    store = kvg.Store(dims, kvg.KVG_RESIDENCY_HBM, HBM_CAP)
    bid = kvg.kvg_deposit(store.h, src.h, 0, 0, nb)
    c = kvg.Cache(dims, n_pages, 3, max_slots)
    kvg.kvg_cache_set_free_order(c.h, syn.permutation(n_pages, 142))
    oc = oracle.OracleCache(od, n_pages, 3, max_slots)
    oc.set_free_order(syn.permutation(n_pages, 142))
    kvg.kvg_graft(store.h, bid, c.h, 0, -1, 0, kvg.KVG_GRAFT_SYNC)
    oc.graft(0, oracle.block_from_kv(od, k[:, :nb], v[:, :nb], syn.positions(0, nb)))
    _append(kvg, c, 0, k[:, nb:], v[:, nb:], syn.positions(nb, nf))
    oc.append(0, k[:, nb:], v[:, nb:], syn.positions(nb, nf))
    # the same rows written fresh (seq 1), and a short sequence (seq 2)
    _append(kvg, c, 1, k, v, syn.positions(0, nb + nf))
    _append(kvg, c, 2, k[:, :3], v[:, :3], syn.positions(0, 3))
    oc.append(2, k[:, :3], v[:, :3], syn.positions(0, 3))
    scale = 1.0 / math.sqrt(w.head_dim)
    q = syn.as_u16(syn.queries(w, w.n_layers, 2, 143))
    o = _decode(kvg, c, w, [0, 2], q)
    for l in range(w.n_layers):
        compare_decode(oracle, o[l, 0], oc.decode(0, l, q[l, 0], scale))
        compare_decode(oracle, o[l, 1], oc.decode(2, l, q[l, 1], scale))
        ol = _decode(kvg, c, w, [0], q[l:l + 1, :1], layer=l)
        compare_decode(oracle, ol[0, 0], oc.decode(0, l, q[l, 0], scale))
    q1 = q[:, :1]
    og = _decode(kvg, c, w, [0], q1)
    assert hashlib.sha256(og.tobytes()).digest() == hashlib.sha256(_decode(kvg, c, w, [1], q1).tobytes()).digest()
    for _ in range(2):
        assert _decode(kvg, c, w, [0], q1).tobytes() == og.tobytes()
    # sliding windows apply to fp8 caches the same way
    wins = [(P + 3) if l % 2 == 0 else 0 for l in range(w.n_layers)]
    kvg.kvg_cache_set_layer_windows(c.h, wins)
    oc.set_layer_windows(wins)
    ow = _decode(kvg, c, w, [0, 2], q)
    for l in range(w.n_layers):
        compare_decode(oracle, ow[l, 0], oc.decode(0, l, q[l, 0], scale))
        compare_decode(oracle, ow[l, 1], oc.decode(2, l, q[l, 1], scale))
    kvg.kvg_sync(c.h)


def test_fp8_decode_rejects_head_dim_64():
    kvg = need_gpu()
    w = geometry("tiny")
    c = kvg.Cache(_dims(kvg, w, 1.0, 1.0), 8, 1, 64)
    k, v = _kv(w, 5, 151)
    _append(kvg, c, 0, k, v, syn.positions(0, 5))
    q = torch.zeros((w.n_layers, 1, w.n_q_heads, w.head_dim), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(kvg.KvgError) as e:
        kvg.kvg_decode_attention(c.h, -1, [0], q.data_ptr(), w.n_q_heads, q.data_ptr(), 0.125)
    assert e.value.status == kvg.KVG_ERR_ARG
