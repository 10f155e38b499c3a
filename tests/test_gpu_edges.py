"""GPU edge cases against the CPU oracle: every query-group size the decode
kernel is built for (bf16 and fp8), one-row pages, a one-token block, the
largest decode batch, an empty append, and position tags at the top of the
int32 range."""
import math

import numpy as np
import pytest
import torch

import kvg_synth as syn
from kvg_testlib import (CANARY, append, check_rotation_rounding, compare_decode, decode, dims_for, fill_canary, geometry,
                         need_gpu,
                         oracle_dims, pool_u16, tables, to_dev, u16)

pytestmark = pytest.mark.gpu

HBM_CAP = 1 << 30


def _kv(w, n, seed):
    k, v = syn.kv_rows(w, n, seed)
    return syn.as_u16(k), syn.as_u16(v)


# (head_dim, group, fp8): every instance of the decode kernel
BF16_CASES = [(64, 1), (64, 4), (64, 8), (128, 1), (256, 1)]
FP8_CASES = [(128, 1), (256, 1)]


def _sequence_case(kvg, oracle, w, fp8=False, ks=0.0625, vs=0.125):
    """Two sequences: a ragged block grafted then fresh rows; one row only."""
    P = w.page_size
    if fp8:
        dims = kvg.make_dims(w.n_layers, w.n_kv_heads, w.head_dim, P, w.rope_theta, 0,
                             kv_dtype=kvg.KVG_KV_E4M3, k_scale=ks, v_scale=vs)
        od = oracle.Dims(w.n_layers, w.n_kv_heads, w.head_dim, P, w.rope_theta, 0, oracle.KV_E4M3, ks, vs)
    else:
        dims, od = dims_for(kvg, w), oracle_dims(oracle, w)
    nb, nf = 3 * P + 5, 2 * P + 3
    k, v = _kv(w, nb + nf, 171 + w.head_dim + w.n_q_heads)
    max_slots = 8 * P + 64
    src = kvg.Cache(dims, 32, 1, max_slots)
    append(kvg, src, 0, k[:, :nb], v[:, :nb], syn.positions(0, nb))
    store = kvg.Store(dims, kvg.KVG_RESIDENCY_HBM, HBM_CAP)
    bid = kvg.kvg_deposit(store.h, src.h, 0, 0, nb)
    c = kvg.Cache(dims, 32, 2, max_slots)
    if fp8:
        oc = oracle.OracleCache(od, 32, 2, max_slots)
    else:  # both pools canary-filled, so every byte can be compared
        fill_canary(c)
        oc = oracle.OracleCache(od, 32, 2, max_slots, fill=CANARY)
    kvg.kvg_graft(store.h, bid, c.h, 0, -1, 0, kvg.KVG_GRAFT_VERIFY | kvg.KVG_GRAFT_SYNC)
    oc.graft(0, oracle.block_from_kv(od, k[:, :nb], v[:, :nb], syn.positions(0, nb)))
    append(kvg, c, 0, k[:, nb:], v[:, nb:], syn.positions(nb, nf))
    oc.append(0, k[:, nb:], v[:, nb:], syn.positions(nb, nf))
    append(kvg, c, 1, k[:, :1], v[:, :1], syn.positions(0, 1))
    oc.append(1, k[:, :1], v[:, :1], syn.positions(0, 1))
    return c, oc, (src, store)


@pytest.mark.parametrize("D,G", BF16_CASES, ids=[f"D{d}_G{g}" for d, g in BF16_CASES])
def test_decode_every_group_size(oracle, D, G):
    kvg = need_gpu()
    w = syn.Workload(f"d{D}g{G}", 2, 2 * G, 2, D, 16, 10000.0, 0x61 + G)
    c, oc, _keep = _sequence_case(kvg, oracle, w)
    q = syn.as_u16(syn.queries(w, w.n_layers, 2, 172))
    o = decode(kvg, c, w, [0, 1], q)
    scale = 1.0 / math.sqrt(D)
    for l in range(w.n_layers):
        for b in range(2):
            compare_decode(oracle, o[l, b], oc.decode(b, l, q[l, b], scale))
        # one row: the softmax weight is exactly 1, so o is that value row
        for h in range(w.n_q_heads):
            assert np.array_equal(o[l, 1, h], oc.pool[l, 1, oc.page_table[1, 0], h // G, 0])
    kvg.kvg_sync(c.h)


@pytest.mark.parametrize("D,G", FP8_CASES, ids=[f"D{d}_G{g}_fp8" for d, g in FP8_CASES])
def test_fp8_decode_every_group_size(oracle, D, G):
    kvg = need_gpu()
    w = syn.Workload(f"f{D}g{G}", 2, 2 * G, 2, D, 64, 10000.0, 0x71 + G)
    c, oc, _keep = _sequence_case(kvg, oracle, w, fp8=True)
    q = syn.as_u16(syn.queries(w, w.n_layers, 2, 173))
    o = decode(kvg, c, w, [0, 1], q)
    scale = 1.0 / math.sqrt(D)
    for l in range(w.n_layers):
        for b in range(2):
            compare_decode(oracle, o[l, b], oc.decode(b, l, q[l, b], scale))
    kvg.kvg_sync(c.h)


def test_one_row_pages(oracle):
    """page_size 1: every row its own page; grafts, appends and decode stay
    bit-exact / within tolerance."""
    kvg = need_gpu()
    w = syn.Workload("p1", 2, 4, 2, 64, 1, 10000.0, 0x81)
    c, oc, _keep = _sequence_case(kvg, oracle, w)
    assert np.array_equal(pool_u16(c, w), oc.pool)
    pt, pf, ps = tables(c)
    assert np.array_equal(pt, oc.page_table) and np.array_equal(pf, oc.page_fill)
    assert np.array_equal(ps, oc.positions)
    q = syn.as_u16(syn.queries(w, w.n_layers, 2, 174))
    o = decode(kvg, c, w, [0, 1], q)
    for l in range(w.n_layers):
        for b in range(2):
            compare_decode(oracle, o[l, b], oc.decode(b, l, q[l, b], 0.125))
    kvg.kvg_sync(c.h)


def test_one_token_block(oracle):
    """A block of one token: deposited, grafted (verified), decoded: o is its
    value row bit for bit."""
    kvg = need_gpu()
    w = syn.TINY
    dims, od = dims_for(kvg, w), oracle_dims(oracle, w)
    k, v = _kv(w, 1, 175)
    src = kvg.Cache(dims, 4, 1, 64)
    append(kvg, src, 0, k, v, syn.positions(7, 1))
    store = kvg.Store(dims, kvg.KVG_RESIDENCY_HBM, HBM_CAP)
    bid = kvg.kvg_deposit(store.h, src.h, 0, 0, 1)
    assert kvg.kvg_store_export(store.h, bid) == oracle.block_from_kv(od, k, v, syn.positions(7, 1)).serialize()
    c = kvg.Cache(dims, 4, 1, 64)
    kvg.kvg_graft(store.h, bid, c.h, 0, -1, 0, kvg.KVG_GRAFT_VERIFY | kvg.KVG_GRAFT_SYNC)
    assert kvg.kvg_cache_seq_info(c.h, 0) == (1, 1)
    q = syn.as_u16(syn.queries(w, w.n_layers, 1, 176))
    o = decode(kvg, c, w, [0], q)
    for l in range(w.n_layers):
        for h in range(w.n_q_heads):
            assert np.array_equal(o[l, 0, h], v[l, 0, h // w.group])
    kvg.kvg_sync(c.h)


def test_largest_decode_batch(oracle):
    """B = 4096 sequences (16 launches of 256 rows) of 1..19 rows each:
    sampled rows match the oracle; B = 4097 is refused."""
    kvg = need_gpu()
    w = syn.TINY
    P = w.page_size
    B = 4096
    dims, od = dims_for(kvg, w), oracle_dims(oracle, w)
    c = kvg.Cache(dims, 2 * B + 4, B + 1, 2 * P)
    oc = oracle.OracleCache(od, 2 * B + 4, B + 1, 2 * P)
    k, v = _kv(w, P + 3, 177)
    lens = [1 + (b * 5) % (P + 3) for b in range(B)]
    kd, vd = to_dev(k), to_dev(v)  # [L][P+3][Hkv][D]: each sequence takes a prefix of rows of every layer
    for b, n in enumerate(lens):
        kb = kd[:, :n].contiguous()
        vb = vd[:, :n].contiguous()
        pb = to_dev(syn.positions(0, n))
        kvg.kvg_cache_append(c.h, b, kb.data_ptr(), vb.data_ptr(), pb.data_ptr(), n)
        del kb, vb, pb  # freed after the call is enqueued: later reuse is ordered after it on this stream
        if b % 257 == 0 or b == B - 1:
            oc.append(b, np.ascontiguousarray(k[:, :n]), np.ascontiguousarray(v[:, :n]), syn.positions(0, n))
    torch.cuda.synchronize()
    q = syn.as_u16(syn.queries(w, w.n_layers, B, 178))
    o = decode(kvg, c, w, list(range(B)), q)
    scale = 1.0 / math.sqrt(w.head_dim)
    for b in list(range(0, B, 257)) + [B - 1]:
        for l in range(w.n_layers):
            compare_decode(oracle, o[l, b], oc.decode(b, l, q[l, b], scale))
    qd = to_dev(np.zeros((w.n_layers, B + 1, w.n_q_heads, w.head_dim), np.uint16))
    with pytest.raises(kvg.KvgError) as e:
        kvg.kvg_decode_attention(c.h, -1, list(range(B + 1)), qd.data_ptr(), w.n_q_heads, qd.data_ptr(), scale)
    assert e.value.status == kvg.KVG_ERR_ARG
    kvg.kvg_sync(c.h)


def test_empty_append_is_a_noop(oracle):
    kvg = need_gpu()
    w = syn.TINY
    c = kvg.Cache(dims_for(kvg, w), 8, 1, 64)
    k, v = _kv(w, 5, 179)
    append(kvg, c, 0, k, v, syn.positions(0, 5))
    before = tables(c)
    n0 = kvg.kvg_launch_count()
    kvg.kvg_cache_append(c.h, 0, 0, 0, 0, 0)
    assert kvg.kvg_launch_count() == n0
    assert kvg.kvg_cache_seq_info(c.h, 0) == (5, 1)
    after = tables(c)
    assert all(np.array_equal(a, b) for a, b in zip(before, after))


def test_positions_at_the_top_of_int32(oracle):
    """Position tags up to 2^31 - 1 graft and relocate; one more is refused."""
    kvg = need_gpu()
    w = syn.TINY
    dims, od = dims_for(kvg, w), oracle_dims(oracle, w)
    n = 21
    top = 2**31 - 1
    pos = np.arange(top - 40, top - 40 + n, dtype=np.int64).astype(np.int32)  # last tag top - 20
    k, v = _kv(w, n, 180)
    src = kvg.Cache(dims, 8, 1, 64)
    append(kvg, src, 0, k, v, pos)
    store = kvg.Store(dims, kvg.KVG_RESIDENCY_HBM, HBM_CAP)
    bid = kvg.kvg_deposit(store.h, src.h, 0, 0, n)
    c = kvg.Cache(dims, 16, 3, 64)
    fill_canary(c)
    oc = oracle.OracleCache(od, 16, 3, 64, fill=CANARY)
    kvg.kvg_graft(store.h, bid, c.h, 0, -1, 0, kvg.KVG_GRAFT_SYNC)
    oc.graft(0, oracle.block_from_kv(od, k, v, pos))
    assert np.array_equal(pool_u16(c, w), oc.pool)  # delta 0: bit-exact
    kvg.kvg_graft(store.h, bid, c.h, 1, -1, 20, kvg.KVG_GRAFT_SYNC)  # last tag exactly 2^31 - 1
    with pytest.raises(kvg.KvgError) as e:
        kvg.kvg_graft(store.h, bid, c.h, 2, -1, 21)
    assert e.value.status == kvg.KVG_ERR_POSITION
    _, _, ps = tables(c)
    assert np.array_equal(ps[0, :n], pos)
    assert int(ps[1, n - 1]) == top and np.array_equal(ps[1, :n], (pos.astype(np.int64) + 20).astype(np.int32))
    assert kvg.kvg_cache_seq_info(c.h, 2) == (0, 0)
    kvg.kvg_sync(c.h)


_CHILD = r'''
import hashlib, math, sys
sys.path.insert(0, sys.argv[1])
sys.path.insert(0, sys.argv[1] + "/tests")
import numpy as np, torch
import kvg_synth as syn
from kvg_testlib import append, decode, dims_for, need_gpu
kvg = need_gpu()
w = syn.Workload("repro", 3, 8, 4, 128, 64, 10000.0, 0x91)
k, v = syn.kv_rows(w, 1000, w.seed)
k, v = syn.as_u16(k), syn.as_u16(v)
dims = dims_for(kvg, w)
src = kvg.Cache(dims, 64, 1, 1088)
append(kvg, src, 0, k[:, :600], v[:, :600], syn.positions(0, 600))
store = kvg.Store(dims, kvg.KVG_RESIDENCY_HBM, 1 << 28)
bid = kvg.kvg_deposit(store.h, src.h, 0, 0, 600)
c = kvg.Cache(dims, 64, 1, 1088)
kvg.kvg_cache_set_free_order(c.h, syn.permutation(64, int(sys.argv[2])))
kvg.kvg_graft(store.h, bid, c.h, 0, -1, 0, kvg.KVG_GRAFT_VERIFY | kvg.KVG_GRAFT_SYNC)
append(kvg, c, 0, np.ascontiguousarray(k[:, 600:]), np.ascontiguousarray(v[:, 600:]), syn.positions(600, 400))
q = syn.as_u16(syn.queries(w, w.n_layers, 1, 0x92))
o = decode(kvg, c, w, [0], q)
print(hashlib.sha256(o.tobytes()).hexdigest())
'''


def test_outputs_are_identical_across_processes():
    """The paper's gate is byte equality between separate runs: the same
    graft + decode, run in two fresh processes (with different physical page
    placement), gives SHA-256-identical attention output."""
    import os
    import subprocess
    import sys
    need_gpu()
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    digests = []
    for placement_seed in (1, 2):
        r = subprocess.run([sys.executable, "-c", _CHILD, root, str(placement_seed)], capture_output=True, text=True,
                           timeout=600)
        assert r.returncode == 0, r.stderr[-2000:]
        digests.append(r.stdout.strip().splitlines()[-1])
    assert len(digests[0]) == 64 and digests[0] == digests[1]


_RELOC_CHILD = r'''
import hashlib, sys
sys.path.insert(0, sys.argv[1])
sys.path.insert(0, sys.argv[1] + "/tests")
import numpy as np, torch
import kvg_synth as syn
from kvg_testlib import append, dims_for, fill_canary, need_gpu, pool_u16
kvg = need_gpu()
out = []
for style in (0, 1):
    w = syn.Workload("reloc", 3, 8, 4, 128, 64, 1e6, 0x93)
    nb = 1000
    k, v = syn.kv_rows(w, nb, w.seed)
    k, v = syn.as_u16(k), syn.as_u16(v)
    dims = dims_for(kvg, w, style)
    src = kvg.Cache(dims, 40, 1, 1088)
    append(kvg, src, 0, k, v, syn.positions(0, nb))
    store = kvg.Store(dims, kvg.KVG_RESIDENCY_HBM, 1 << 28)
    bid = kvg.kvg_deposit(store.h, src.h, 0, 0, nb)
    c = kvg.Cache(dims, 40, 2, 1088)
    fill_canary(c)  # pages no graft writes hold known bytes
    kvg.kvg_graft(store.h, bid, c.h, 0, -1, 4096, kvg.KVG_GRAFT_SYNC)
    kvg.kvg_graft(store.h, bid, c.h, 1, -1, 0, kvg.KVG_GRAFT_SYNC)
    torch.cuda.synchronize()
    out.append(hashlib.sha256(pool_u16(c, w).tobytes()).hexdigest())
print(" ".join(out))
'''


def test_staged_and_register_grafts_write_identical_bytes():
    """An HBM-store graft runs through shared-memory stages by default and
    through registers with KVG_GRAFT_TMA_KB=0 (the pinned-host path): the
    relocated (delta 4096, half-split and interleaved) and own-position
    grafts of a ragged 1,000-token block leave byte-identical pools."""
    import os
    import subprocess
    import sys
    need_gpu()
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    digests = []
    for kb in ("192", "0"):
        env = dict(os.environ, KVG_GRAFT_TMA_KB=kb)
        r = subprocess.run([sys.executable, "-c", _RELOC_CHILD, root], capture_output=True, text=True, timeout=600,
                           env=env)
        assert r.returncode == 0, r.stderr[-2000:]
        digests.append(r.stdout.strip().splitlines()[-1])
    assert len(digests[0]) == 2 * 64 + 1 and digests[0] == digests[1]


def test_graft_of_pages_too_large_for_two_stages(oracle):
    """page_size 1023 (2 kv heads, head_dim 128): a page of 523,776 bytes
    halves once into 261,888-byte units (its rows do not halve again), more
    than two shared-memory stages hold, so the HBM-store graft takes the
    register copy instead.  The own-position graft of a ragged two-page block
    is bit-exact with the oracle (every pool byte, tables, positions); a
    relocated one (delta 4096, both RoPE styles) keeps values and padding
    bit-exact and keys within 2e-2 of the fp64 rotation."""
    kvg = need_gpu()
    w = syn.Workload("p1023", 2, 4, 2, 128, 1023, 10000.0, 0x95)
    P = w.page_size
    nb = P + 500
    k, v = _kv(w, nb, 176)
    max_slots, n_pages = 4 * P, 8
    for style in (0, 1):
        dims, od = dims_for(kvg, w, style), oracle_dims(oracle, w, style)
        src = kvg.Cache(dims, n_pages, 1, max_slots)
        append(kvg, src, 0, k, v, syn.positions(0, nb))
        store = kvg.Store(dims, kvg.KVG_RESIDENCY_HBM, HBM_CAP)
        bid = kvg.kvg_deposit(store.h, src.h, 0, 0, nb)
        c = kvg.Cache(dims, n_pages, 2, max_slots)
        fill_canary(c)
        oc = oracle.OracleCache(od, n_pages, 2, max_slots, fill=CANARY)
        oblk = oracle.block_from_kv(od, k, v, syn.positions(0, nb))
        kvg.kvg_graft(store.h, bid, c.h, 0, -1, 0, kvg.KVG_GRAFT_SYNC)
        oc.graft(0, oblk)
        assert np.array_equal(pool_u16(c, w), oc.pool)
        kvg.kvg_graft(store.h, bid, c.h, 1, -1, 4096, kvg.KVG_GRAFT_SYNC)
        oc.graft(1, oblk, delta=4096)
        pool = pool_u16(c, w)
        pt, pf, ps = tables(c)
        assert np.array_equal(pt, oc.page_table) and np.array_equal(pf, oc.page_fill)
        assert np.array_equal(ps, oc.positions)
        assert np.array_equal(pool[:, 1], oc.pool[:, 1])  # values
        k64 = np.stack([oracle.rope_rotate_rows(k[l], 4096, w.rope_theta, style) for l in range(w.n_layers)])
        kg = np.empty_like(k)
        for t in range(nb):
            j, r = divmod(t, P)
            kg[:, t] = pool[:, 0, pt[1, j], :, r, :]
        assert np.abs(oracle.bf16_to_f64(kg) - k64).max() <= 2e-2
        check_rotation_rounding(oracle, kg, k64)
        j, r = divmod(nb, P)  # padding rows of the last page: copied unchanged (zeros)
        assert not pool[:, 0, pt[1, j], :, r:, :].any()
        kvg.kvg_sync(c.h)


def test_large_verified_graft_with_ragged_leaves(oracle):
    """A verified graft large enough for the shared-memory ring form of the
    one-pass kernel (a full wave of it: 98,304 leaves here) on pages of 4,224
    bytes, so every page has a full 4 KiB leaf and a 128-byte one: the
    deposited block equals the oracle's (49,152 page digests), the graft
    restores every pool byte as the oracle's cache holds it and checks every
    page, and a flipped byte is reported at its page."""
    kvg = need_gpu()
    w = syn.Workload("ragleaf", 24, 2, 1, 64, 33, 10000.0, 0x7A)  # page: 1 x 33 x 64 x 2 = 4,224 bytes
    P = w.page_size
    npb = 1024
    n = npb * P
    k, v = syn.kv_rows(w, n, w.seed)
    k, v = syn.as_u16(k), syn.as_u16(v)
    dims = dims_for(kvg, w)
    src = kvg.Cache(dims, npb + 2, 1, n + P)
    append(kvg, src, 0, k, v, syn.positions(0, n))
    store = kvg.Store(dims, kvg.KVG_RESIDENCY_HBM, 1 << 30)
    bid = kvg.kvg_deposit(store.h, src.h, 0, 0, n)
    od = oracle_dims(oracle, w)
    blk = oracle.block_from_kv(od, k, v, syn.positions(0, n))
    ser = blk.serialize()
    assert kvg.kvg_store_export(store.h, bid) == ser
    src.close()
    dst = kvg.Cache(dims, npb + 2, 1, n + P)
    fill_canary(dst)
    oc = oracle.OracleCache(od, npb + 2, 1, n + P, fill=CANARY)
    rep = kvg.kvg_graft_report()
    kvg.kvg_graft(store.h, bid, dst.h, 0, -1, 0, kvg.KVG_GRAFT_VERIFY | kvg.KVG_GRAFT_SYNC, report=rep)
    assert rep.n_mismatch == 0 and rep.n_pages_checked == w.n_layers * 2 * npb
    oc.graft(0, blk)
    assert np.array_equal(pool_u16(dst, w), oc.pool)
    # one flipped byte in the short leaf of page (plane 37, page 700)
    info = kvg.kvg_store_block_info(store.h, bid)
    bad = bytearray(ser)
    bad_page = 37 * npb + 700
    bad[info.pages_offset + bad_page * w.page_bytes + 4096 + 77] ^= 0x10
    bid2 = kvg.kvg_store_import(store.h, bytes(bad), 0)
    kvg.kvg_cache_release(dst.h, 0)
    with pytest.raises(kvg.KvgError) as e:
        kvg.kvg_graft(store.h, bid2, dst.h, 0, -1, 0, kvg.KVG_GRAFT_VERIFY | kvg.KVG_GRAFT_SYNC, report=rep)
    assert e.value.status == kvg.KVG_ERR_DIGEST
    assert rep.n_mismatch == 1 and rep.mismatch_pages[0] == bad_page
    kvg.kvg_sync(dst.h)


def test_graft_batch_host_checks_change_nothing(oracle):
    """kvg_graft_batch's host checks: an empty or oversized batch, a bad
    sequence id, an unknown block, a delta pushing a tag out of range, and a
    pool-resident store are all refused with their status before any work,
    and the cache is unchanged (no pages taken, no tags written)."""
    kvg = need_gpu()
    w = syn.TINY
    dims = dims_for(kvg, w)
    src = kvg.Cache(dims, 40, 1, 512)
    k, v = _kv(w, 100, 0x51)
    append(kvg, src, 0, k, v, syn.positions(0, 100))
    store = kvg.Store(dims, kvg.KVG_RESIDENCY_HBM, 1 << 24)
    bid = kvg.kvg_deposit(store.h, src.h, 0, 0, 100)
    c = kvg.Cache(dims, 40, 2, 512)
    fill_canary(c)
    before = pool_u16(c, w).copy()
    cases = [
        (lambda: kvg.kvg_graft_batch(store.h, [bid] * 4097, c.h, [0] * 4097), kvg.KVG_ERR_ARG),
        (lambda: kvg.kvg_graft_batch(store.h, [bid], c.h, [2]), kvg.KVG_ERR_ARG),
        (lambda: kvg.kvg_graft_batch(store.h, [bid, bid + 7], c.h, [0, 1]), kvg.KVG_ERR_NOT_FOUND),
        (lambda: kvg.kvg_graft_batch(store.h, [bid, bid], c.h, [0, 1], deltas=[3, -4]), kvg.KVG_ERR_POSITION),
        (lambda: kvg.kvg_graft_batch(store.h, [bid, bid], c.h, [0, 1], deltas=[0, 2 ** 31 - 50]),
         kvg.KVG_ERR_POSITION),
    ]
    pool_store = kvg.PoolStore(src, 1 << 22)
    pbid = kvg.kvg_deposit(pool_store.h, src.h, 0, 0, 100)
    cases.append((lambda: kvg.kvg_graft_batch(pool_store.h, [pbid], src.h, [0]), kvg.KVG_ERR_ARG))
    for call, status in cases:
        with pytest.raises(kvg.KvgError) as e:
            call()
        assert e.value.status == status, (e.value.status, status)
    assert kvg.kvg_cache_seq_info(c.h, 0) == (0, 0) and kvg.kvg_cache_seq_info(c.h, 1) == (0, 0)
    assert np.array_equal(pool_u16(c, w), before)
    pt, pf, ps = tables(c)
    assert (pt == -1).all() and (pf == 0).all() and (ps == -1).all()
    # and the same batch with valid arguments then works
    kvg.kvg_graft_batch(store.h, [bid, bid], c.h, [0, 1], kvg.KVG_GRAFT_VERIFY | kvg.KVG_GRAFT_SYNC, deltas=[0, 9])
    assert kvg.kvg_cache_seq_info(c.h, 1)[0] == 100
    kvg.kvg_sync(c.h)


def test_two_caches_on_two_streams_match_serial(oracle):
    """Different caches are independent: the same deposit / verified graft /
    append / decode sequence issued on two caches from two streams at once,
    each with its own store, gives the same bytes as the sequence run alone,
    and the oracle's decode through the gate."""
    kvg = need_gpu()
    w = geometry("d256")
    P = w.page_size
    dims = dims_for(kvg, w)
    nb, nf = 5 * P + 9, 3 * P + 1
    k, v = _kv(w, nb + nf, 0x2C)
    q = syn.as_u16(syn.queries(w, w.n_layers, 1, 0x2D))
    scale = 1.0 / math.sqrt(w.head_dim)

    def run(stream, sync_each=False):
        src = kvg.Cache(dims, 16, 1, 16 * P)
        store = kvg.Store(dims, kvg.KVG_RESIDENCY_HBM, 1 << 26)
        dst = kvg.Cache(dims, 16, 1, 16 * P)
        # k, v arguments are [L][n][Hkv][D] for the n rows appended
        kd, vd = to_dev(np.ascontiguousarray(k[:, :nb])), to_dev(np.ascontiguousarray(v[:, :nb]))
        pos = to_dev(syn.positions(0, nb))
        h = stream.cuda_stream
        kvg.kvg_cache_append(src.h, 0, kd.data_ptr(), vd.data_ptr(), pos.data_ptr(), nb, h)
        bid = kvg.kvg_deposit(store.h, src.h, 0, 0, nb, h)
        kvg.kvg_graft(store.h, bid, dst.h, 0, -1, 0, kvg.KVG_GRAFT_VERIFY, h)
        kf, vf = to_dev(np.ascontiguousarray(k[:, nb:])), to_dev(np.ascontiguousarray(v[:, nb:]))
        pf = to_dev(syn.positions(nb, nf))
        kvg.kvg_cache_append(dst.h, 0, kf.data_ptr(), vf.data_ptr(), pf.data_ptr(), nf, h)
        qd = to_dev(q)
        out = torch.empty_like(qd)
        kvg.kvg_decode_attention(dst.h, -1, [0], qd.data_ptr(), w.n_q_heads, out.data_ptr(), scale, h)
        return out, (src, store, dst, kd, vd, pos, kf, vf, pf, qd)

    s0 = torch.cuda.Stream()
    ref, keep0 = run(s0)
    s0.synchronize()
    ref = u16(ref)
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    o1, keep1 = run(s1)
    o2, keep2 = run(s2)
    torch.cuda.synchronize()
    for keep in (keep0, keep1, keep2):
        kvg.kvg_sync(keep[2].h)
    assert np.array_equal(u16(o1), ref) and np.array_equal(u16(o2), ref)
    for l in range(w.n_layers):
        compare_decode(oracle, ref[l, 0], oracle.gqa_decode(q[l, 0], k[l], v[l], scale), what=f"two streams l {l}")


@pytest.mark.gpu
def test_paged_digests_on_two_streams_match_the_oracle(oracle):
    """Paged digests share the device's leaf scratch: two calls launched
    back to back on two streams (the second larger than the first, so the
    scratch may have to grow) each give the oracle's page digests."""
    kvg = need_gpu()
    pb = 262144
    rng = np.random.default_rng(77)
    sizes = (128, 256)  # pages of 256 KiB
    host = [rng.integers(0, 256, n * pb, dtype=np.uint8) for n in sizes]
    want = [oracle.page_digests(h, pb) for h in host]
    bufs = [torch.from_numpy(h).cuda() for h in host]
    streams = [torch.cuda.Stream(), torch.cuda.Stream()]
    for rep in range(3):
        outs = [torch.zeros(n * 32, dtype=torch.uint8, device="cuda") for n in sizes]
        torch.cuda.synchronize()
        order = (0, 1) if rep % 2 == 0 else (1, 0)
        for i in order:
            kvg.kvg_digest(bufs[i].data_ptr(), bufs[i].numel(), kvg.KVG_SHA256_PAGED, pb, outs[i].data_ptr(),
                           streams[i])
        torch.cuda.synchronize()
        for i, n in enumerate(sizes):
            assert np.array_equal(outs[i].cpu().numpy().reshape(n, 32), want[i]), (rep, i)


@pytest.mark.gpu
def test_decodes_of_one_cache_on_two_streams_match_serial(oracle):
    """Decodes of one cache share its split-K scratch: a long decode (32
    sequences of 4,096 rows, two layers: 512 MiB of K/V) and a second one
    with other queries and the batch rows in reverse order, launched back to
    back on two streams, each give the bytes they give one after the other
    on one stream."""
    kvg = need_gpu()
    w = geometry("d256")
    P = w.page_size
    dims = dims_for(kvg, w)
    n_seq, n = 32, 64 * P
    k, v = _kv(w, n, 0x31)
    cache = kvg.Cache(dims, n_seq * (n // P), n_seq, n)
    kd, vd = to_dev(k), to_dev(v)
    pos = to_dev(syn.positions(0, n))
    h = torch.cuda.current_stream().cuda_stream
    for s in range(n_seq):
        kvg.kvg_cache_append(cache.h, s, kd.data_ptr(), vd.data_ptr(), pos.data_ptr(), n, h)
    qa = syn.as_u16(syn.queries(w, w.n_layers, n_seq, 0x32))
    qb = syn.as_u16(syn.queries(w, w.n_layers, n_seq, 0x33))
    qa_d, qb_d = to_dev(qa), to_dev(qb)
    seqs_a, seqs_b = list(range(n_seq)), list(range(n_seq))[::-1]
    scale = 1.0 / math.sqrt(w.head_dim)

    def dec(q_d, seqs, stream):
        out = torch.empty_like(q_d)
        kvg.kvg_decode_attention(cache.h, -1, seqs, q_d.data_ptr(), w.n_q_heads, out.data_ptr(), scale,
                                 stream.cuda_stream)
        return out

    torch.cuda.synchronize()
    s0 = torch.cuda.Stream()
    ra, rb = dec(qa_d, seqs_a, s0), dec(qb_d, seqs_b, s0)
    s0.synchronize()
    ref_a, ref_b = u16(ra), u16(rb)
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    for rep in range(3):
        oa = dec(qa_d, seqs_a, s1)
        ob = dec(qb_d, seqs_b, s2)
        torch.cuda.synchronize()
        assert np.array_equal(u16(oa), ref_a) and np.array_equal(u16(ob), ref_b), rep
    kvg.kvg_sync(cache.h)
    for l in range(w.n_layers):
        compare_decode(oracle, ref_a[l, 0], oracle.gqa_decode(qa[l, 0], k[l], v[l], scale), what=f"stream a l {l}")
        compare_decode(oracle, ref_b[l, 0], oracle.gqa_decode(qb[l, 0], k[l], v[l], scale), what=f"stream b l {l}")


_DIGEST_CHILD = r'''
import sys
sys.path.insert(0, sys.argv[1])
sys.path.insert(0, sys.argv[1] + "/tests")
import numpy as np, torch
import kvg_synth as syn
from kvg_testlib import append, dims_for, need_gpu, geometry
kvg = need_gpu()
rng = np.random.default_rng(91)
out = []
# paged digests of a small launch: 96 pages of 4 KiB and 40 pages of 64 KiB
for n, pb in ((96, 4096), (40, 65536)):
    buf = torch.from_numpy(rng.integers(0, 256, n * pb, dtype=np.uint8)).cuda()
    o = torch.zeros(n * 32, dtype=torch.uint8, device="cuda")
    kvg.kvg_digest(buf.data_ptr(), buf.numel(), kvg.KVG_SHA256_PAGED, pb, o.data_ptr())
    out.append(bytes(o.cpu().numpy()).hex())
# a plain digest of 100,000 bytes
buf = torch.from_numpy(rng.integers(0, 256, 100000, dtype=np.uint8)).cuda()
o = torch.zeros(32, dtype=torch.uint8, device="cuda")
kvg.kvg_digest(buf.data_ptr(), buf.numel(), kvg.KVG_SHA256_PLAIN, 0, o.data_ptr())
out.append(bytes(o.cpu().numpy()).hex())
# a deposit and a verified graft of a 100-token block (tiny geometry: 4 KiB pages)
w = geometry("tiny")
k, v = syn.kv_rows(w, 100, 0x77)
dims = dims_for(kvg, w)
src = kvg.Cache(dims, 32, 1, 256)
append(kvg, src, 0, syn.as_u16(k), syn.as_u16(v), syn.positions(0, 100))
store = kvg.Store(dims, kvg.KVG_RESIDENCY_HBM, 1 << 24)
bid = kvg.kvg_deposit(store.h, src.h, 0, 0, 100)
out.append(kvg.kvg_store_export(store.h, bid).hex())
dst = kvg.Cache(dims, 32, 1, 256)
kvg.kvg_graft(store.h, bid, dst.h, 0, -1, 0, kvg.KVG_GRAFT_VERIFY | kvg.KVG_GRAFT_SYNC)
print("\n".join(out))
'''


def test_two_warp_and_one_warp_hashing_agree_with_the_oracle(oracle):
    """Small launches hash in the two-warp form; KVG_SHA_NO_SPLIT=1 keeps the
    one-warp forms.  Both give the oracle's page digests, plain digest and
    deposited block (whose page and block digests they compute), and a
    verified graft of the block passes in both."""
    import os
    import subprocess
    import sys
    need_gpu()
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    res = []
    for off in ("0", "1"):
        env = dict(os.environ, KVG_SHA_NO_SPLIT=off)
        r = subprocess.run([sys.executable, "-c", _DIGEST_CHILD, root], capture_output=True, text=True, timeout=600,
                           env=env)
        assert r.returncode == 0, r.stderr[-2000:]
        res.append(r.stdout.strip().splitlines()[-4:])
    assert res[0] == res[1]
    rng = np.random.default_rng(91)
    for got, (n, pb) in zip(res[0][:2], ((96, 4096), (40, 65536))):
        assert bytes.fromhex(got) == oracle.page_digests(rng.integers(0, 256, n * pb, dtype=np.uint8), pb).tobytes()
    assert bytes.fromhex(res[0][2]) == oracle.sha256(rng.integers(0, 256, 100000, dtype=np.uint8).tobytes())
    w = geometry("tiny")
    k, v = syn.kv_rows(w, 100, 0x77)
    blk = oracle.block_from_kv(oracle_dims(oracle, w), syn.as_u16(k), syn.as_u16(v), syn.positions(0, 100))
    assert bytes.fromhex(res[0][3]) == blk.serialize()
