"""GPU parity: the CUDA library (through its C ABI) against the CPU oracle on
the same seeded inputs.  Graft, page tables, positions, block bytes and
digests must match bit for bit; decode attention within 1e-2 max-abs of the
fp64 oracle (bf16 out, fp32 accumulate), within 2^-7 of its largest element
and with at least 35% of elements equal to the oracle's bf16 rounding
(kvg_testlib.compare_decode); relocated keys within 2e-2 of the fp64
rotation; grafted-vs-fresh attention outputs SHA-256-identical."""
import hashlib
import math

import numpy as np
import pytest
import torch

import kvg_synth as syn
from kvg_testlib import (CANARY, REL_TOL_RELOCATED, RNE_FLOOR_RELOCATED, append, check_rotation_rounding, compare_decode,
                         decode, dev_view,
                         dims_for, fill_canary, geometry, need_gpu, oracle_dims, pool_u16, tables, to_dev, u16)

pytestmark = pytest.mark.gpu

HBM_CAP = 8 << 30


def _kv(w, n, seed):
    k, v = syn.kv_rows(w, n, seed)
    return syn.as_u16(k), syn.as_u16(v)


def _slots(w, n):
    return (-(-n // w.page_size) + 2) * w.page_size


def _sha(a: np.ndarray) -> bytes:
    return hashlib.sha256(np.ascontiguousarray(a).tobytes()).digest()


# ------------------------------------------------------------------- digests

NIST = [b"", b"abc", b"abcdbcdecdefdefgefghfghighijhijkijkljklmklmnlmnomnopnopq", b"a" * 1_000_000,
        bytes(range(256)) * 3 + b"xyz"]


@pytest.mark.parametrize("msg", NIST, ids=["empty", "abc", "448bit", "million_a", "odd_len"])
def test_digest_plain_matches_hashlib(msg):
    kvg = need_gpu()
    buf = torch.frombuffer(bytearray(msg or b"\0"), dtype=torch.uint8).cuda()
    out = torch.zeros(32, dtype=torch.uint8, device="cuda")
    kvg.kvg_digest(buf.data_ptr(), len(msg), kvg.KVG_SHA256_PLAIN, 0, out.data_ptr())
    torch.cuda.synchronize()
    assert bytes(out.cpu().numpy()) == hashlib.sha256(msg).digest()


@pytest.mark.parametrize("page_bytes,n_pages", [(4096, 7), (262144, 5), (10000, 3), (64, 9), (65552, 2)])
def test_digest_paged_matches_oracle(oracle, page_bytes, n_pages):
    kvg = need_gpu()
    rng = np.random.default_rng(page_bytes)
    data = rng.integers(0, 256, page_bytes * n_pages, dtype=np.uint8)
    d = torch.from_numpy(data).cuda()
    out = torch.zeros(32 * n_pages, dtype=torch.uint8, device="cuda")
    kvg.kvg_digest(d.data_ptr(), data.size, kvg.KVG_SHA256_PAGED, page_bytes, out.data_ptr())
    torch.cuda.synchronize()
    assert np.array_equal(out.cpu().numpy().reshape(n_pages, 32), oracle.page_digests(data, page_bytes))


# ------------------------------------------------------------ graft parity

CASES = [("tiny", 256, 0), ("tiny", 250, 37), ("d128", 1000, 700), ("d256", 700, 300), ("g4", 333, 100)]


def _build_both(kvg, oracle, w, nb, nf, residency=0, style=0, seed=1, copies=1):
    """Deposits an nb-token block from a freshly written sequence and grafts
    it (then appends nf fresh tokens) into a canary-filled cache, on both
    sides.  Returns everything the tests compare."""
    k, v = _kv(w, nb + nf, seed)
    max_slots = _slots(w, nb + nf)
    n_pages = (max_slots // w.page_size + 3) * copies
    dims = dims_for(kvg, w, style)
    src = kvg.Cache(dims, n_pages, 2, max_slots)
    kvg.kvg_cache_set_free_order(src.h, syn.permutation(n_pages, seed + 7))
    append(kvg, src, 0, k[:, :nb], v[:, :nb], syn.positions(0, nb))
    store = kvg.Store(dims, residency, HBM_CAP)
    bid = kvg.kvg_deposit(store.h, src.h, 0, 0, nb)
    dst = kvg.Cache(dims, n_pages, 3, max_slots)
    fill_canary(dst)
    od = oracle_dims(oracle, w, style)
    oblk = oracle.block_from_kv(od, k[:, :nb], v[:, :nb], syn.positions(0, nb))
    ocache = oracle.OracleCache(od, n_pages, 3, max_slots, fill=CANARY)
    return dict(k=k, v=v, src=src, store=store, bid=bid, dst=dst, oblk=oblk, ocache=ocache,
                n_pages=n_pages, max_slots=max_slots, dims=dims)


@pytest.mark.parametrize("geo,nb,nf", CASES)
def test_deposit_graft_append_bit_exact(oracle, geo, nb, nf):
    kvg = need_gpu()
    w = geometry(geo)
    s = _build_both(kvg, oracle, w, nb, nf)
    # deposit: the serialized block equals the oracle's byte for byte
    assert kvg.kvg_store_export(s["store"].h, s["bid"]) == s["oblk"].serialize()
    info = kvg.kvg_store_block_info(s["store"].h, s["bid"])
    assert bytes(info.block_digest) == s["oblk"].block_digest
    rep = kvg.kvg_graft_report()
    kvg.kvg_graft(s["store"].h, s["bid"], s["dst"].h, 1, -1, 0, kvg.KVG_GRAFT_VERIFY | kvg.KVG_GRAFT_SYNC,
                  report=rep)
    assert rep.n_mismatch == 0 and rep.n_pages_checked == w.n_layers * 2 * s["oblk"].n_pages
    append(kvg, s["dst"], 1, s["k"][:, nb:], s["v"][:, nb:], syn.positions(nb, nf))
    oc = s["ocache"]
    oc.graft(1, s["oblk"])
    oc.append(1, s["k"][:, nb:], s["v"][:, nb:], syn.positions(nb, nf))
    assert np.array_equal(pool_u16(s["dst"], w), oc.pool)
    pt, pf, ps = tables(s["dst"])
    assert np.array_equal(pt, oc.page_table) and np.array_equal(pf, oc.page_fill)
    assert np.array_equal(ps, oc.positions)
    assert kvg.kvg_cache_seq_info(s["dst"].h, 1) == (nb + nf, int((oc.page_table[1] >= 0).sum()))


@pytest.mark.parametrize("geo,nb,nf", [("tiny", 250, 37), ("d256", 700, 300)])
def test_pinned_host_store_graft_bit_exact(oracle, geo, nb, nf):
    kvg = need_gpu()
    w = geometry(geo)
    s = _build_both(kvg, oracle, w, nb, nf, residency=kvg.KVG_RESIDENCY_PINNED_HOST, seed=3)
    assert kvg.kvg_store_export(s["store"].h, s["bid"]) == s["oblk"].serialize()
    kvg.kvg_graft(s["store"].h, s["bid"], s["dst"].h, 0, -1, 0, kvg.KVG_GRAFT_VERIFY | kvg.KVG_GRAFT_SYNC)
    s["ocache"].graft(0, s["oblk"])
    assert np.array_equal(pool_u16(s["dst"], w), s["ocache"].pool)


# ----------------------------------------------------------- decode parity

@pytest.mark.parametrize("geo,nb,nf", CASES)
def test_decode_matches_oracle_and_grafted_equals_fresh(oracle, geo, nb, nf):
    kvg = need_gpu()
    w = geometry(geo)
    s = _build_both(kvg, oracle, w, nb, nf, seed=11)
    kvg.kvg_graft(s["store"].h, s["bid"], s["dst"].h, 2, -1, 0, kvg.KVG_GRAFT_SYNC)
    append(kvg, s["dst"], 2, s["k"][:, nb:], s["v"][:, nb:], syn.positions(nb, nf))
    q = syn.as_u16(syn.queries(w, w.n_layers, 1, 11))
    o = decode(kvg, s["dst"], w, [2], q)
    scale = 1.0 / math.sqrt(w.head_dim)
    for l in range(w.n_layers):
        ref = oracle.gqa_decode(q[l, 0], s["k"][l], s["v"][l], scale)
        compare_decode(oracle, o[l, 0], ref)
    # the same rows written fresh into differently placed pages: identical bytes
    fresh = kvg.Cache(s["dims"], s["n_pages"], 1, s["max_slots"])
    kvg.kvg_cache_set_free_order(fresh.h, syn.permutation(s["n_pages"], 99))
    append(kvg, fresh, 0, s["k"], s["v"], syn.positions(0, nb + nf))
    of = decode(kvg, fresh, w, [0], q)
    assert _sha(of) == _sha(o)
    # run-to-run bitwise determinism
    for _ in range(3):
        assert _sha(decode(kvg, s["dst"], w, [2], q)) == _sha(o)
    # one layer at a time is within tolerance too
    for l in range(w.n_layers):
        ol = decode(kvg, s["dst"], w, [2], q[l:l + 1], layer=l)
        compare_decode(oracle, ol[0, 0], oracle.gqa_decode(q[l, 0], s["k"][l], s["v"][l], scale))


def _windows(w):
    P = w.page_size
    return [(1, P + 3, 0, 2 * P + 5)[l % 4] for l in range(w.n_layers)]


@pytest.mark.parametrize("geo", ["tiny", "d128", "d256", "g4"])
def test_windowed_decode_matches_oracle(oracle, geo):
    """Sliding-window layers over a full-size cache: per-layer windows 1,
    P+3, 0 (global), 2P+5.  Seq 0 holds a ragged grafted block, fresh rows on
    its last page, a second block grafted at the next page boundary (leaving
    unfilled rows the window must skip) and more fresh rows; seq 1 one long
    fresh write; seq 2 three rows.  All layers in one call and one layer at a
    time match the fp64 oracle; a window of one returns the last value row bit
    for bit; a grafted sequence equals the same rows written fresh, bit for
    bit, under the windows."""
    kvg = need_gpu()
    w = geometry(geo)
    P = w.page_size
    dims = dims_for(kvg, w)
    od = oracle_dims(oracle, w)
    na, nb_, nc, nd = 2 * P + 5, P + 2, P + 7, 3
    k, v = _kv(w, na + nb_ + nc + nd + 5 * P, 81)
    parts, t = [], 0
    for n in (na, nb_, nc, nd):
        parts.append((k[:, t:t + n], v[:, t:t + n], syn.positions(t, n)))
        t += n
    n_long = 5 * P
    k_long, v_long = k[:, t:t + n_long], v[:, t:t + n_long]
    max_slots = 8 * P + 64
    n_pages = 64
    # the two blocks, deposited from a source cache
    src = kvg.Cache(dims, n_pages, 2, max_slots)
    store = kvg.Store(dims, 0, HBM_CAP)
    bids = []
    for i, (kk, vv, pp) in enumerate((parts[0], parts[2])):
        append(kvg, src, i, kk, vv, pp)
        bids.append(kvg.kvg_deposit(store.h, src.h, i, 0, pp.size))
    c = kvg.Cache(dims, n_pages, 5, max_slots)
    fill_canary(c)
    kvg.kvg_cache_set_free_order(c.h, syn.permutation(n_pages, 82))
    oc = oracle.OracleCache(od, n_pages, 5, max_slots, fill=CANARY)
    oc.set_free_order(syn.permutation(n_pages, 82))
    kvg.kvg_graft(store.h, bids[0], c.h, 0, -1, 0, kvg.KVG_GRAFT_SYNC)
    oc.graft(0, oracle.block_from_kv(od, *parts[0]))
    append(kvg, c, 0, *parts[1])
    oc.append(0, *parts[1])
    kvg.kvg_graft(store.h, bids[1], c.h, 0, -1, 0, kvg.KVG_GRAFT_SYNC)
    oc.graft(0, oracle.block_from_kv(od, *parts[2]))
    append(kvg, c, 0, *parts[3])
    oc.append(0, *parts[3])
    append(kvg, c, 1, k_long, v_long, syn.positions(0, n_long))
    oc.append(1, k_long, v_long, syn.positions(0, n_long))
    append(kvg, c, 2, k[:, :3], v[:, :3], syn.positions(0, 3))
    oc.append(2, k[:, :3], v[:, :3], syn.positions(0, 3))
    # grafted (seq 3) and fresh (seq 4) copies of block A + fresh rows
    kvg.kvg_graft(store.h, bids[0], c.h, 3, -1, 0, kvg.KVG_GRAFT_SYNC)
    append(kvg, c, 3, *parts[1])
    append(kvg, c, 4, np.concatenate([parts[0][0], parts[1][0]], 1), np.concatenate([parts[0][1], parts[1][1]], 1),
           syn.positions(0, na + nb_))
    wins = _windows(w)
    kvg.kvg_cache_set_layer_windows(c.h, wins)
    oc.set_layer_windows(wins)
    scale = 1.0 / math.sqrt(w.head_dim)
    rows = [0, 1, 2]
    q = syn.as_u16(syn.queries(w, w.n_layers, len(rows), 83))
    o = decode(kvg, c, w, rows, q)
    G = w.group
    for l in range(w.n_layers):
        for b, sq in enumerate(rows):
            compare_decode(oracle, o[l, b], oc.decode(sq, l, q[l, b], scale))
            ol = decode(kvg, c, w, [sq], q[l:l + 1, b:b + 1], layer=l)
            compare_decode(oracle, ol[0, 0], oc.decode(sq, l, q[l, b], scale))
        if wins[l] == 1:
            kk, vv, _ = oc.logical_kv(0, l)
            for h in range(w.n_q_heads):
                assert np.array_equal(o[l, 0, h], vv[-1, h // G])
    q2 = syn.as_u16(syn.queries(w, w.n_layers, 1, 84))
    assert _sha(decode(kvg, c, w, [3], q2)) == _sha(decode(kvg, c, w, [4], q2))
    # the windows only select rows: resetting them gives global attention again
    kvg.kvg_cache_set_layer_windows(c.h, [])
    og = decode(kvg, c, w, [0], q[:, :1])
    for l in range(w.n_layers):
        kk, vv, _ = oc.logical_kv(0, l)
        compare_decode(oracle, og[l, 0], oracle.gqa_decode(q[l, 0], kk, vv, scale))
    kvg.kvg_sync(c.h)


def test_decode_closed_forms(oracle):
    kvg = need_gpu()
    w = geometry("d128")
    dims = dims_for(kvg, w)
    cache = kvg.Cache(dims, 16, 4, 512)
    scale = 1 / math.sqrt(w.head_dim)
    # one token: the softmax weight is exactly 1, so o is v0 bit for bit
    k, v = _kv(w, 1, 21)
    append(kvg, cache, 0, k, v, syn.positions(0, 1))
    q = syn.as_u16(syn.queries(w, w.n_layers, 1, 21))
    o = decode(kvg, cache, w, [0], q)
    G = w.group
    for l in range(w.n_layers):
        for h in range(w.n_q_heads):
            assert np.array_equal(o[l, 0, h], v[l, 0, h // G])
    # every value row equal: o equals that row
    n = 300
    k2, _ = _kv(w, n, 22)
    row = syn.as_u16(syn.normal_bf16((w.n_layers, 1, w.n_kv_heads, w.head_dim), 23))
    v2 = np.repeat(row, n, axis=1)
    append(kvg, cache, 1, k2, v2, syn.positions(0, n))
    o2 = decode(kvg, cache, w, [1], q)
    for l in range(w.n_layers):
        for h in range(w.n_q_heads):
            assert np.array_equal(o2[l, 0, h], row[l, 0, h // G])
    # empty sequence: zeros; a batch mixing empty and non-empty rows
    o3 = decode(kvg, cache, w, [3, 0, 1], np.repeat(q, 3, axis=1))
    assert not o3[:, 0].any()
    assert np.array_equal(o3[:, 1], o[:, 0])


def test_decode_batch_ragged_vs_oracle(oracle):
    kvg = need_gpu()
    w = geometry("d256")
    dims = dims_for(kvg, w)
    lens = [1, 63, 64, 65, 500, 1111]
    max_slots = _slots(w, max(lens))
    cache = kvg.Cache(dims, sum(-(-n // w.page_size) for n in lens) + 4, len(lens), max_slots)
    kvs = []
    for i, n in enumerate(lens):
        k, v = _kv(w, n, 30 + i)
        kvs.append((k, v))
        append(kvg, cache, i, k, v, syn.positions(0, n))
    order = [5, 0, 3, 1, 4, 2]
    q = syn.as_u16(syn.queries(w, w.n_layers, len(order), 31))
    o = decode(kvg, cache, w, order, q)
    for bi, sq in enumerate(order):
        k, v = kvs[sq]
        for l in range(w.n_layers):
            compare_decode(oracle, o[l, bi], oracle.gqa_decode(q[l, bi], k[l], v[l], 1 / math.sqrt(w.head_dim)))


# --------------------------------------------------------------- relocation

def _logical_k(pool, pt, w, seq, n):
    out = np.zeros((w.n_layers, n, w.n_kv_heads, w.head_dim), np.uint16)
    for t in range(n):
        j, r = divmod(t, w.page_size)
        out[:, t] = pool[:, 0, pt[seq, j], :, r, :]
    return out


@pytest.mark.parametrize("geo,style", [("tiny", 0), ("d128", 0), ("d128", 1), ("d256", 0)])
def test_relocated_graft_within_tolerance(oracle, geo, style):
    kvg = need_gpu()
    w = geometry(geo)
    nb = 200 if geo != "d128" else 333
    s = _build_both(kvg, oracle, w, nb, 0, style=style, seed=41, copies=3)
    # own position through the relocation entry with delta = 0 is the pure copy
    kvg.kvg_graft(s["store"].h, s["bid"], s["dst"].h, 0, -1, 0, kvg.KVG_GRAFT_SYNC)
    s["ocache"].graft(0, s["oblk"])
    mask = None
    for i, delta in enumerate([1, 4096, 100000]):
        seq = 1 + (i % 2)
        if i == 2:
            kvg.kvg_cache_release(s["dst"].h, 1)
            s["ocache"].release(1)
        kvg.kvg_graft(s["store"].h, s["bid"], s["dst"].h, seq, -1, delta,
                      kvg.KVG_GRAFT_VERIFY | kvg.KVG_GRAFT_SYNC)
        s["ocache"].graft(seq, s["oblk"], delta=delta)
        pool = pool_u16(s["dst"], w)
        if mask is None:
            mask = np.ones(pool[:, 0].shape, bool)
        pt, pf, ps = tables(s["dst"])
        oc = s["ocache"]
        assert np.array_equal(pt, oc.page_table) and np.array_equal(pf, oc.page_fill)
        assert np.array_equal(ps, oc.positions)
        # values, padding rows and untouched pages: bit-exact
        assert np.array_equal(pool[:, 1], oc.pool[:, 1])
        kg = _logical_k(pool, pt, w, seq, nb)
        k64 = np.stack([oracle.rope_rotate_rows(s["k"][l, :nb], delta, w.rope_theta, style)
                        for l in range(w.n_layers)])
        err = np.abs(oracle.bf16_to_f64(kg) - k64).max()
        assert err <= 2e-2, err
        check_rotation_rounding(oracle, kg, k64)  # finer than the tolerance
        # bytes outside every key row ever rotated (released pages keep theirs) equal the oracle's
        for t in range(nb):
            j, r = divmod(t, w.page_size)
            mask[:, pt[seq, j], :, r, :] = False
        assert np.array_equal(pool[:, 0][mask], oc.pool[:, 0][mask])


def test_relocated_decode_is_delta_invariant_within_tolerance(oracle):
    # keys re-based by delta and the query rotated by delta: the fp64 oracle is
    # delta-invariant; the GPU output stays within tolerance of it
    kvg = need_gpu()
    w = geometry("d128")
    nb = 512
    s = _build_both(kvg, oracle, w, nb, 0, seed=43, copies=3)
    q0 = syn.as_u16(syn.queries(w, w.n_layers, 1, 43))
    scale = 1 / math.sqrt(w.head_dim)
    ref = [oracle.gqa_decode(q0[l, 0], s["k"][l], s["v"][l], scale) for l in range(w.n_layers)]
    for seq, delta in enumerate([0, 1, 4096]):
        kvg.kvg_graft(s["store"].h, s["bid"], s["dst"].h, seq, -1, delta, kvg.KVG_GRAFT_SYNC)
        qd = np.stack([oracle.rope_rotate_rows_bf16(q0[l], delta, w.rope_theta, 0) for l in range(w.n_layers)])
        o = decode(kvg, s["dst"], w, [seq], qd)
        for l in range(w.n_layers):
            # the same query over the keys as the cache holds them (rotated,
            # rounded to bf16): only the kernel's own rounding remains
            kr = s["k"][l] if delta == 0 else oracle.rope_rotate_rows_bf16(s["k"][l], delta, w.rope_theta, 0)
            compare_decode(oracle, o[l, 0], oracle.gqa_decode(qd[l, 0], kr, s["v"][l], scale), what=f"reloc {delta}")
            # against the un-rotated fp64 reference: q and k also carry the
            # bf16 rounding of their rotation
            compare_decode(oracle, o[l, 0], ref[l], rel=REL_TOL_RELOCATED, floor=RNE_FLOOR_RELOCATED,
                           what=f"reloc-invariance {delta}")


# ------------------------------------------------------- integrity & errors

def test_verify_detects_a_flipped_byte(oracle):
    kvg = need_gpu()
    w = geometry("d128")
    s = _build_both(kvg, oracle, w, 300, 0, seed=51, copies=3)
    blob = bytearray(kvg.kvg_store_export(s["store"].h, s["bid"]))
    info = kvg.kvg_store_block_info(s["store"].h, s["bid"])
    npb = info.n_pages
    bad_page = (1 * 2 + 1) * npb + 2  # layer 1, V, page 2
    blob[info.pages_offset + bad_page * s["dims"].n_kv_heads * w.page_size * w.head_dim * 2 + 100] ^= 0x10
    with pytest.raises(kvg.KvgError) as e:
        kvg.kvg_store_import(s["store"].h, bytes(blob), kvg.KVG_GRAFT_VERIFY)
    assert e.value.status == kvg.KVG_ERR_DIGEST
    bid2 = kvg.kvg_store_import(s["store"].h, bytes(blob), 0)
    rep = kvg.kvg_graft_report()
    with pytest.raises(kvg.KvgError) as e:
        kvg.kvg_graft(s["store"].h, bid2, s["dst"].h, 0, -1, 0, kvg.KVG_GRAFT_VERIFY | kvg.KVG_GRAFT_SYNC,
                      report=rep)
    assert e.value.status == kvg.KVG_ERR_DIGEST
    assert rep.n_mismatch == 1 and rep.mismatch_pages[0] == bad_page and rep.seq == 0
    # asynchronous form: the mismatch surfaces at kvg_sync
    kvg.kvg_graft(s["store"].h, bid2, s["dst"].h, 1, -1, 0, kvg.KVG_GRAFT_VERIFY)
    rep2 = kvg.kvg_graft_report()
    with pytest.raises(kvg.KvgError) as e:
        kvg.kvg_sync(s["dst"].h, None, 10.0, rep2)
    assert e.value.status == kvg.KVG_ERR_DIGEST and rep2.mismatch_pages[0] == bad_page
    # the intact block verifies and imports cleanly
    good = kvg.kvg_store_export(s["store"].h, s["bid"])
    bid3 = kvg.kvg_store_import(s["store"].h, good, kvg.KVG_GRAFT_VERIFY)
    assert kvg.kvg_store_export(s["store"].h, bid3) == good
    kvg.kvg_sync(s["dst"].h)


@pytest.mark.parametrize("residency", [0, 1])
def test_failed_import_gives_back_its_store_space(oracle, residency):
    """A block whose digests do not verify is not added, and the store space
    it was copied into is free again: a store with room for exactly one block
    refuses the corrupted copy and then takes the intact one."""
    kvg = need_gpu()
    w = geometry("tiny")
    s = _build_both(kvg, oracle, w, 100, 0, seed=53)
    good = kvg.kvg_store_export(s["store"].h, s["bid"])
    bad = bytearray(good)
    info = kvg.kvg_store_block_info(s["store"].h, s["bid"])
    bad[info.pages_offset + 7] ^= 0x01
    small = kvg.Store(s["dims"], residency, len(good))
    for _ in range(3):
        with pytest.raises(kvg.KvgError) as e:
            kvg.kvg_store_import(small.h, bytes(bad), kvg.KVG_GRAFT_VERIFY)
        assert e.value.status == kvg.KVG_ERR_DIGEST
    bid = kvg.kvg_store_import(small.h, good, kvg.KVG_GRAFT_VERIFY)
    assert kvg.kvg_store_export(small.h, bid) == good
    with pytest.raises(kvg.KvgError) as e:
        kvg.kvg_store_import(small.h, good, 0)
    assert e.value.status == kvg.KVG_ERR_CAPACITY


@pytest.mark.parametrize("hkv,P", [(3, 7), (1, 33), (4, 64)], ids=["2688B_page", "4224B_page", "64KiB_page"])
def test_fused_verified_graft(oracle, hkv, P):
    """A verified own-position graft copies and hashes in one pass.  Pages of
    2,688 B (one short leaf), 4,224 B (a full and a short leaf) and 64 KiB: the
    restored cache equals the oracle's and the unverified copy's byte for byte;
    a flipped byte in a short leaf is reported on exactly its page, and the
    pass still restores the bytes it read."""
    kvg = need_gpu()
    w = syn.Workload("odd", 2, 2 * hkv, hkv, 64, P, 10000.0, 0x61 + P)
    nb = 5 * P + 3
    s = _build_both(kvg, oracle, w, nb, 0, seed=P, copies=3)
    rep = kvg.kvg_graft_report()
    kvg.kvg_graft(s["store"].h, s["bid"], s["dst"].h, 0, -1, 0, kvg.KVG_GRAFT_VERIFY | kvg.KVG_GRAFT_SYNC,
                  report=rep)
    assert rep.n_mismatch == 0 and rep.n_pages_checked == w.n_layers * 2 * s["oblk"].n_pages
    kvg.kvg_graft(s["store"].h, s["bid"], s["dst"].h, 1, -1, 0, kvg.KVG_GRAFT_SYNC)
    s["ocache"].graft(0, s["oblk"])
    s["ocache"].graft(1, s["oblk"])
    assert np.array_equal(pool_u16(s["dst"], w), s["ocache"].pool)
    pt, pf, ps = tables(s["dst"])
    assert np.array_equal(pt, s["ocache"].page_table) and np.array_equal(ps, s["ocache"].positions)
    # corrupt the last byte of the last leaf of (layer 1, K, page 4)
    blob = bytearray(kvg.kvg_store_export(s["store"].h, s["bid"]))
    info = kvg.kvg_store_block_info(s["store"].h, s["bid"])
    page_bytes = hkv * P * w.head_dim * 2
    bad_page = (1 * 2 + 0) * info.n_pages + 4
    at = info.pages_offset + bad_page * page_bytes + page_bytes - 1
    blob[at] ^= 0x01
    bid2 = kvg.kvg_store_import(s["store"].h, bytes(blob), 0)
    rep2 = kvg.kvg_graft_report()
    with pytest.raises(kvg.KvgError) as e:
        kvg.kvg_graft(s["store"].h, bid2, s["dst"].h, 2, -1, 0, kvg.KVG_GRAFT_VERIFY | kvg.KVG_GRAFT_SYNC,
                      report=rep2)
    assert e.value.status == kvg.KVG_ERR_DIGEST
    assert rep2.n_mismatch == 1 and rep2.mismatch_pages[0] == bad_page and rep2.seq == 2
    pool = pool_u16(s["dst"], w)
    pt, _, _ = tables(s["dst"])
    pid = int(pt[2, 4])
    got = pool[1, 0, pid].tobytes()
    want = bytes(blob[at - page_bytes + 1: at + 1])
    assert got == want


@pytest.mark.parametrize("geo,nb,bad", [("tiny", 250, (3, 15)), ("d128", 1000, (4, 0)), ("d128", 1000, (5, 9)),
                                        ("d128", 2583, (5, 40)), ("d128", 2583, (0, 39)), ("d128", 8320, (3, 129)),
                                        ("d128", 8320, (2, 127))])
def test_host_store_verified_graft_reports_the_bad_page(oracle, geo, nb, bad):
    """A verified graft from a pinned-host store copies page-range chunks and
    hashes each chunk's restored pages on a second stream: a flipped byte in
    page (plane, j) is reported as that block page, whichever chunk holds it
    (41 and 130 pages: after the equal chunks, a chunk of three pages and
    one of one), and an intact block grafts clean."""
    kvg = need_gpu()
    w = geometry(geo)
    s = _build_both(kvg, oracle, w, nb, 0, seed=61, copies=3)
    host = kvg.Store(s["dims"], kvg.KVG_RESIDENCY_PINNED_HOST, 1 << 30)
    blob = bytearray(kvg.kvg_store_export(s["store"].h, s["bid"]))
    hid = kvg.kvg_store_import(host.h, bytes(blob), kvg.KVG_GRAFT_VERIFY)
    rep = kvg.kvg_graft_report()
    kvg.kvg_graft(host.h, hid, s["dst"].h, 0, -1, 0, kvg.KVG_GRAFT_VERIFY | kvg.KVG_GRAFT_SYNC, report=rep)
    assert rep.n_mismatch == 0
    info = kvg.kvg_store_block_info(s["store"].h, s["bid"])
    page_bytes = w.n_kv_heads * w.page_size * w.head_dim * 2
    plane, j = bad
    bad_page = plane * info.n_pages + j
    blob[info.pages_offset + bad_page * page_bytes + 7] ^= 0x40
    hid2 = kvg.kvg_store_import(host.h, bytes(blob), 0)
    rep2 = kvg.kvg_graft_report()
    with pytest.raises(kvg.KvgError) as e:
        kvg.kvg_graft(host.h, hid2, s["dst"].h, 1, -1, 0, kvg.KVG_GRAFT_VERIFY | kvg.KVG_GRAFT_SYNC, report=rep2)
    assert e.value.status == kvg.KVG_ERR_DIGEST
    assert rep2.n_mismatch == 1 and rep2.mismatch_pages[0] == bad_page
    # the intact graft restored the oracle's bytes
    s["ocache"].graft(0, s["oblk"])
    pool = pool_u16(s["dst"], w)
    pt, _, _ = tables(s["dst"])
    for jj in range(info.n_pages):
        pid = int(pt[0, jj])
        assert np.array_equal(pool[:, :, pid], s["ocache"].pool[:, :, int(s["ocache"].page_table[0, jj])])
    kvg.kvg_sync(s["dst"].h)


@pytest.mark.parametrize("geo,residency", [("tiny", 0), ("d128", 0), ("d128", 1)])
def test_graft_batch_equals_sequential_grafts(oracle, geo, residency):
    """kvg_graft_batch: blocks of several lengths (ragged ones too) into
    sequences that repeat, stitched page-aligned in call order, in one launch
    (from an HBM store, or from a pinned-host store on a capped grid): pool
    bytes, page tables, fills and positions equal the oracle's sequential
    grafts; with verification every graft is checked; a batch that does not
    fit changes nothing."""
    kvg = need_gpu()
    w = geometry(geo)
    P = w.page_size
    dims = dims_for(kvg, w)
    od = oracle_dims(oracle, w)
    lens = [3 * P, 2 * P + 5, P - 3, 4 * P + 1, 7]
    src = kvg.Cache(dims, 64, 1, 8 * P)
    store = kvg.Store(dims, residency, HBM_CAP)
    bids, oblks = [], []
    for i, n in enumerate(lens):
        k, v = _kv(w, n, 160 + i)
        append(kvg, src, 0, k, v, syn.positions(0, n))
        bids.append(kvg.kvg_deposit(store.h, src.h, 0, 0, n))
        kvg.kvg_cache_release(src.h, 0)
        oblks.append(oracle.block_from_kv(od, k, v, syn.positions(0, n)))
    order = [(0, 2), (1, 0), (0, 1), (4, 2), (3, 1), (4, 0), (2, 2)]  # (block, seq)
    n_pages = 64
    max_slots = 16 * P
    c = kvg.Cache(dims, n_pages, 3, max_slots)
    fill_canary(c)
    kvg.kvg_cache_set_free_order(c.h, syn.permutation(n_pages, 170))
    oc = oracle.OracleCache(od, n_pages, 3, max_slots, fill=CANARY)
    oc.set_free_order(syn.permutation(n_pages, 170))
    # a short sequence first, so the first batched graft lands after a ragged page
    k0, v0 = _kv(w, 3, 171)
    append(kvg, c, 1, k0, v0, syn.positions(0, 3))
    oc.append(1, k0, v0, syn.positions(0, 3))
    rep = kvg.kvg_graft_report()
    kvg.kvg_graft_batch(store.h, [bids[b] for b, _ in order], c.h, [q for _, q in order],
                        kvg.KVG_GRAFT_VERIFY | kvg.KVG_GRAFT_SYNC, report=rep)
    assert rep.n_mismatch == 0
    assert rep.n_pages_checked == w.n_layers * 2 * sum(oblks[b].n_pages for b, _ in order)
    for b, q in order:
        oc.graft(q, oblks[b])
    assert np.array_equal(pool_u16(c, w), oc.pool)
    pt, pf, ps = tables(c)
    assert np.array_equal(pt, oc.page_table) and np.array_equal(pf, oc.page_fill)
    assert np.array_equal(ps, oc.positions)
    for q in range(3):
        assert kvg.kvg_cache_seq_info(c.h, q)[0] == oc.n_slots[q]
    # too many pages for what is left: refused whole
    before = pool_u16(c, w).copy()
    with pytest.raises(kvg.KvgError) as e:
        kvg.kvg_graft_batch(store.h, [bids[3]] * 12, c.h, [0, 1, 2] * 4)
    assert e.value.status == kvg.KVG_ERR_CAPACITY
    with pytest.raises(kvg.KvgError) as e:
        kvg.kvg_graft_batch(store.h, [bids[0], 999], c.h, [0, 1])
    assert e.value.status == kvg.KVG_ERR_NOT_FOUND
    assert np.array_equal(pool_u16(c, w), before)
    assert all(kvg.kvg_cache_seq_info(c.h, q)[0] == oc.n_slots[q] for q in range(3))
    kvg.kvg_sync(c.h)


@pytest.mark.parametrize("geo,style,residency", [("d128", 0, 0), ("d128", 1, 0), ("d256", 0, 0), ("tiny", 0, 0),
                                                 ("d128", 0, 1)])
def test_relocate_to_consecutive_composition(oracle, geo, style, residency):
    """Sequential composition at the KV level (Sec. 4.8), re-basing blocks
    (Sec. 4.2): four blocks deposited at their own positions [0, N_b) go into
    one sequence, each at the next page boundary; block 1 at its own
    positions, block b > 1 re-based by delta = the tokens already present, so
    the position tags run 0 .. sum(N) - 1 without a gap.  One
    kvg_graft_batch call with per-graft deltas and four kvg_graft calls give
    the same pool bytes; page tables, fills and tags equal the oracle's;
    values and padding are bit-exact, re-based keys within 2e-2 of the fp64
    rotation; the decode over the composed sequence passes the decode gate
    against the oracle's cache built with the same deltas; verification of
    every graft passes (re-based ones hash their stored pages).  From an HBM
    store, and from a pinned-host store (read over the host link)."""
    kvg = need_gpu()
    w = geometry(geo)
    P = w.page_size
    dims = dims_for(kvg, w, style)
    od = oracle_dims(oracle, w, style)
    lens = [3 * P + 7, 2 * P, P - 5, 2 * P + 1]
    src = kvg.Cache(dims, 32, 1, 8 * P)
    store = kvg.Store(dims, residency, HBM_CAP)
    bids, oblks, rows = [], [], []
    for i, n in enumerate(lens):
        k, v = _kv(w, n, 310 + i)
        append(kvg, src, 0, k, v, syn.positions(0, n))
        bids.append(kvg.kvg_deposit(store.h, src.h, 0, 0, n))
        kvg.kvg_cache_release(src.h, 0)
        oblks.append(oracle.block_from_kv(od, k, v, syn.positions(0, n)))
        rows.append((k, v))
    deltas = [int(sum(lens[:i])) for i in range(len(lens))]
    n_pages, max_slots = 48, 16 * P
    caches = []
    for _ in range(2):
        c = kvg.Cache(dims, n_pages, 2, max_slots)
        fill_canary(c)
        kvg.kvg_cache_set_free_order(c.h, syn.permutation(n_pages, 320))
        caches.append(c)
    flags = kvg.KVG_GRAFT_VERIFY | kvg.KVG_GRAFT_SYNC
    rep = kvg.kvg_graft_report()
    kvg.kvg_graft_batch(store.h, bids, caches[0].h, [1] * 4, flags, report=rep, deltas=deltas)
    assert rep.n_mismatch == 0 and rep.n_pages_checked == w.n_layers * 2 * sum(b.n_pages for b in oblks)
    for b, d in zip(bids, deltas):
        kvg.kvg_graft(store.h, b, caches[1].h, 1, -1, d, flags)
    pool = pool_u16(caches[0], w)
    assert np.array_equal(pool, pool_u16(caches[1], w))
    oc = oracle.OracleCache(od, n_pages, 2, max_slots, fill=CANARY)
    oc.set_free_order(syn.permutation(n_pages, 320))
    for blk, d in zip(oblks, deltas):
        oc.graft(1, blk, delta=d)
    pt, pf, ps = tables(caches[0])
    assert np.array_equal(pt, oc.page_table) and np.array_equal(pf, oc.page_fill)
    assert np.array_equal(ps, oc.positions)
    # the position tags of the valid rows run 0 .. sum(N) - 1
    valid = np.concatenate([np.arange(j * P, j * P + pf[1, j]) for j in range(int((pt[1] >= 0).sum()))])
    assert np.array_equal(ps[1, valid], np.arange(sum(lens)))
    # values, padding rows and untouched pages bit-exact; re-based keys
    # within 2e-2 of the fp64 rotation
    assert np.array_equal(pool[:, 1], oc.pool[:, 1])
    j0 = 0
    mask = np.ones(pool[:, 0].shape, bool)
    for (k, _), n, d in zip(rows, lens, deltas):
        kg = np.stack([np.stack([pool[l, 0, pt[1, j0 + t // P], :, t % P] for t in range(n)]) for l in range(w.n_layers)])
        if d == 0:
            assert np.array_equal(kg, k)
        else:
            k64 = np.stack([oracle.rope_rotate_rows(k[l], d, w.rope_theta, style) for l in range(w.n_layers)])
            assert np.abs(oracle.bf16_to_f64(kg) - k64).max() <= 2e-2
            check_rotation_rounding(oracle, kg, k64)
        for t in range(n):
            mask[:, pt[1, j0 + t // P], :, t % P] = False
        j0 += -(-n // P)
    assert np.array_equal(pool[:, 0][mask], oc.pool[:, 0][mask])
    # decode over the composed sequence against the oracle's cache
    q = syn.as_u16(syn.queries(w, w.n_layers, 1, 330))
    scale = 1 / math.sqrt(w.head_dim)
    o = decode(kvg, caches[0], w, [1], q)
    assert np.array_equal(o, decode(kvg, caches[1], w, [1], q))
    for l in range(w.n_layers):
        compare_decode(oracle, o[l, 0], oc.decode(1, l, q[l, 0], scale), what=f"consecutive {geo} layer {l}")
    # a delta that pushes a tag out of [0, 2^31): refused whole
    before = pool_u16(caches[0], w).copy()
    with pytest.raises(kvg.KvgError) as e:
        kvg.kvg_graft_batch(store.h, bids[:2], caches[0].h, [0, 0], deltas=[0, 2 ** 31 - lens[1] + 1])
    assert e.value.status == kvg.KVG_ERR_POSITION
    assert np.array_equal(pool_u16(caches[0], w), before)
    assert kvg.kvg_cache_seq_info(caches[0].h, 0)[0] == 0
    for c in caches:
        kvg.kvg_sync(c.h)


def test_corrupt_page_table_entries_are_reported_not_followed(oracle):
    """A page id outside the pool written into the device page table (through
    the exported view) is never dereferenced: decode records
    KVG_ERR_DEVICE_CHECK and skips that page; verification reports that page
    as a digest mismatch."""
    kvg = need_gpu()
    w = geometry("d128")
    s = _build_both(kvg, oracle, w, 300, 0, seed=181)
    kvg.kvg_graft(s["store"].h, s["bid"], s["dst"].h, 0, -1, 0, kvg.KVG_GRAFT_SYNC)
    v = s["dst"].view
    pt = dev_view(v.page_table, v.max_seqs * v.max_pages * 4, torch.int32).view(v.max_seqs, v.max_pages)
    good = int(pt[0, 2].item())
    pt[0, 2] = s["n_pages"] + 7
    torch.cuda.synchronize()
    q = syn.as_u16(syn.queries(w, w.n_layers, 1, 182))
    decode(kvg, s["dst"], w, [0], q)
    with pytest.raises(kvg.KvgError) as e:
        kvg.kvg_sync(s["dst"].h)
    assert e.value.status == kvg.KVG_ERR_DEVICE_CHECK
    rep = kvg.kvg_graft_report()
    with pytest.raises(kvg.KvgError) as e:
        kvg.kvg_verify(s["store"].h, s["bid"], s["dst"].h, 0, 0, kvg.KVG_GRAFT_SYNC, report=rep)
    assert e.value.status == kvg.KVG_ERR_DIGEST
    npb = (300 + w.page_size - 1) // w.page_size
    assert sorted(rep.mismatch_pages[:rep.n_mismatch]) == [pl * npb + 2 for pl in range(w.n_layers * 2)]
    # restored, everything is clean again
    pt[0, 2] = good
    torch.cuda.synchronize()
    kvg.kvg_verify(s["store"].h, s["bid"], s["dst"].h, 0, 0, kvg.KVG_GRAFT_SYNC)
    kvg.kvg_sync(s["dst"].h)


def test_host_checks_reject_bad_calls(oracle):
    kvg = need_gpu()
    w = geometry("tiny")
    s = _build_both(kvg, oracle, w, 40, 0, seed=61)
    st, dst = s["store"].h, s["dst"].h
    E = kvg.KvgError
    with pytest.raises(E) as e:
        kvg.kvg_graft(st, 99, dst, 0)
    assert e.value.status == kvg.KVG_ERR_NOT_FOUND
    with pytest.raises(E) as e:
        kvg.kvg_graft(st, s["bid"], dst, 0, 16)  # not the next page boundary (0)
    assert e.value.status == kvg.KVG_ERR_ARG
    with pytest.raises(E) as e:
        kvg.kvg_graft(st, s["bid"], dst, 0, -1, -5)  # positions 0.. + delta < 0
    assert e.value.status == kvg.KVG_ERR_POSITION
    with pytest.raises(E) as e:
        kvg.kvg_graft(st, s["bid"], dst, 0, -1, 2**31 - 20)
    assert e.value.status == kvg.KVG_ERR_POSITION
    assert kvg.kvg_cache_seq_info(dst, 0) == (0, 0)  # failed calls changed nothing
    small = kvg.Cache(s["dims"], 2, 1, 64)
    with pytest.raises(E) as e:
        kvg.kvg_graft(st, s["bid"], small.h, 0)  # 3 pages needed, 2 exist
    assert e.value.status == kvg.KVG_ERR_CAPACITY
    with pytest.raises(E) as e:
        kvg.kvg_deposit(st, s["src"].h, 0, 8, 10)  # slot0 not page-aligned
    assert e.value.status == kvg.KVG_ERR_ARG
    q = torch.zeros((w.n_layers, 1, 3, w.head_dim), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(E) as e:
        kvg.kvg_decode_attention(dst, -1, [0], q.data_ptr(), 3, q.data_ptr(), 0.1)
    assert e.value.status == kvg.KVG_ERR_ARG
    with pytest.raises(E) as e:
        kvg.kvg_cache_set_free_order(s["src"].h, list(range(s["n_pages"])))  # pages in use
    assert e.value.status == kvg.KVG_ERR_ARG


@pytest.mark.parametrize("geo", ["tiny", "g4", "d256"])
def test_append_sizes_and_offsets(oracle, geo):
    """Appends of 1, P-1, P, P+1 and 3P+5 rows at ragged slot offsets (rows
    shorter than a page go through the warp-per-row kernel, longer ones
    through the tensor-copy kernel), and one long append into a second
    sequence: pool bytes, page tables, fills and positions equal the
    oracle's."""
    kvg = need_gpu()
    w = geometry(geo)
    P = w.page_size
    sizes = [1, P - 1, P, P + 1, 3 * P + 5, 2]
    total = sum(sizes)
    k, v = _kv(w, total + 5 * P + 3, 71)
    max_slots = _slots(w, total + 5 * P + 3)
    n_pages = 2 * (max_slots // P) + 4
    dims = dims_for(kvg, w)
    c = kvg.Cache(dims, n_pages, 2, max_slots)
    fill_canary(c)
    kvg.kvg_cache_set_free_order(c.h, syn.permutation(n_pages, 72))
    oc = oracle.OracleCache(oracle_dims(oracle, w), n_pages, 2, max_slots, fill=CANARY)
    oc.set_free_order(syn.permutation(n_pages, 72))
    t = 0
    for n in sizes:
        pos = syn.positions(t, n)
        append(kvg, c, 0, k[:, t:t + n], v[:, t:t + n], pos)
        oc.append(0, k[:, t:t + n], v[:, t:t + n], pos)
        t += n
    n = 5 * P + 3
    pos = syn.positions(1000, n)
    append(kvg, c, 1, k[:, t:t + n], v[:, t:t + n], pos)
    oc.append(1, k[:, t:t + n], v[:, t:t + n], pos)
    assert np.array_equal(pool_u16(c, w), oc.pool)
    pt, pf, ps = tables(c)
    assert np.array_equal(pt, oc.page_table) and np.array_equal(pf, oc.page_fill)
    assert np.array_equal(ps, oc.positions)
    kvg.kvg_sync(c.h)


def test_append_batch_matches_oracle(oracle):
    kvg = need_gpu()
    w = geometry("d128")
    dims = dims_for(kvg, w)
    lens = [63, 64, 1, 130]  # one row lands in a fresh page, one mid-page
    max_slots = 256
    n_pages = 20
    cache = kvg.Cache(dims, n_pages, 5, max_slots)
    fill_canary(cache)
    od = oracle_dims(oracle, w)
    oc = oracle.OracleCache(od, n_pages, 5, max_slots, fill=CANARY)
    for i, n in enumerate(lens):
        k, v = _kv(w, n, 90 + i)
        append(kvg, cache, i, k, v, syn.positions(0, n))
        oc.append(i, k, v, syn.positions(0, n))
    seqs = [3, 0, 1, 2]
    for step in range(3):
        k, v = _kv(w, len(seqs), 95 + step)  # [L][B][Hkv][D]: one row per sequence
        pos = np.array([1000 + 10 * step + b for b in range(len(seqs))], np.int32)
        kd, vd, pd = to_dev(k), to_dev(v), to_dev(pos)
        kvg.kvg_cache_append_batch(cache.h, seqs, kd.data_ptr(), vd.data_ptr(), pd.data_ptr())
        torch.cuda.synchronize()
        oc.append_batch(seqs, k, v, pos)
    assert np.array_equal(pool_u16(cache, w), oc.pool)
    pt, pf, ps = tables(cache)
    assert np.array_equal(pt, oc.page_table) and np.array_equal(pf, oc.page_fill)
    assert np.array_equal(ps, oc.positions)
    with pytest.raises(kvg.KvgError) as e:
        kvg.kvg_cache_append_batch(cache.h, [0, 0], kd.data_ptr(), vd.data_ptr(), pd.data_ptr())
    assert e.value.status == kvg.KVG_ERR_ARG


def test_sync_times_out_while_the_stream_is_busy_then_succeeds():
    # host-side failure detection: kvg_sync gives up after its limit and
    # reports KVG_ERR_TIMEOUT without touching the work in flight (the busy
    # stream is a bounded spin of ~50 ms queued ahead of the call)
    kvg = need_gpu()
    w = geometry("tiny")
    cache = kvg.Cache(dims_for(kvg, w), 4, 1, 64)
    s = torch.cuda.current_stream()
    torch.cuda._sleep(100_000_000)
    with pytest.raises(kvg.KvgError) as e:
        kvg.kvg_sync(cache.h, s, 1e-3)
    assert e.value.status == kvg.KVG_ERR_TIMEOUT
    kvg.kvg_sync(cache.h, s, 60.0)


@pytest.mark.parametrize("residency", [0, 1])
def test_prefetch_then_graft_is_bit_exact(oracle, residency):
    """kvg_store_prefetch only reads: a pinned-host block prefetched on a
    side stream, then grafted on another, restores the oracle's bytes; on an
    HBM store the call does nothing; an unknown block is KVG_ERR_NOT_FOUND."""
    kvg = need_gpu()
    w = geometry("d128")
    s = _build_both(kvg, oracle, w, 300, 0, residency=residency, seed=131)
    side, main = torch.cuda.Stream(), torch.cuda.Stream()
    ev = torch.cuda.Event()
    kvg.kvg_store_prefetch(s["store"].h, s["bid"], side)
    ev.record(side)
    main.wait_event(ev)
    kvg.kvg_graft(s["store"].h, s["bid"], s["dst"].h, 0, -1, 0, kvg.KVG_GRAFT_VERIFY, main)
    main.synchronize()
    kvg.kvg_sync(s["dst"].h, main)
    s["ocache"].graft(0, s["oblk"])
    assert np.array_equal(pool_u16(s["dst"], w), s["ocache"].pool)
    assert kvg.kvg_store_export(s["store"].h, s["bid"]) == s["oblk"].serialize()
    with pytest.raises(kvg.KvgError) as e:
        kvg.kvg_store_prefetch(s["store"].h, s["bid"] + 1, side)
    assert e.value.status == kvg.KVG_ERR_NOT_FOUND
    # a block held in a cache's own pool needs no translations: nothing to do
    pc = kvg.Cache(s["dims"], 64, 1, 1024)
    append(kvg, pc, 0, s["k"][:, :100], s["v"][:, :100], syn.positions(0, 100))
    pool = kvg.PoolStore(pc, 1 << 26)
    pbid = kvg.kvg_deposit(pool.h, pc.h, 0, 0, 100)
    kvg.kvg_store_prefetch(pool.h, pbid, side)
    side.synchronize()


def test_block_files_round_trip_and_are_verified(oracle, tmp_path):
    # a block is a plain file: saved, copied, loaded elsewhere with its digests
    # checked (Sec. 4.4, Sec. 4.11)
    kvg = need_gpu()
    w = geometry("d128")
    s = _build_both(kvg, oracle, w, 300, 0, seed=121)
    path = str(tmp_path / "block.kvg")
    kvg.kvg_store_save(s["store"].h, s["bid"], path)
    data = open(path, "rb").read()
    assert data == s["oblk"].serialize()
    host = kvg.Store(s["dims"], kvg.KVG_RESIDENCY_PINNED_HOST, 1 << 30)
    bid = kvg.kvg_store_load(host.h, path, kvg.KVG_GRAFT_VERIFY)
    assert kvg.kvg_store_export(host.h, bid) == data
    kvg.kvg_graft(host.h, bid, s["dst"].h, 0, -1, 0, kvg.KVG_GRAFT_VERIFY | kvg.KVG_GRAFT_SYNC)
    s["ocache"].graft(0, s["oblk"])
    assert np.array_equal(pool_u16(s["dst"], w), s["ocache"].pool)
    bad = bytearray(data)
    bad[-5] ^= 0x01
    open(path, "wb").write(bytes(bad))
    with pytest.raises(kvg.KvgError) as e:
        kvg.kvg_store_load(host.h, path, kvg.KVG_GRAFT_VERIFY)
    assert e.value.status == kvg.KVG_ERR_DIGEST
    open(path, "wb").write(data[:1000])
    with pytest.raises(kvg.KvgError) as e:
        kvg.kvg_store_load(host.h, path, 0)
    assert e.value.status == kvg.KVG_ERR_FORMAT


@pytest.mark.parametrize("residency", [0, 1])
def test_block_file_loads_in_chunks(oracle, tmp_path, residency):
    """A block file of several 16 MiB read chunks (51 MB: 12,800 tokens of
    the d256 geometry) loads byte-exact into an HBM or pinned-host store with
    every digest checked; a flipped byte in a later chunk is caught, a
    truncated file is refused, and neither is added."""
    kvg = need_gpu()
    w = geometry("d256")
    nb = 200 * w.page_size
    s = _build_both(kvg, oracle, w, nb, 0, seed=131)
    path = str(tmp_path / "big.kvg")
    kvg.kvg_store_save(s["store"].h, s["bid"], path)
    data = open(path, "rb").read()
    assert data == s["oblk"].serialize() and len(data) > 3 * (16 << 20)
    st = kvg.Store(s["dims"], residency, 1 << 30)
    bid = kvg.kvg_store_load(st.h, path, kvg.KVG_GRAFT_VERIFY)
    assert kvg.kvg_store_export(st.h, bid) == data
    assert bytes(kvg.kvg_store_block_info(st.h, bid).block_digest) == s["oblk"].block_digest
    kvg.kvg_graft(st.h, bid, s["dst"].h, 0, -1, 0, kvg.KVG_GRAFT_VERIFY | kvg.KVG_GRAFT_SYNC)
    s["ocache"].graft(0, s["oblk"])
    assert np.array_equal(pool_u16(s["dst"], w), s["ocache"].pool)
    bad = bytearray(data)
    bad[(40 << 20) + 12345] ^= 0x40  # inside the third chunk
    open(path, "wb").write(bytes(bad))
    with pytest.raises(kvg.KvgError) as e:
        kvg.kvg_store_load(st.h, path, kvg.KVG_GRAFT_VERIFY)
    assert e.value.status == kvg.KVG_ERR_DIGEST
    open(path, "wb").write(data[:(20 << 20)])
    with pytest.raises(kvg.KvgError) as e:
        kvg.kvg_store_load(st.h, path, kvg.KVG_GRAFT_VERIFY)
    assert e.value.status == kvg.KVG_ERR_FORMAT
    # the store holds the one good block; a second good load still fits and matches
    open(path, "wb").write(data)
    bid2 = kvg.kvg_store_load(st.h, path, 0)
    assert bid2 == bid + 1 and kvg.kvg_store_export(st.h, bid2) == data
    kvg.kvg_sync(s["dst"].h)


@pytest.mark.parametrize("residency", [0, 1])
def test_consecutive_deposits_serialize_exactly(oracle, residency):
    """Deposits of different lengths into one store, back to back (a
    pinned-host store reuses its HBM staging buffer): each block's bytes,
    including the zero gaps after its position tags and page digests, equal
    the oracle's serialization, and its block digest is written even though
    the call does not wait for it."""
    kvg = need_gpu()
    w = geometry("d128")
    lens = [1000, 37, 333, 64]
    k, v = _kv(w, max(lens), 141)
    dims = dims_for(kvg, w)
    od = oracle_dims(oracle, w)
    src = kvg.Cache(dims, 64, 1, _slots(w, max(lens)))
    append(kvg, src, 0, k, v, syn.positions(0, max(lens)))
    store = kvg.Store(dims, residency, HBM_CAP)
    bids = [kvg.kvg_deposit(store.h, src.h, 0, 0, n) for n in lens]
    for n, bid in zip(lens, bids):
        oblk = oracle.block_from_kv(od, np.ascontiguousarray(k[:, :n]), np.ascontiguousarray(v[:, :n]),
                                    syn.positions(0, n))
        assert kvg.kvg_store_export(store.h, bid) == oblk.serialize()
        assert bytes(kvg.kvg_store_block_info(store.h, bid).block_digest) == oblk.block_digest


def test_deposit_then_verified_import_on_other_streams(oracle):
    """A deposit returns before its page hashing runs; a verified import
    into the same store, issued at once on another stream, and a second
    deposit on a third stream still see their own leaf digests: all three
    blocks equal the oracle's and the import verifies."""
    kvg = need_gpu()
    w = geometry("d256")
    n1, n2 = 125 * w.page_size, 40 * w.page_size + 9
    k, v = _kv(w, n1, 151)
    dims = dims_for(kvg, w)
    od = oracle_dims(oracle, w)
    src = kvg.Cache(dims, 400, 1, _slots(w, n1))
    append(kvg, src, 0, k, v, syn.positions(0, n1))
    other = kvg.Store(dims, 0, HBM_CAP)
    good = kvg.kvg_store_export(other.h, kvg.kvg_deposit(other.h, src.h, 0, 0, n2))
    store = kvg.Store(dims, 0, HBM_CAP)
    sa, sb = torch.cuda.Stream(), torch.cuda.Stream()
    torch.cuda.synchronize()
    b1 = kvg.kvg_deposit(store.h, src.h, 0, 0, n1, sa)
    b2 = kvg.kvg_store_import(store.h, good, kvg.KVG_GRAFT_VERIFY)
    b3 = kvg.kvg_deposit(store.h, src.h, 0, 0, n2, sb)
    torch.cuda.synchronize()
    o1 = oracle.block_from_kv(od, k, v, syn.positions(0, n1)).serialize()
    o2 = oracle.block_from_kv(od, np.ascontiguousarray(k[:, :n2]), np.ascontiguousarray(v[:, :n2]),
                              syn.positions(0, n2)).serialize()
    assert good == o2
    assert kvg.kvg_store_export(store.h, b1) == o1
    assert kvg.kvg_store_export(store.h, b2) == o2
    assert kvg.kvg_store_export(store.h, b3) == o2


def test_pool_store_zero_copy_graft(oracle):
    # blocks living in the cache's own pool: a graft writes only the page
    # table (full pages shared), a ragged last page is copied, two sequences
    # share the block's pages while their appends diverge
    kvg = need_gpu()
    w = geometry("d128")
    nb, nf = 333, 100
    k, v = _kv(w, nb + nf, 131)
    P = w.page_size
    max_slots = (-(-(nb + nf) // P) + 2) * P
    n_pages = 40
    dims = dims_for(kvg, w)
    perm = syn.permutation(n_pages, 133)
    cache = kvg.Cache(dims, n_pages, 4, max_slots)
    fill_canary(cache)
    kvg.kvg_cache_set_free_order(cache.h, perm)
    od = oracle_dims(oracle, w)
    oc = oracle.OracleCache(od, n_pages, 4, max_slots, fill=CANARY)
    oc.set_free_order(perm)
    append(kvg, cache, 0, k[:, :nb], v[:, :nb], syn.positions(0, nb))
    oc.append(0, k[:, :nb], v[:, :nb], syn.positions(0, nb))
    store = kvg.PoolStore(cache, 64 << 20)
    bid = kvg.kvg_deposit(store.h, cache.h, 0, 0, nb)
    opb = oc.pin_block(0, 0, nb)
    assert kvg.kvg_store_export(store.h, bid) == opb.block.serialize()
    kvg.kvg_cache_release(cache.h, 0)
    oc.release(0)
    for seq in (1, 2):
        kvg.kvg_graft(store.h, bid, cache.h, seq, -1, 0, kvg.KVG_GRAFT_VERIFY | kvg.KVG_GRAFT_SYNC)
        oc.graft_pinned(seq, opb)
    kvg.kvg_verify(store.h, bid, cache.h, 1, 0, kvg.KVG_GRAFT_SYNC)  # before appends fill the last page
    append(kvg, cache, 1, k[:, nb:], v[:, nb:], syn.positions(nb, nf))
    oc.append(1, k[:, nb:], v[:, nb:], syn.positions(nb, nf))
    k2, v2 = _kv(w, 50, 132)
    append(kvg, cache, 2, k2, v2, syn.positions(nb, 50))
    oc.append(2, k2, v2, syn.positions(nb, 50))
    assert np.array_equal(pool_u16(cache, w), oc.pool)
    pt, pf, ps = tables(cache)
    assert np.array_equal(pt, oc.page_table) and np.array_equal(pf, oc.page_fill)
    assert np.array_equal(ps, oc.positions)
    full = nb // P
    assert list(pt[1, :full]) == list(pt[2, :full]) == opb.pids[:full]  # shared, not copied
    assert pt[1, full] != pt[2, full] != opb.pids[full]                 # ragged page copied per sequence
    # attention over the aliased rows equals attention over the same rows written fresh
    q = syn.as_u16(syn.queries(w, w.n_layers, 1, 134))
    fresh = kvg.Cache(dims, n_pages, 1, max_slots)
    append(kvg, fresh, 0, k, v, syn.positions(0, nb + nf))
    assert _sha(decode(kvg, cache, w, [1], q)) == _sha(decode(kvg, fresh, w, [0], q))
    # releases keep the block's pages; a relocating graft needs a copying store
    kvg.kvg_cache_release(cache.h, 1)
    kvg.kvg_cache_release(cache.h, 2)
    oc.release(1)
    oc.release(2)
    # (through kvg_graft_chunked: a pool-resident block grafts in one piece, one event)
    evs = [torch.cuda.Event() for _ in range(3)]
    for e in evs:
        e.record()
    ends = kvg.kvg_graft_chunked(store.h, bid, cache.h, 3, [e.cuda_event for e in evs],
                                 flags=kvg.KVG_GRAFT_VERIFY | kvg.KVG_GRAFT_SYNC)
    assert ends == [nb] and evs[0].query()
    oc.graft_pinned(3, opb)
    pt, pf, ps = tables(cache)
    assert np.array_equal(pt, oc.page_table) and np.array_equal(pool_u16(cache, w), oc.pool)
    with pytest.raises(kvg.KvgError) as e:
        kvg.kvg_graft(store.h, bid, cache.h, 0, -1, 4096)
    assert e.value.status == kvg.KVG_ERR_ARG
    # a flipped byte in a shared page is caught by verification of the sequence
    v_ = cache.view
    off = ((1 * 2 + 0) * v_.n_pages + opb.pids[2]) * w.page_bytes + 10
    page = dev_view(v_.pool + off, 16)
    page[0] ^= 1
    torch.cuda.synchronize()
    with pytest.raises(kvg.KvgError) as e:
        kvg.kvg_verify(store.h, bid, cache.h, 3, 0, kvg.KVG_GRAFT_SYNC)
    assert e.value.status == kvg.KVG_ERR_DIGEST
    store.close()
    fresh.close()
    cache.close()


def test_launch_chunking_limits(oracle):
    # > 1,024 pages per graft / deposit / append (several launches each) and
    # > 256 decode rows per call (several batch chunks): same bytes, same
    # attention as the oracle
    kvg = need_gpu()
    w = syn.Workload("p8", 1, 2, 1, 64, 8, 10000.0, 0x61)
    n = 9000  # 1,125 pages of 8 rows
    k, v = _kv(w, n, 141)
    P = w.page_size
    n_pages = 2 * (-(-n // P)) + 4
    dims = dims_for(kvg, w)
    src = kvg.Cache(dims, n_pages, 2, n + 2 * P)
    append(kvg, src, 0, k, v, syn.positions(0, n))
    store = kvg.Store(dims, kvg.KVG_RESIDENCY_HBM, 1 << 30)
    bid = kvg.kvg_deposit(store.h, src.h, 0, 0, n)
    od = oracle_dims(oracle, w)
    oblk = oracle.block_from_kv(od, k, v, syn.positions(0, n))
    assert kvg.kvg_store_export(store.h, bid) == oblk.serialize()
    dst = kvg.Cache(dims, n_pages, 2, n + 2 * P)
    fill_canary(dst)
    oc = oracle.OracleCache(od, n_pages, 2, n + 2 * P, fill=CANARY)
    kvg.kvg_graft(store.h, bid, dst.h, 0, -1, 0, kvg.KVG_GRAFT_VERIFY | kvg.KVG_GRAFT_SYNC)
    oc.graft(0, oblk)
    kvg.kvg_graft(store.h, bid, dst.h, 1, -1, 77, kvg.KVG_GRAFT_SYNC)
    oc.graft(1, oblk, delta=77)
    pool = pool_u16(dst, w)
    pt, pf, ps = tables(dst)
    assert np.array_equal(pt, oc.page_table) and np.array_equal(pf, oc.page_fill)
    assert np.array_equal(ps, oc.positions)
    assert np.array_equal(pool[:, 1], oc.pool[:, 1])
    assert np.array_equal(pool[:, 0, pt[0, :(n + P - 1) // P]], oc.pool[:, 0, pt[0, :(n + P - 1) // P]])
    kg = _logical_k(pool, pt, w, 1, n)
    k64 = oracle.rope_rotate_rows(k[0], 77, w.rope_theta, 0)
    assert np.abs(oracle.bf16_to_f64(kg[0]) - k64).max() <= 2e-2
    check_rotation_rounding(oracle, kg[0], k64)
    # 300 decode rows over the two sequences (rows alternate; 2 batch chunks)
    ids = [i % 2 for i in range(300)]
    q = syn.as_u16(syn.queries(w, 1, 300, 142))
    o = decode(kvg, dst, w, ids, q)
    scale = 1 / math.sqrt(w.head_dim)
    kk1, vv1, _ = oc.logical_kv(1, 0)
    for b in (0, 1, 255, 256, 299):
        kk, vv = (k[0], v[0]) if ids[b] == 0 else (kk1, vv1)
        compare_decode(oracle, o[0, b], oracle.gqa_decode(q[0, b], kk, vv, scale))
    o_noalloc = torch.empty_like(to_dev(q))
    qd = to_dev(q)
    kvg.kvg_decode_attention_noalloc(dst.h, -1, ids, qd.data_ptr(), w.n_q_heads, o_noalloc.data_ptr(), scale)
    torch.cuda.synchronize()
    # the same plan and worker count (the static scratch's cap does not bind
    # at 256 rows per launch here), so the same bytes
    assert np.array_equal(u16(o_noalloc), o)


def test_device_wait_gives_up_and_reports(oracle):
    # every kernel wait on an asynchronous copy is bounded; a wait that nothing
    # completes gives up, records a device-check status, and the context stays
    # usable (no trap, no hang)
    kvg = need_gpu()
    w = geometry("tiny")
    cache = kvg.Cache(dims_for(kvg, w), 20, 1, 320)
    kvg.kvg_selftest_bounded_wait(cache.h, 20_000_000)  # 20 ms
    with pytest.raises(kvg.KvgError) as e:
        kvg.kvg_sync(cache.h, None, 10.0)
    assert e.value.status == kvg.KVG_ERR_DEVICE_CHECK
    kvg.kvg_sync(cache.h, None, 10.0)  # status word cleared
    k, v = _kv(w, 100, 151)
    append(kvg, cache, 0, k, v, syn.positions(0, 100))
    q = syn.as_u16(syn.queries(w, w.n_layers, 1, 152))
    o = decode(kvg, cache, w, [0], q)
    compare_decode(oracle, o[0, 0], oracle.gqa_decode(q[0, 0], k[0], v[0], 1 / math.sqrt(w.head_dim)))
