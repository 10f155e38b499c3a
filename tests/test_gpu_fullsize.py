"""Parity at the benchmark's full sizes, in the launch configuration bench.py
times (its workload classes build the state): bit-exact block bytes, page
digests, page tables and restored pages against the oracle; attention on
every query head of two layers (of several sequences where there are
several), through the decode gate of kvg_testlib.compare_decode, and
relocated keys on sampled pages; the grafted-vs-fresh SHA-256 gate and
run-to-run determinism at 32k context; the deep store's planted needles on
every one of 1,000 grafts."""
import hashlib
import math

import numpy as np
import pytest
import torch

import kvg_synth as syn
from kvg_testlib import check_rotation_rounding, compare_decode, dev_view, need_gpu, tables

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _free_device_memory():
    """Each workload takes most of the GPU: release what earlier tests cached."""
    import gc
    gc.collect()
    if torch.cuda.is_available():
        torch.cuda.empty_cache()
    yield
    gc.collect()
    if torch.cuda.is_available():
        torch.cuda.empty_cache()


def _od(oracle, w):
    return oracle.Dims(w.n_layers, w.n_kv_heads, w.head_dim, w.page_size, w.rope_theta, 0)


def _pool_page(cache, w, l, kv, pid):
    """Bytes of one (layer, K/V) page of the pool, as uint16 [Hkv][P][D]."""
    v = cache.view
    pb = w.page_bytes
    off = ((l * 2 + kv) * v.n_pages + int(pid)) * pb
    t = dev_view(v.pool + off, pb, torch.int16).cpu().numpy().view(np.uint16)
    return t.reshape(w.n_kv_heads, w.page_size, w.head_dim)


def _sha(t: torch.Tensor) -> bytes:
    return hashlib.sha256(t.contiguous().view(torch.int16).cpu().numpy().tobytes()).digest()


def _close(*objs):
    for o in objs:
        o.close()
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


def test_12b_single_graft_full_size(oracle):
    kvg = need_gpu()
    import bench
    dev = torch.device("cuda", 0)
    s, side = torch.cuda.Stream(), torch.cuda.Stream()
    st = bench.Step12B(kvg, dev, s, side)
    fresh = None
    try:
        st.run_step()
        s.synchronize()
        kvg.kvg_sync(st.cache.h, s, 60.0)  # every restored page matched its stored digest
        w, nb, nf, P = st.w, st.nb, st.nf, st.w.page_size
        kb, vb = syn.as_u16(st.kb), syn.as_u16(st.vb)
        od = _od(oracle, w)
        blk = oracle.block_from_kv(od, kb, vb, syn.positions(0, nb))
        ser = blk.serialize()  # 12,288 page digests computed by the oracle
        assert kvg.kvg_store_export(st.store.h, st.bid) == ser
        assert kvg.kvg_store_export(st.hstore.h, st.hbid) == ser
        # page tables, fills and position tags: the oracle's bookkeeping of the same calls
        meta = oracle.OracleCache(od, st.cache.view.n_pages, 2, syn.B12_CTX, with_pool=False)
        meta.append(1, None, None, syn.positions(0, nb))
        meta.release(1)
        meta.release(0)
        meta.graft(0, oracle.BlockMeta(od, syn.positions(0, nb)))
        meta.append(0, None, None, syn.positions(nb, nf))
        pt, pf, ps = tables(st.cache)
        assert np.array_equal(pt, meta.page_table) and np.array_equal(pf, meta.page_fill)
        assert np.array_equal(ps, meta.positions)
        # restored pages equal the block's pages: 48 sampled (layer, K/V, page)
        rng = np.random.default_rng(1)
        for _ in range(48):
            l, kv, j = int(rng.integers(w.n_layers)), int(rng.integers(2)), int(rng.integers(nb // P))
            assert np.array_equal(_pool_page(st.cache, w, l, kv, pt[0, j]), blk.pages[l, kv, j])
        # decode: every query head of two layers against fp64 attention over
        # all 32,768 rows, through the decode gate
        kf, vf = st.kf, st.vf
        rows = {}
        for l in (0, 17, w.n_layers - 1):
            rows[l] = (np.concatenate([kb[l], syn.as_u16(kf[l])]), np.concatenate([vb[l], syn.as_u16(vf[l])]))
        for l in (0, w.n_layers - 1):
            ref = oracle.gqa_decode(syn.as_u16(st.q[l, 0]), rows[l][0], rows[l][1], st.scale)
            compare_decode(oracle, syn.as_u16(st.out[l, 0]), ref, what=f"12b layer {l}")
        # the same 32,768 rows written fresh into other pages: SHA-256-identical output
        out_grafted = st.out.clone()
        fresh = kvg.Cache(st.dims, st.cache.view.n_pages, 1, syn.B12_CTX)
        kvg.kvg_cache_set_free_order(fresh.h, syn.permutation(st.cache.view.n_pages, 5))
        pb_ = torch.arange(nb, dtype=torch.int32, device=dev)
        kvg.kvg_cache_append(fresh.h, 0, st.kb.data_ptr(), st.vb.data_ptr(), pb_.data_ptr(), nb, s)
        kvg.kvg_cache_append(fresh.h, 0, kf.data_ptr(), vf.data_ptr(), st.pf.data_ptr(), nf, s)
        out_fresh = torch.empty_like(st.q)
        kvg.kvg_decode_attention(fresh.h, -1, [0], st.q.data_ptr(), w.n_q_heads, out_fresh.data_ptr(),
                                 st.scale, s)
        s.synchronize()
        assert _sha(out_fresh) == _sha(out_grafted)
        # run-to-run: two more full steps give the same bytes
        for _ in range(2):
            st.run_step()
            s.synchronize()
            assert _sha(st.out) == _sha(out_grafted)
        # the end-to-end form: verified graft from the pinned-host store (16
        # chunks on a capped grid) with the split decode (fresh rows while the
        # block streams in, the block's rows merged after): digests verified,
        # restored pages bit-exact, every head of two layers through the decode
        # gate, bitwise reproducible
        st.run_step_split(st.hstore.h, st.hbid)
        s.synchronize()
        kvg.kvg_sync(st.cache.h, s, 60.0)
        pt, _, _ = tables(st.cache)
        for _ in range(16):
            l, kv, j = int(rng.integers(w.n_layers)), int(rng.integers(2)), int(rng.integers(nb // P))
            assert np.array_equal(_pool_page(st.cache, w, l, kv, pt[0, j]), blk.pages[l, kv, j])
        out_split = st.out.clone()
        for l in (17, w.n_layers - 1):
            ref = oracle.gqa_decode(syn.as_u16(st.q[l, 0]), rows[l][0], rows[l][1], st.scale)
            compare_decode(oracle, syn.as_u16(out_split[l, 0]), ref, what=f"12b split layer {l}")
        assert float((out_split.float() - out_grafted.float()).abs().max()) <= 1e-2
        st.run_step_split(st.hstore.h, st.hbid)
        s.synchronize()
        assert _sha(st.out) == _sha(out_split)
    finally:
        _close(*(x for x in (fresh, st.cache, st.store, st.hstore) if x is not None))


def _rows31(st, dev, layers, seqs):
    """Host copies (uint16 [len(layers)][rows][Hkv][D]) of the K/V rows the
    31B workload wrote: the block's rows (as deposited) and each listed
    sequence's fresh rows, regenerated chunk by chunk from their seeds."""
    li = torch.tensor(layers, device=dev)
    kb, vb = [], []
    for i in range(st.nb // st.CHUNK):
        k, v = st.block_rows(i, dev)
        kb.append(syn.as_u16(k.index_select(0, li)))
        vb.append(syn.as_u16(v.index_select(0, li)))
        del k, v
    fresh = {}
    for sq in seqs:
        kf, vf = [], []
        for i in range(st.n_fresh_chunks):
            k, v = st.fresh_rows(sq, i, dev)
            kf.append(syn.as_u16(k.index_select(0, li)))
            vf.append(syn.as_u16(v.index_select(0, li)))
            del k, v
        fresh[sq] = (np.concatenate(kf, axis=1), np.concatenate(vf, axis=1))
    return np.concatenate(kb, axis=1), np.concatenate(vb, axis=1), fresh


def test_31b_relocation_full_size(oracle):
    kvg = need_gpu()
    import bench
    dev = torch.device("cuda", 0)
    s = torch.cuda.Stream()
    st = bench.Step31B(kvg, dev, s)
    try:
        st.run_step()
        s.synchronize()
        kvg.kvg_sync(st.cache.h, s, 60.0)
        w, nb, P = st.w, st.nb, st.w.page_size
        pt, pf, ps = tables(st.cache)
        # position tags: block tags + delta, then the fresh rows' tags
        for sq in range(st.B):
            d = st.deltas[sq]
            assert np.array_equal(ps[sq, :nb], np.arange(nb) + d)
            assert np.array_equal(ps[sq, nb:st.ctx], np.arange(nb, st.ctx) + d)
        assert np.array_equal(ps[st.B, :nb], np.arange(nb) + 4096)  # the timed relocation
        sample_layers = [0, 29, w.n_layers - 1]
        seqs = [0, 1, 3, 6]  # delta 0, 1, 100000, 4096
        kb, vb, fresh = _rows31(st, dev, sample_layers, seqs)
        # relocated keys (every kv head) within 2e-2 of the fp64 rotation;
        # values and delta-0 keys bit-exact
        rng = np.random.default_rng(3)
        for sq, d in [(3, st.deltas[3]), (1, st.deltas[1]), (0, 0), (st.B, 4096)]:
            for _ in range(6):
                li, j = int(rng.integers(len(sample_layers))), int(rng.integers(nb // P))
                l = sample_layers[li]
                kpage = _pool_page(st.cache, w, l, 0, pt[sq, j])
                vpage = _pool_page(st.cache, w, l, 1, pt[sq, j])
                rows_k = kb[li, j * P:(j + 1) * P].transpose(1, 0, 2)  # [Hkv][P][D]
                rows_v = vb[li, j * P:(j + 1) * P].transpose(1, 0, 2)
                assert np.array_equal(vpage, rows_v)
                if d == 0:
                    assert np.array_equal(kpage, rows_k)
                else:
                    ref = oracle.rope_rotate_rows(rows_k, d, w.rope_theta, 0)
                    assert np.abs(oracle.bf16_to_f64(kpage) - ref).max() <= 2e-2
                    check_rotation_rounding(oracle, kpage, ref)
        # the fresh rows landed where the oracle's bookkeeping puts them (one
        # sampled page per sampled sequence and layer)
        for sq in seqs:
            j = nb // P + int(rng.integers((st.ctx - nb) // P))
            t0 = j * P - nb
            for li, l in enumerate(sample_layers):
                assert np.array_equal(_pool_page(st.cache, w, l, 0, pt[sq, j]),
                                      fresh[sq][0][li, t0:t0 + P].transpose(1, 0, 2))
        # decode: every query head of two layers of four sequences against
        # fp64 attention over all 65,536 rows, through the decode gate
        for sq in seqs:
            d = st.deltas[sq]
            for li in (0, len(sample_layers) - 1):
                l = sample_layers[li]
                kblk = kb[li] if d == 0 else oracle.rope_rotate_rows_bf16(kb[li], d, w.rope_theta, 0)
                k = np.concatenate([kblk, fresh[sq][0][li]])
                v = np.concatenate([vb[li], fresh[sq][1][li]])
                ref = oracle.gqa_decode(syn.as_u16(st.q[l, sq]), k, v, st.scale)
                compare_decode(oracle, syn.as_u16(st.out[l, sq]), ref, what=f"31b seq {sq} layer {l}")
    finally:
        _close(st.cache, st.store)


@pytest.mark.parametrize("consecutive", [False, True])
def test_batched_library_full_size(oracle, consecutive):
    """The batched library at its 4-layer slice; consecutive: blocks 2-4 of
    every sequence re-based by the tokens before them (per-graft deltas in
    the one batched call)."""
    kvg = need_gpu()
    import bench
    dev = torch.device("cuda", 0)
    s = torch.cuda.Stream()
    st = bench.StepBatched(kvg, dev, s, 4, consecutive=consecutive)
    try:
        st.run_step()
        s.synchronize()
        kvg.kvg_sync(st.cache.h, s, 60.0)
        w, P, nS = st.w, st.w.page_size, syn.BATCHED_SEQS
        od = _od(oracle, w)
        # page tables, fills, positions: the oracle's bookkeeping of the same calls
        meta = oracle.OracleCache(od, st.cache.view.n_pages, nS + 1, st.max_slots, with_pool=False)
        for n in st.lens:
            meta.append(nS, None, None, syn.positions(0, int(n)))
            meta.release(nS)
        delta_of = {}
        for sq in range(nS):
            meta.release(sq)
            run = 0
            for b in st.ids[sq]:
                d = run if consecutive else 0
                delta_of[(sq, int(b))] = d
                meta.graft(sq, oracle.BlockMeta(od, syn.positions(0, int(st.lens[b]))), delta=d)
                run += int(st.lens[b])
        posn = st.pos.cpu().numpy()
        for t in range(st.steps):  # one decode-step row per sequence, in batch order
            for sq in range(nS):
                meta.append(sq, None, None, posn[t, sq:sq + 1])
        pt, pf, ps = tables(st.cache)
        assert np.array_equal(pt, meta.page_table) and np.array_equal(pf, meta.page_fill)
        assert np.array_equal(ps, meta.positions)
        # grafted pages equal the deposited blocks' pages (sampled), incl. ragged tail pages
        for sq in (0, 13, nS - 1):
            j0 = 0
            for b in st.ids[sq]:
                n = int(st.lens[b])
                k, v = syn.kv_rows(w, n, w.seed + int(b), "cuda")
                blk = oracle.block_from_kv(od, syn.as_u16(k), syn.as_u16(v), syn.positions(0, n))
                d = delta_of[(sq, int(b))]
                for j in (0, blk.n_pages - 1):
                    for kv in (0, 1):
                        got = _pool_page(st.cache, w, w.n_layers - 1, kv, pt[sq, j0 + j])
                        want = blk.pages[w.n_layers - 1, kv, j]
                        if j == blk.n_pages - 1 and n % P:
                            # the tail page's fill rows are the block's; later rows
                            # belong to the decode appends of the last block only
                            got, want = got[:, :n % P], want[:, :n % P]
                        if kv == 0 and d:
                            ref = oracle.rope_rotate_rows(want, d, w.rope_theta, 0)
                            assert np.abs(oracle.bf16_to_f64(got) - ref).max() <= 2e-2
                            check_rotation_rounding(oracle, got, ref)
                        else:
                            assert np.array_equal(got, want)
                j0 += blk.n_pages
        # decode after the last step: every query head of two layers of three
        # sequences against fp64 attention, through the decode gate
        for sq in (0, 13, nS - 1):
            for l in (0, w.n_layers - 1):
                ks, vs = [], []
                for b in st.ids[sq]:
                    k, v = syn.kv_rows(w, int(st.lens[b]), w.seed + int(b), "cuda")
                    kl = syn.as_u16(k[l])
                    d = delta_of[(sq, int(b))]
                    ks.append(oracle.rope_rotate_rows_bf16(kl, d, w.rope_theta, 0) if d else kl)
                    vs.append(syn.as_u16(v[l]))
                ks.append(syn.as_u16(st.kd[l, sq::nS]))
                vs.append(syn.as_u16(st.vd[l, sq::nS]))
                ref = oracle.gqa_decode(syn.as_u16(st.q[l, sq]), np.concatenate(ks), np.concatenate(vs), st.scale)
                compare_decode(oracle, syn.as_u16(st.out[l, sq]), ref,
                               what=f"batched{' consecutive' if consecutive else ''} seq {sq} layer {l}")
        if not consecutive:
            # every page of all 128 grafts: the batch again, digest-verified
            # (each restored page's SHA-256 against the block's stored digest)
            # before any decode-step row lands in a ragged tail page
            for sq in range(nS):
                kvg.kvg_cache_release(st.cache.h, sq, s)
            rep = kvg.kvg_graft_report()
            kvg.kvg_graft_batch(st.store.h, st.batch_bids, st.cache.h, st.batch_seqs,
                                kvg.KVG_GRAFT_VERIFY | kvg.KVG_GRAFT_SYNC, s, report=rep)
            n_blk_pages = sum(-(-int(st.lens[b]) // P) for sq in range(nS) for b in st.ids[sq])
            assert rep.n_mismatch == 0 and rep.n_pages_checked == w.n_layers * 2 * n_blk_pages
    finally:
        _close(st.cache, st.store)


def test_deep_store_needles_full_size(oracle):
    kvg = need_gpu()
    import bench
    dev = torch.device("cuda", 0)
    s = torch.cuda.Stream()
    st = bench.StepDeep(kvg, dev, s)
    try:
        w = st.w
        od = _od(oracle, w)
        # blocks at several depths: serialized bytes equal the oracle's block
        for b in (0, 697, st.n_blocks - 1):
            k, v = st.block_rows(b, dev)
            blk = oracle.block_from_kv(od, syn.as_u16(k), syn.as_u16(v), syn.positions(0, st.nb))
            assert kvg.kvg_store_export(st.store.h, b) == blk.serialize()
        # every one of the 1,000 random grafts: every restored page's SHA-256
        # equals the block's stored page digest (the block bytes, pinned to
        # the oracle above), and the decode reads its own block's needle (and
        # so not the previous block's: the window really moves)
        prev = None
        rep = kvg.kvg_graft_report()
        for _ in range(len(st.order)):
            b = st.run_step()
            kvg.kvg_verify(st.store.h, b, st.cache.h, 0, 0, kvg.KVG_GRAFT_SYNC, s, report=rep)
            assert rep.n_mismatch == 0 and rep.n_pages_checked == w.n_layers * 2 * (st.nb // w.page_size), b
            assert st.needle_error(b) <= 1e-2, b
            if prev is not None and st.tag(prev) != st.tag(b):
                assert float((st.out.float() - st.tag(prev)).abs().max()) > 1e-2
            prev = b
        # the needle read matches fp64 attention over the grafted rows (sampled)
        b = int(st.order[-1])
        k, v = st.block_rows(b, dev)
        for l in range(w.n_layers):
            ref = oracle.gqa_decode(syn.as_u16(st.q[l, 0]), syn.as_u16(k[l]), syn.as_u16(v[l]), st.scale)
            compare_decode(oracle, syn.as_u16(st.out[l, 0]), ref, what=f"deep block {b} layer {l}")
    finally:
        _close(st.cache, st.store)
