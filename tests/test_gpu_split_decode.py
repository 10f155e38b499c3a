"""GPU parity of the split decode (kvg_decode_attention_range +
kvg_decode_state_finish) against the CPU oracle: one part over a slot range
equals the fp64 attention over that range's rows (within 1e-2); parts over
disjoint ranges merged into one state equal the attention over all rows;
windows intersect the range; empty ranges leave the state unchanged; the
result is run-to-run bitwise reproducible and identical for grafted and
freshly written rows under the same split."""
import hashlib
import math

import numpy as np
import pytest
import torch

import kvg_synth as syn
from kvg_testlib import (CANARY, append, compare_decode, dims_for, fill_canary, geometry, need_gpu,
                         oracle_dims, to_dev, u16)

pytestmark = pytest.mark.gpu

HBM_CAP = 1 << 30


def _kv(w, n, seed):
    k, v = syn.kv_rows(w, n, seed)
    return syn.as_u16(k), syn.as_u16(v)


def _sha(a: np.ndarray) -> bytes:
    return hashlib.sha256(np.ascontiguousarray(a).tobytes()).digest()


def _split(kvg, c, w, seq_ids, q, parts, layer=-1):
    """Runs the parts [(slot_begin, slot_end, flags)] into one state and
    finishes it; returns (bf16 bits [Lrun][B][Hq][D], state)."""
    qd = to_dev(q)
    Lr, B = q.shape[0], q.shape[1]
    state = torch.full((Lr, B, w.n_q_heads, w.head_dim + 4), float("nan"), dtype=torch.float32, device="cuda")
    scale = 1.0 / math.sqrt(w.head_dim)
    for lo, hi, fl in parts:
        kvg.kvg_decode_attention_range(c.h, layer, seq_ids, qd.data_ptr(), w.n_q_heads, scale, lo, hi, fl,
                                       state.data_ptr())
    out = torch.empty_like(qd)
    kvg.kvg_decode_state_finish(state.data_ptr(), Lr * B * w.n_q_heads, w.head_dim, out.data_ptr())
    torch.cuda.synchronize()
    return u16(out), state


def _stitched_case(kvg, oracle, w, seed):
    """Seq 0: ragged block grafted, fresh rows on its last page, a second
    block at the next page boundary (unfilled rows before it), fresh rows;
    seq 1 a long fresh write; seq 2 three rows; seq 3 one row; seqs 4 / 5:
    block A + fresh rows, grafted / written fresh."""
    P = w.page_size
    dims = dims_for(kvg, w)
    od = oracle_dims(oracle, w)
    na, nb_, nc, nd = 2 * P + 5, P + 2, P + 7, 3
    k, v = _kv(w, na + nb_ + nc + nd + 5 * P, seed)
    parts, t = [], 0
    for n in (na, nb_, nc, nd):
        parts.append((k[:, t:t + n], v[:, t:t + n], syn.positions(t, n)))
        t += n
    k_long, v_long = k[:, t:t + 5 * P], v[:, t:t + 5 * P]
    max_slots, n_pages = 8 * P + 64, 80
    src = kvg.Cache(dims, n_pages, 2, max_slots)
    store = kvg.Store(dims, 0, HBM_CAP)
    bids = []
    for i, (kk, vv, pp) in enumerate((parts[0], parts[2])):
        append(kvg, src, i, kk, vv, pp)
        bids.append(kvg.kvg_deposit(store.h, src.h, i, 0, pp.size))
    c = kvg.Cache(dims, n_pages, 6, max_slots)
    fill_canary(c)
    kvg.kvg_cache_set_free_order(c.h, syn.permutation(n_pages, seed + 1))
    oc = oracle.OracleCache(od, n_pages, 6, max_slots, fill=CANARY)
    oc.set_free_order(syn.permutation(n_pages, seed + 1))
    kvg.kvg_graft(store.h, bids[0], c.h, 0, -1, 0, kvg.KVG_GRAFT_SYNC)
    oc.graft(0, oracle.block_from_kv(od, *parts[0]))
    append(kvg, c, 0, *parts[1])
    oc.append(0, *parts[1])
    kvg.kvg_graft(store.h, bids[1], c.h, 0, -1, 0, kvg.KVG_GRAFT_SYNC)
    oc.graft(0, oracle.block_from_kv(od, *parts[2]))
    append(kvg, c, 0, *parts[3])
    oc.append(0, *parts[3])
    append(kvg, c, 1, k_long, v_long, syn.positions(0, 5 * P))
    oc.append(1, k_long, v_long, syn.positions(0, 5 * P))
    append(kvg, c, 2, k[:, :3], v[:, :3], syn.positions(0, 3))
    oc.append(2, k[:, :3], v[:, :3], syn.positions(0, 3))
    append(kvg, c, 3, k[:, 7:8], v[:, 7:8], syn.positions(0, 1))
    oc.append(3, k[:, 7:8], v[:, 7:8], syn.positions(0, 1))
    kvg.kvg_graft(store.h, bids[0], c.h, 4, -1, 0, kvg.KVG_GRAFT_SYNC)
    append(kvg, c, 4, *parts[1])
    append(kvg, c, 5, np.concatenate([parts[0][0], parts[1][0]], 1), np.concatenate([parts[0][1], parts[1][1]], 1),
           syn.positions(0, na + nb_))
    return c, oc, k, v, max_slots


def _windows(w):
    P = w.page_size
    return [(1, P + 3, 0, 2 * P + 5)[l % 4] for l in range(w.n_layers)]


@pytest.mark.parametrize("geo,windowed", [("tiny", False), ("tiny", True), ("d128", True), ("d256", False),
                                          ("g4", True)])
def test_split_decode_matches_oracle(oracle, geo, windowed):
    kvg = need_gpu()
    w = geometry(geo)
    P = w.page_size
    c, oc, k, v, max_slots = _stitched_case(kvg, oracle, w, 91)
    if windowed:
        kvg.kvg_cache_set_layer_windows(c.h, _windows(w))
        oc.set_layer_windows(_windows(w))
    scale = 1.0 / math.sqrt(w.head_dim)
    rows = [0, 1, 2, 3]
    q = syn.as_u16(syn.queries(w, w.n_layers, len(rows), 92))
    M = kvg.KVG_DECODE_MERGE
    end = max_slots
    # one part over everything
    o_all, _ = _split(kvg, c, w, rows, q, [(0, end, 0)])
    # three parts merged, a range out past every sequence's end in the middle
    cuts = [(0, P, 0), (3 * P, end, M), (P, 3 * P, M), (5 * P, 5 * P, M)]
    o_3, st3 = _split(kvg, c, w, rows, q, cuts)
    # one part alone
    o_mid, _ = _split(kvg, c, w, rows, q, [(P, 3 * P, 0)])
    for l in range(w.n_layers):
        for b, sq in enumerate(rows):
            full = oc.decode(sq, l, q[l, b], scale)
            compare_decode(oracle, o_all[l, b], full)
            compare_decode(oracle, o_3[l, b], full)
            compare_decode(oracle, o_mid[l, b], oc.decode_range(sq, l, q[l, b], scale, P, 3 * P))
    # a one-row sequence: weight exactly 1, so o is that value row bit for bit
    G = w.group
    for l in range(w.n_layers):
        for h in range(w.n_q_heads):
            assert np.array_equal(o_3[l, 3, h], v[l, 7, h // G])
            assert float(st3[l, 3, h, w.head_dim + 1]) == 1.0
    # run-to-run bitwise determinism of the same call sequence
    for _ in range(2):
        assert _sha(_split(kvg, c, w, rows, q, cuts)[0]) == _sha(o_3)
    # grafted (seq 4) and fresh (seq 5) rows: identical bytes under the same split
    q2 = syn.as_u16(syn.queries(w, w.n_layers, 1, 93))
    assert _sha(_split(kvg, c, w, [4], q2, cuts)[0]) == _sha(_split(kvg, c, w, [5], q2, cuts)[0])
    # one layer at a time
    l = w.n_layers - 1
    ol, _ = _split(kvg, c, w, rows, q[l:l + 1], cuts, layer=l)
    for b, sq in enumerate(rows):
        compare_decode(oracle, ol[0, b], oc.decode(sq, l, q[l, b], scale))
    kvg.kvg_sync(c.h)


def test_split_decode_empty_parts_keep_the_state():
    kvg = need_gpu()
    w = geometry("tiny")
    P = w.page_size
    dims = dims_for(kvg, w)
    c = kvg.Cache(dims, 16, 2, 8 * P)
    k, v = _kv(w, 3 * P + 2, 94)
    append(kvg, c, 0, k, v, syn.positions(0, 3 * P + 2))
    q = syn.as_u16(syn.queries(w, w.n_layers, 2, 95))
    M = kvg.KVG_DECODE_MERGE
    o1, s1 = _split(kvg, c, w, [0, 1], q, [(0, 2 * P, 0), (2 * P, 8 * P, M)])
    o2, s2 = _split(kvg, c, w, [0, 1], q, [(0, 2 * P, 0), (2 * P, 8 * P, M), (P, P, M), (6 * P, 8 * P, M)])
    assert torch.equal(s1, s2) and _sha(o1) == _sha(o2)
    # seq 1 is empty: state l = 0, m = -inf, o = 0, output 0
    assert not o1[:, 1].any()
    assert (s1[:, 1, :, w.head_dim + 1] == 0).all() and torch.isinf(s1[:, 1, :, w.head_dim]).all()
    assert (s1[:, 1, :, :w.head_dim] == 0).all()


def test_split_decode_many_rows_per_call(oracle):
    """More batch rows than one launch takes (256): the state rows of the
    second launch land at their own batch index."""
    kvg = need_gpu()
    w = geometry("tiny")
    P = w.page_size
    B = 300
    dims = dims_for(kvg, w)
    c = kvg.Cache(dims, 2 * B + 8, B, 4 * P)
    od = oracle_dims(oracle, w)
    oc = oracle.OracleCache(od, 2 * B + 8, B, 4 * P)
    k, v = _kv(w, P + 5, 96)
    for b in range(B):
        n = 1 + (b * 7) % (P + 5)
        append(kvg, c, b, k[:, :n], v[:, :n], syn.positions(0, n))
        oc.append(b, k[:, :n], v[:, :n], syn.positions(0, n))
    q = syn.as_u16(syn.queries(w, w.n_layers, B, 97))
    o, _ = _split(kvg, c, w, list(range(B)), q, [(P, 4 * P, 0), (0, P, kvg.KVG_DECODE_MERGE)])
    scale = 1.0 / math.sqrt(w.head_dim)
    for l in range(w.n_layers):
        for b in range(0, B, 7):
            compare_decode(oracle, o[l, b], oc.decode(b, l, q[l, b], scale))


def test_split_decode_host_checks():
    kvg = need_gpu()
    w = geometry("tiny")
    P = w.page_size
    c = kvg.Cache(dims_for(kvg, w), 8, 1, 4 * P)
    q = to_dev(syn.as_u16(syn.queries(w, w.n_layers, 1, 98)))
    st = torch.zeros((w.n_layers, 1, w.n_q_heads, w.head_dim + 4), dtype=torch.float32, device="cuda")
    bad = [(1, 2 * P, 0), (P, 0, 0), (-P, P, 0), (0, P + 1, 0), (0, P, 4)]
    for lo, hi, fl in bad:
        with pytest.raises(kvg.KvgError) as e:
            kvg.kvg_decode_attention_range(c.h, -1, [0], q.data_ptr(), w.n_q_heads, 0.125, lo, hi, fl, st.data_ptr())
        assert e.value.status == kvg.KVG_ERR_ARG
    with pytest.raises(kvg.KvgError):
        kvg.kvg_decode_attention_range(c.h, -1, [0], q.data_ptr(), w.n_q_heads, 0.125, 0, P, 0, 0)
    with pytest.raises(kvg.KvgError):
        kvg.kvg_decode_state_finish(st.data_ptr(), 4, 96, q.data_ptr())
    # slot_end at or past max_slots means "to the end", page-aligned or not
    kvg.kvg_decode_attention_range(c.h, -1, [0], q.data_ptr(), w.n_q_heads, 0.125, 0, 4 * P + 3, 0, st.data_ptr())
    torch.cuda.synchronize()


@pytest.mark.parametrize("residency,n_pages_block,n_events", [(1, 41, 16), (1, 130, 16), (0, 41, 16), (1, 41, 4),
                                                                (1, 130, 1)])
def test_chunked_graft_feeds_a_pipelined_split_decode(oracle, residency, n_pages_block, n_events):
    """kvg_graft_chunked (verified) on a side stream, and on the main stream:
    the fresh rows appended and decoded into a state, then each chunk's
    slots merged in as soon as its event fires.  The output equals, bit for
    bit, the same parts merged in the same order after a synchronous graft
    (so no part read rows that had not landed yet: the destination starts
    as canary bytes), and the oracle within 1e-2.  The chunk ends are page-aligned, increasing and
    end at the block's length; a pinned-host store's verified graft uses
    several chunks (the last one short), an HBM store's one; with fewer
    events than chunks (4, or 1) consecutive chunks share an event."""
    kvg = need_gpu()
    w = geometry("d128")
    P = w.page_size
    nb, nf = n_pages_block * P, 3 * P + 11
    dims = dims_for(kvg, w)
    od = oracle_dims(oracle, w)
    k, v = _kv(w, nb + nf, 91)
    pos = syn.positions(0, nb + nf)
    max_slots = nb + nf + 2 * P
    n_pages = max_slots // P + 4
    src = kvg.Cache(dims, n_pages, 1, max_slots)
    append(kvg, src, 0, k[:, :nb], v[:, :nb], pos[:nb])
    store = kvg.Store(dims, residency, 1 << 30)
    bid = kvg.kvg_deposit(store.h, src.h, 0, 0, nb)
    torch.cuda.synchronize()
    q = syn.as_u16(syn.queries(w, w.n_layers, 1, 92))
    qd = to_dev(q)
    kf, vf, pf = to_dev(np.ascontiguousarray(k[:, nb:])), to_dev(np.ascontiguousarray(v[:, nb:])), to_dev(pos[nb:])
    scale = 1.0 / math.sqrt(w.head_dim)

    def run(chunked, same_ends=None):
        c = kvg.Cache(dims, n_pages, 1, max_slots)
        fill_canary(c)
        kvg.kvg_cache_set_free_order(c.h, syn.permutation(n_pages, 93))
        main, side = torch.cuda.Stream(), torch.cuda.Stream()
        state = torch.full((w.n_layers, 1, w.n_q_heads, w.head_dim + 4), float("nan"), dtype=torch.float32,
                           device="cuda")
        out = torch.empty_like(qd)
        torch.cuda.synchronize()
        if chunked:
            events = [torch.cuda.Event() for _ in range(n_events)]
            for e in events:
                e.record(side)  # creates the event
            ends = kvg.kvg_graft_chunked(store.h, bid, c.h, 0, [e.cuda_event for e in events],
                                         flags=kvg.KVG_GRAFT_VERIFY, stream=side)
        else:
            kvg.kvg_graft(store.h, bid, c.h, 0, -1, 0, kvg.KVG_GRAFT_VERIFY | kvg.KVG_GRAFT_SYNC)
            ends = same_ends  # the same parts, merged in the same order
        kvg.kvg_cache_append(c.h, 0, kf.data_ptr(), vf.data_ptr(), pf.data_ptr(), nf, main)
        kvg.kvg_decode_attention_range(c.h, -1, [0], qd.data_ptr(), w.n_q_heads, scale, nb, max_slots, 0,
                                       state.data_ptr(), main)
        lo = 0
        for j, hi in enumerate(ends):
            if chunked:
                main.wait_event(events[j])
            kvg.kvg_decode_attention_range(c.h, -1, [0], qd.data_ptr(), w.n_q_heads, scale, lo, hi,
                                           kvg.KVG_DECODE_MERGE, state.data_ptr(), main)
            lo = hi
        main.wait_stream(side)  # the digest verdict covers the whole block
        kvg.kvg_decode_state_finish(state.data_ptr(), w.n_layers * w.n_q_heads, w.head_dim, out.data_ptr(), main)
        kvg.kvg_sync(c.h, main, 60.0)  # raises on a digest mismatch
        torch.cuda.synchronize()
        return u16(out), ends, c

    got, ends, c = run(True)
    assert 1 <= len(ends) <= n_events and ends[-1] == nb
    assert all(e % P == 0 for e in ends) and all(a < b for a, b in zip(ends, ends[1:]))
    if residency == kvg.KVG_RESIDENCY_PINNED_HOST and n_events == 16:
        assert len(ends) > 1 and ends[-1] - ends[-2] <= ends[0]  # the last chunk is short
    elif residency == kvg.KVG_RESIDENCY_PINNED_HOST:
        assert len(ends) == n_events  # fewer events than chunks: chunks share events
    else:
        assert ends == [nb]
    want, _, _ = run(False, ends)
    assert np.array_equal(got, want)
    oc = oracle.OracleCache(od, n_pages, 1, max_slots)
    oc.append(0, k, v, pos)
    o_ref = np.stack([oc.decode(0, l, q[l, 0], scale) for l in range(w.n_layers)])[:, None]
    compare_decode(oracle, got, o_ref)
