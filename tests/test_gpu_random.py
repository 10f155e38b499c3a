"""Seeded random scenarios against the oracle: random geometries (head_dim,
query group, KV heads, layers, page size, RoPE pairing and base), several
sequences, each built by a random mix of own-position grafts, re-based
grafts and fresh appends of ragged lengths, through single grafts and
batched ones; then every table, tag and pool byte is compared with the
oracle's cache (re-based key rows within 2e-2 of the fp64 rotation, every
other byte exact) and one decode over every sequence goes through the decode
gate, whole and split at a random page boundary into two merged parts
(odd seeds with random sliding windows).  fp8 E4M3 caches get their own
scenarios (own-position grafts and appends).  The scenarios are drawn from
fixed seeds, so a failure names a case that reproduces."""
import math
import os

import numpy as np
import pytest
import torch

import kvg_synth as syn
from kvg_testlib import (CANARY, append, check_rotation_rounding, compare_decode, decode, dev_view, dims_for,
                         fill_canary, need_gpu,
                         oracle_dims, pool_u16, tables, to_dev, u16)

pytestmark = pytest.mark.gpu

# (head_dim, query group) pairs the decode kernel is built for (bf16)
GROUPS = {64: (1, 2, 4, 8), 128: (1, 2, 4), 256: (1, 2)}
# KVG_RANDOM_CASES widens the draw for a longer soak (default 64)
N_CASES = int(os.environ.get("KVG_RANDOM_CASES", "64"))
N_FP8_CASES = int(os.environ.get("KVG_RANDOM_FP8_CASES", "16"))


def _case(seed):
    rng = np.random.default_rng(0x5CE0 + seed)
    D = int(rng.choice([64, 128, 256]))
    G = int(rng.choice(GROUPS[D]))
    Hkv = int(rng.choice([1, 2, 4]))
    L = int(rng.integers(1, 4))
    P = int(rng.choice([16, 32, 64]))
    style = int(rng.integers(0, 2))
    theta = float(rng.choice([1e4, 1e6]))
    w = syn.Workload(f"rand{seed}", L, G * Hkv, Hkv, D, P, theta, 0x5CE0 + seed)
    return rng, w, style


@pytest.mark.parametrize("seed", range(N_CASES))
def test_random_scenario_matches_oracle(oracle, seed):
    kvg = need_gpu()
    rng, w, style = _case(seed)
    P, L = w.page_size, w.n_layers
    dims = dims_for(kvg, w, style)
    od = oracle_dims(oracle, w, style)
    # the store: 1-3 blocks of ragged lengths, deposited at positions 0 .. n-1
    lens = [int(x) for x in rng.integers(1, 3 * P + 9, size=int(rng.integers(1, 4)))]
    src = kvg.Cache(dims, 4 * max(lens) // P + 8, 1, 4 * max(lens) + 4 * P)
    store = kvg.Store(dims, int(rng.integers(0, 2)), 1 << 28)  # HBM or pinned host
    bids, oblks, krows = [], [], []
    for i, n in enumerate(lens):
        k, v = syn.kv_rows(w, n, w.seed + i)
        k, v = syn.as_u16(k), syn.as_u16(v)
        append(kvg, src, 0, k, v, syn.positions(0, n))
        bids.append(kvg.kvg_deposit(store.h, src.h, 0, 0, n))
        kvg.kvg_cache_release(src.h, 0)
        oblks.append(oracle.block_from_kv(od, k, v, syn.positions(0, n)))
        krows.append(k)
    # the destination: 1-4 sequences, each a random list of operations
    n_seqs = int(rng.integers(1, 5))
    ops = []  # (seq, "graft", block, delta) or (seq, "append", n)
    for sq in range(n_seqs):
        for _ in range(int(rng.integers(1, 4))):
            if rng.random() < 0.6:
                b = int(rng.integers(len(lens)))
                delta = int(rng.choice([0, 0, int(rng.integers(1, 5000)), int(rng.integers(100_000, 2_000_000))]))
                ops.append((sq, "graft", b, delta))
            else:
                ops.append((sq, "append", int(rng.integers(1, 2 * P + 4))))
    slots_bound = sum(-(-(o[2] if o[1] == "append" else lens[o[2]]) // P) + 1 for o in ops) * P
    n_pages = slots_bound // P + 4
    c = kvg.Cache(dims, n_pages, n_seqs, slots_bound)
    fill_canary(c)
    order = syn.permutation(n_pages, seed)
    kvg.kvg_cache_set_free_order(c.h, order)
    oc = oracle.OracleCache(od, n_pages, n_seqs, slots_bound, fill=CANARY)
    oc.set_free_order(order)
    use_batch = seed % 2 == 0
    rotated = []  # (seq, first slot, block, delta) of re-based grafts
    next_tag = [0] * n_seqs
    i = 0
    while i < len(ops):
        # even seeds: a run of consecutive grafts goes through one kvg_graft_batch
        j = i
        while use_batch and j < len(ops) and ops[j][1] == "graft":
            j += 1
        run = ops[i:j] if j > i else [ops[i]]
        if run[0][1] == "graft" and len(run) > 1:
            kvg.kvg_graft_batch(store.h, [bids[o[2]] for o in run], c.h, [o[0] for o in run],
                                kvg.KVG_GRAFT_VERIFY | kvg.KVG_GRAFT_SYNC, deltas=[o[3] for o in run])
        for o in run:
            sq = o[0]
            if o[1] == "graft":
                b, delta = o[2], o[3]
                dst = -(-int(oc.n_slots[sq]) // P) * P
                if len(run) == 1:
                    kvg.kvg_graft(store.h, bids[b], c.h, sq, -1, delta, kvg.KVG_GRAFT_VERIFY | kvg.KVG_GRAFT_SYNC)
                oc.graft(sq, oblks[b], delta=delta)
                if delta:
                    rotated.append((sq, dst, b, delta))
                next_tag[sq] = max(next_tag[sq], delta + lens[b])
            else:
                n = o[2]
                k, v = syn.kv_rows(w, n, w.seed + 1000 + i)
                k, v = syn.as_u16(k), syn.as_u16(v)
                pos = syn.positions(next_tag[sq], n)
                append(kvg, c, sq, k, v, pos)
                oc.append(sq, k, v, pos)
                next_tag[sq] += n
        i += len(run)
    pt, pf, ps = tables(c)
    assert np.array_equal(pt, oc.page_table) and np.array_equal(pf, oc.page_fill)
    assert np.array_equal(ps, oc.positions)
    pool = pool_u16(c, w)
    assert np.array_equal(pool[:, 1], oc.pool[:, 1])
    mask = np.ones(pool[:, 0].shape, bool)
    for sq, dst, b, delta in rotated:
        n = lens[b]
        got = np.stack([np.stack([pool[l, 0, pt[sq, (dst + t) // P], :, (dst + t) % P] for t in range(n)])
                        for l in range(L)])
        ref = np.stack([oracle.rope_rotate_rows(krows[b][l], delta, w.rope_theta, style) for l in range(L)])
        assert np.abs(oracle.bf16_to_f64(got) - ref).max() <= 2e-2, (sq, b, delta)
        check_rotation_rounding(oracle, got, ref)
        for t in range(n):
            mask[:, pt[sq, (dst + t) // P], :, (dst + t) % P] = False
    assert np.array_equal(pool[:, 0][mask], oc.pool[:, 0][mask])
    # one decode over every sequence (in a shuffled order, one repeated),
    # on odd seeds with a random sliding window on some layers
    if seed % 2:
        windows = [int(rng.choice([0, int(rng.integers(1, 2 * P + 5))])) for _ in range(L)]
        kvg.kvg_cache_set_layer_windows(c.h, windows)
        oc.set_layer_windows(windows)
    seq_ids = [int(x) for x in rng.permutation(n_seqs)] + [0]
    q = syn.as_u16(syn.queries(w, L, len(seq_ids), w.seed + 7))
    o = decode(kvg, c, w, seq_ids, q)
    scale = 1.0 / math.sqrt(w.head_dim)
    for bi, sq in enumerate(seq_ids):
        for l in range(L):
            compare_decode(oracle, o[l, bi], oc.decode(sq, l, q[l, bi], scale), what=f"random {seed} seq {sq} l {l}")
    # the same decode split at a random page boundary into two parts whose
    # softmax states merge, then finished
    cut = int(rng.integers(0, slots_bound // P + 1)) * P
    qd = to_dev(q)
    state = torch.zeros((L, len(seq_ids), w.n_q_heads, w.head_dim + 4), dtype=torch.float32, device="cuda")
    kvg.kvg_decode_attention_range(c.h, -1, seq_ids, qd.data_ptr(), w.n_q_heads, scale, 0, cut, 0, state.data_ptr())
    kvg.kvg_decode_attention_range(c.h, -1, seq_ids, qd.data_ptr(), w.n_q_heads, scale, cut, slots_bound,
                                   kvg.KVG_DECODE_MERGE, state.data_ptr())
    out = torch.empty_like(qd)
    kvg.kvg_decode_state_finish(state.data_ptr(), L * len(seq_ids) * w.n_q_heads, w.head_dim, out.data_ptr())
    torch.cuda.synchronize()
    os_ = u16(out)
    for bi, sq in enumerate(seq_ids):
        for l in range(L):
            compare_decode(oracle, os_[l, bi], oc.decode(sq, l, q[l, bi], scale),
                           what=f"random split {seed} seq {sq} l {l}")
    kvg.kvg_sync(c.h)


FP8_GROUPS = {128: (1, 2, 4), 256: (1, 2)}


@pytest.mark.parametrize("seed", range(N_FP8_CASES))
def test_random_fp8_scenario_matches_oracle(oracle, seed):
    """The same for fp8 E4M3 caches with random per-tensor scales: own-position
    grafts and appends only (relocation needs bf16 keys); pool codes, tables
    and tags exact, decode through the gate against the oracle over the
    dequantized rows."""
    kvg = need_gpu()
    rng = np.random.default_rng(0xF8E0 + seed)
    D = int(rng.choice([128, 256]))
    G = int(rng.choice(FP8_GROUPS[D]))
    Hkv = int(rng.choice([1, 2, 4]))
    L = int(rng.integers(1, 4))
    P = int(rng.choice([16, 32, 64]))
    ks, vs = float(rng.choice([0.0625, 0.03, 0.3, 1.0])), float(rng.choice([0.0625, 0.11, 0.5]))
    w = syn.Workload(f"rf8{seed}", L, G * Hkv, Hkv, D, P, 1e4, 0xF8E0 + seed)
    dims = kvg.make_dims(L, Hkv, D, P, 1e4, 0, kv_dtype=kvg.KVG_KV_E4M3, k_scale=ks, v_scale=vs)
    od = oracle.Dims(L, Hkv, D, P, 1e4, 0, oracle.KV_E4M3, ks, vs)
    lens = [int(x) for x in rng.integers(1, 3 * P + 9, size=int(rng.integers(1, 3)))]
    src = kvg.Cache(dims, 4 * max(lens) // P + 8, 1, 4 * max(lens) + 4 * P)
    store = kvg.Store(dims, int(rng.integers(0, 2)), 1 << 28)
    bids, oblks = [], []
    for i, n in enumerate(lens):
        k, v = syn.kv_rows(w, n, w.seed + i)
        k, v = syn.as_u16(k), syn.as_u16(v)
        append(kvg, src, 0, k, v, syn.positions(0, n))
        bids.append(kvg.kvg_deposit(store.h, src.h, 0, 0, n))
        kvg.kvg_cache_release(src.h, 0)
        oblks.append(oracle.block_from_kv(od, k, v, syn.positions(0, n)))
    n_seqs = int(rng.integers(1, 4))
    ops = [(sq, "graft", int(rng.integers(len(lens)))) if rng.random() < 0.6 else
           (sq, "append", int(rng.integers(1, 2 * P + 4))) for sq in range(n_seqs) for _ in range(int(rng.integers(1, 4)))]
    slots_bound = sum(-(-(o[2] if o[1] == "append" else lens[o[2]]) // P) + 1 for o in ops) * P
    n_pages = slots_bound // P + 4
    c = kvg.Cache(dims, n_pages, n_seqs, slots_bound)
    v_ = c.view
    dev_view(v_.pool, v_.pool_bytes, torch.uint8).fill_(0x7F)  # the E4M3 NaN code: never written
    torch.cuda.synchronize()
    oc = oracle.OracleCache(od, n_pages, n_seqs, slots_bound, fill=0x7F)
    order = syn.permutation(n_pages, 77 + seed)
    kvg.kvg_cache_set_free_order(c.h, order)
    oc.set_free_order(order)
    for i, o in enumerate(ops):
        sq = o[0]
        if o[1] == "graft":
            kvg.kvg_graft(store.h, bids[o[2]], c.h, sq, -1, 0, kvg.KVG_GRAFT_VERIFY | kvg.KVG_GRAFT_SYNC)
            oc.graft(sq, oblks[o[2]])
        else:
            k, v = syn.kv_rows(w, o[2], w.seed + 1000 + i)
            k, v = syn.as_u16(k), syn.as_u16(v)
            pos = syn.positions(int(oc.n_slots[sq]), o[2])
            append(kvg, c, sq, k, v, pos)
            oc.append(sq, k, v, pos)
    pt, pf, ps = tables(c)
    assert np.array_equal(pt, oc.page_table) and np.array_equal(pf, oc.page_fill)
    assert np.array_equal(ps, oc.positions)
    # every pool byte (canary-filled on both sides first)
    pool = dev_view(v_.pool, v_.pool_bytes, torch.uint8).cpu().numpy().reshape(L, 2, n_pages, Hkv, P, D)
    assert np.array_equal(pool, oc.pool)
    seq_ids = [int(x) for x in rng.permutation(n_seqs)]
    q = syn.as_u16(syn.queries(w, L, len(seq_ids), w.seed + 7))
    o = decode(kvg, c, w, seq_ids, q)
    scale = 1.0 / math.sqrt(D)
    for bi, sq in enumerate(seq_ids):
        for l in range(L):
            compare_decode(oracle, o[l, bi], oc.decode(sq, l, q[l, bi], scale), what=f"random fp8 {seed} seq {sq} l {l}")
    kvg.kvg_sync(c.h)
