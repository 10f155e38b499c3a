"""kvg_decode_attention_noalloc: decode attention for callers that cannot
allocate GPU memory (latency-bound serving loops, where cudaMalloc would
synchronise the device; processes whose memory another allocator already
reserved).  It must give the same results as kvg_decode_attention, call
after call, while keeping its scratch in the library's static device array.
This file is collected last on purpose: it only adds a variant of an entry
point the other tests cover."""
import math

import numpy as np
import pytest
import torch

import kvg_synth as syn
from kvg_testlib import append, dims_for, geometry, need_gpu, to_dev, u16

pytestmark = pytest.mark.gpu

TOL = 1e-2  # the decode tolerance every attention test uses


def _decode_both(kvg, cache, w, seq_ids, q):
    qd = to_dev(q)
    a = torch.empty_like(qd)
    b = torch.empty_like(qd)
    scale = 1.0 / math.sqrt(w.head_dim)
    kvg.kvg_decode_attention(cache.h, -1, seq_ids, qd.data_ptr(), w.n_q_heads, a.data_ptr(), scale)
    kvg.kvg_decode_attention_noalloc(cache.h, -1, seq_ids, qd.data_ptr(), w.n_q_heads, b.data_ptr(), scale)
    torch.cuda.synchronize()
    return u16(a), u16(b)


@pytest.mark.parametrize("geo,lens,windowed", [("tiny", [256], False), ("d256", [700, 1300, 65], False),
                                               ("g4", [333, 1], False), ("d256", [700, 1300, 65], True)])
def test_noalloc_matches_decode_attention_twice(oracle, geo, lens, windowed):
    kvg = need_gpu()
    w = geometry(geo)
    dims = dims_for(kvg, w)
    P = w.page_size
    max_slots = (max(lens) // P + 2) * P
    cache = kvg.Cache(dims, sum(n // P + 1 for n in lens) + 2, len(lens), max_slots)
    if windowed:  # sliding-window layers: the same launch plan for both entry points
        kvg.kvg_cache_set_layer_windows(cache.h, [P + 3] + [0] * (w.n_layers - 1))
    for i, n in enumerate(lens):
        k, v = syn.kv_rows(w, n, 70 + i)
        append(kvg, cache, i, syn.as_u16(k), syn.as_u16(v), syn.positions(0, n))
    seq_ids = list(range(len(lens)))[::-1]
    for call in range(2):  # two calls in a row share the static scratch
        q = syn.as_u16(syn.queries(w, w.n_layers, len(seq_ids), 80 + call))
        ref, got = _decode_both(kvg, cache, w, seq_ids, q)
        err = np.abs(oracle.bf16_to_f64(got) - oracle.bf16_to_f64(ref)).max()
        assert err <= TOL, (call, err)


def test_noalloc_rejects_requests_beyond_its_scratch():
    kvg = need_gpu()
    # all 48 layers x 256 batch rows x 8 query heads x (4*256 + 8) bytes is
    # ~101 MB of partials even unsplit: more than the 16 MiB array holds
    big = syn.Workload("big", 48, 8, 4, 256, 64, 1e4, 1)
    cache_big = kvg.Cache(dims_for(kvg, big), 4, 1, 256)
    q = torch.zeros((big.n_layers, 256, big.n_q_heads, big.head_dim), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(kvg.KvgError) as e:
        kvg.kvg_decode_attention_noalloc(cache_big.h, -1, [0] * 256, q.data_ptr(), big.n_q_heads, q.data_ptr(),
                                         0.1)
    assert e.value.status == kvg.KVG_ERR_CAPACITY
    assert "static scratch" in kvg.kvg_last_error()
