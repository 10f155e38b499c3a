"""kvg_decode_attention_noalloc: decode attention for callers that cannot
allocate GPU memory once they serve (latency-bound serving loops, where a
cudaMalloc would synchronise the device; processes whose memory another
allocator has already reserved, where it could fail).  It must give the
oracle's results, the same bytes as kvg_decode_attention whenever its
static scratch does not force fewer decode workers, and allocate nothing,
call after call.  This file is collected last on purpose: it only adds a
variant of an entry point the other tests cover."""
import math
import os
import subprocess
import sys

import numpy as np
import pytest
import torch

import kvg_synth as syn
from kvg_testlib import append, compare_decode, dims_for, geometry, need_gpu, to_dev, u16

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SCRATCH_BYTES = 16 << 20  # the static array's size (kvg.h)


def _cap_slots(w):
    """Partial-result slots the 16 MiB array holds for this geometry: one slot
    is G * (4 * head_dim + 8) bytes, 256 bytes are alignment slack."""
    return (SCRATCH_BYTES - 256) // (w.group * (4 * w.head_dim + 8))


def _fill(kvg, w, lens, seed, windows=None):
    P = w.page_size
    max_slots = (max(lens) // P + 2) * P
    cache = kvg.Cache(dims_for(kvg, w), sum(n // P + 1 for n in lens) + 2, len(lens), max_slots)
    if windows:
        kvg.kvg_cache_set_layer_windows(cache.h, windows)
    rows = []
    for i, n in enumerate(lens):
        k, v = syn.kv_rows(w, n, seed + i)
        k, v = syn.as_u16(k), syn.as_u16(v)
        append(kvg, cache, i, k, v, syn.positions(0, n))
        rows.append((k, v))
    return cache, rows


def _noalloc(kvg, cache, w, seq_ids, qd):
    out = torch.empty_like(qd)
    kvg.kvg_decode_attention_noalloc(cache.h, -1, seq_ids, qd.data_ptr(), w.n_q_heads, out.data_ptr(),
                                     1.0 / math.sqrt(w.head_dim))
    torch.cuda.synchronize()
    return u16(out)


def _oracle_check(oracle, w, rows, seq_ids, q, o, windows=None, sample=None):
    scale = 1.0 / math.sqrt(w.head_dim)
    for b in (range(len(seq_ids)) if sample is None else sample):
        k, v = rows[seq_ids[b]]
        for l in range(w.n_layers):
            kk, vv = k[l], v[l]
            if windows and windows[l]:
                kk, vv = kk[-windows[l]:], vv[-windows[l]:]
            compare_decode(oracle, o[l, b], oracle.gqa_decode(q[l, b], kk, vv, scale),
                           what=f"noalloc row {b} layer {l}")


@pytest.mark.parametrize("geo,lens,windowed", [("tiny", [256], False), ("d256", [700, 1300, 65], False),
                                               ("g4", [333, 1], False), ("d256", [700, 1300, 65], True)])
def test_noalloc_matches_oracle_and_decode_attention_twice(oracle, geo, lens, windowed):
    kvg = need_gpu()
    w = geometry(geo)
    windows = [w.page_size + 3] + [0] * (w.n_layers - 1) if windowed else None
    cache, rows = _fill(kvg, w, lens, 70, windows)
    seq_ids = list(range(len(lens)))[::-1]
    units = w.n_layers * len(seq_ids) * w.n_kv_heads
    assert units + 152 * 32 < _cap_slots(w)  # the worker cap cannot bind: same plan as kvg_decode_attention
    for call in range(2):  # two calls in a row share the static scratch
        q = syn.as_u16(syn.queries(w, w.n_layers, len(seq_ids), 80 + call))
        qd = to_dev(q)
        got = _noalloc(kvg, cache, w, seq_ids, qd)
        ref = torch.empty_like(qd)
        kvg.kvg_decode_attention(cache.h, -1, seq_ids, qd.data_ptr(), w.n_q_heads, ref.data_ptr(),
                                 1.0 / math.sqrt(w.head_dim))
        torch.cuda.synchronize()
        assert np.array_equal(got, u16(ref)), call
        _oracle_check(oracle, w, rows, seq_ids, q, got, windows)


@pytest.mark.parametrize("n_layers,batch,workers", [(40, 203, 8), (43, 189, 1)])
def test_noalloc_with_few_workers_matches_oracle(oracle, n_layers, batch, workers):
    """Shapes whose partials leave room for only a few decode workers (the
    cap binds: kvg_decode_attention would run hundreds): each worker then
    covers thousands of tiles across many (layer, row, kv head) units, and
    the combine reads a different partial layout."""
    kvg = need_gpu()
    w = syn.Workload("cap", n_layers, 2, 1, 256, 16, 1e4, 0xCA9)
    units = n_layers * batch * w.n_kv_heads
    assert _cap_slots(w) - units == workers
    rng = np.random.default_rng(batch)
    lens = [int(x) for x in rng.integers(1, 120, size=batch)]
    cache, rows = _fill(kvg, w, lens, 900, None)
    seq_ids = list(range(batch))
    for call in range(2):
        q = syn.as_u16(syn.queries(w, w.n_layers, batch, 950 + call))
        got = _noalloc(kvg, cache, w, seq_ids, to_dev(q))
        _oracle_check(oracle, w, rows, seq_ids, q, got, sample=range(0, batch, 7))


_NO_ALLOC_PROBE = r"""
import json, math, sys
sys.path.insert(0, sys.argv[1])
import torch
import kvg_synth as syn
from paper_2607_14431_gb300 import kvg
w = syn.Workload("probe", 5, 16, 8, 256, 64, 1e4, 0x90)
dims = kvg.make_dims(w.n_layers, w.n_kv_heads, w.head_dim, w.page_size, w.rope_theta, 0)
B, n = 150, 300  # 5 x 150 x 8 = 6,000 units: room for any worker count, ~13.6 MB of partials otherwise
def make():
    c = kvg.Cache(dims, B * 6, B, 512)
    k, v = syn.kv_rows(w, n, 5, "cuda")
    p = torch.arange(n, dtype=torch.int32, device="cuda")
    for s in range(B):
        kvg.kvg_cache_append(c.h, s, k.data_ptr(), v.data_ptr(), p.data_ptr(), n)
    return c
q = syn.queries(w, w.n_layers, B, 6, "cuda")
o1, o2, o3 = torch.empty_like(q), torch.empty_like(q), torch.empty_like(q)
ids = list(range(B))
scale = 1 / math.sqrt(w.head_dim)
a = make()
# loads the decode kernels (lazy module loading) and grows a's own scratch
kvg.kvg_decode_attention(a.h, -1, ids, q.data_ptr(), w.n_q_heads, o1.data_ptr(), scale)
b = make()  # a fresh cache, same geometry
torch.cuda.synchronize()
free0 = torch.cuda.mem_get_info()[0]
kvg.kvg_decode_attention_noalloc(b.h, -1, ids, q.data_ptr(), w.n_q_heads, o2.data_ptr(), scale)
torch.cuda.synchronize()
free1 = torch.cuda.mem_get_info()[0]
kvg.kvg_decode_attention_noalloc(b.h, -1, ids, q.data_ptr(), w.n_q_heads, o2.data_ptr(), scale)
torch.cuda.synchronize()
free2 = torch.cuda.mem_get_info()[0]
# the allocating entry point on the same fresh cache: its scratch shows up
kvg.kvg_decode_attention(b.h, -1, ids, q.data_ptr(), w.n_q_heads, o3.data_ptr(), scale)
torch.cuda.synchronize()
free3 = torch.cuda.mem_get_info()[0]
print(json.dumps({"free": [free0, free1, free2, free3], "same": bool(torch.equal(o1, o2) and torch.equal(o2, o3))}))
"""


def test_noalloc_first_call_allocates_nothing_under_lazy_loading():
    """In a fresh process with lazy module loading, the first call on a new
    cache leaves the device's free memory unchanged (the static array was
    made resident when the cache was created), and so does the second; the
    allocating entry point on the same cache then takes ~13.6 MB of
    partials, which shows the measurement would see an allocation.  Outputs
    of all three calls are the same bytes (same plan, same worker count)."""
    need_gpu()
    env = dict(os.environ, CUDA_MODULE_LOADING="LAZY")
    r = subprocess.run([sys.executable, "-c", _NO_ALLOC_PROBE, ROOT], env=env, capture_output=True, text=True,
                       timeout=600)
    assert r.returncode == 0, r.stderr[-3000:]
    import json
    res = json.loads(r.stdout.strip().splitlines()[-1])
    f0, f1, f2, f3 = res["free"]
    assert f0 == f1 == f2, res
    assert f2 - f3 >= 8 << 20, res
    assert res["same"]


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
