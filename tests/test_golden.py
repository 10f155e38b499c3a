"""Stored fixtures under tests/golden/.

* fips180_4_sha256_examples.txt: the SHA-256 examples published with FIPS
  180-4.  They pin the oracle's SHA-256 (and the GPU's plain digest) to
  printed values, independently of hashlib, and hashlib is checked against
  them too, so a typo in the fixture cannot pass unnoticed.
* tiny_ragged_case.json: the oracle's results for one small ragged graft case,
  written by tests/golden/make_golden.py, which calls only the oracle.  The
  CPU test recomputes it (the oracle must not drift without the fixture being
  rewritten); the GPU test runs the same case through the C ABI and checks the
  stored values: block bytes and page tables bit-exact, decode through the
  decode gate of kvg_testlib.compare_decode (1e-2 max-abs, 2^-7 relative,
  RNE-match floor).
"""
import hashlib
import json
import math
import os
import sys

import numpy as np
import pytest

HERE = os.path.dirname(os.path.abspath(__file__))
GOLDEN = os.path.join(HERE, "golden")
sys.path.insert(0, GOLDEN)

import make_golden  # noqa: E402


def _fips_examples():
    out = []
    for line in open(os.path.join(GOLDEN, "fips180_4_sha256_examples.txt")):
        if line.startswith("#") or not line.strip():
            continue
        spec, digest = line.rstrip("\n").rsplit(" ", 1)
        kind, rest = spec.split(":", 1)
        if kind == "ascii":
            msg = rest.encode()
        elif kind == "repeat":
            ch, n = rest.split(":")
            msg = ch.encode() * int(n)
        else:
            raise ValueError(spec)
        out.append((spec[:24], msg, bytes.fromhex(digest)))
    return out


FIPS = _fips_examples()


def _case():
    with open(os.path.join(GOLDEN, "tiny_ragged_case.json")) as f:
        return json.load(f)


def test_fips_fixture_complete():
    assert len(FIPS) == 5


@pytest.mark.parametrize("spec,msg,digest", FIPS, ids=[f[0] for f in FIPS])
def test_oracle_sha256_matches_fips_examples(oracle, spec, msg, digest):
    assert hashlib.sha256(msg).digest() == digest, "fixture disagrees with hashlib"
    assert oracle.sha256(msg) == digest


def test_oracle_reproduces_tiny_ragged_case():
    case = _case()
    got = make_golden.compute()
    for key in ("block_sha256", "block_digest", "page_digests", "page_table", "page_fill", "decode_bf16_rne"):
        assert got[key] == case[key], key
    a = np.array(got["decode_f64"])
    b = np.array(case["decode_f64"])
    assert a.shape == b.shape and np.abs(a - b).max() <= 1e-9 * max(1.0, np.abs(b).max())


@pytest.mark.gpu
@pytest.mark.parametrize("spec,msg,digest", FIPS, ids=[f[0] for f in FIPS])
def test_gpu_plain_digest_matches_fips_examples(spec, msg, digest):
    from kvg_testlib import need_gpu
    import torch
    kvg = need_gpu()
    buf = torch.frombuffer(bytearray(msg or b"\0"), dtype=torch.uint8).cuda()
    out = torch.zeros(32, dtype=torch.uint8, device="cuda")
    kvg.kvg_digest(buf.data_ptr(), len(msg), kvg.KVG_SHA256_PLAIN, 0, out.data_ptr())
    torch.cuda.synchronize()
    assert bytes(out.cpu().numpy()) == digest


@pytest.mark.gpu
def test_gpu_tiny_ragged_case_matches_golden(oracle, tmp_path):
    from kvg_testlib import append, compare_decode, decode, need_gpu, tables
    import kvg_synth as syn
    kvg = need_gpu()
    case = _case()
    g = make_golden
    k, v, q = g.inputs()
    pos = np.arange(g.N_BLOCK + g.N_FRESH, dtype=np.int32)
    dims = kvg.make_dims(g.L, g.HKV, g.D, g.P, g.THETA, 0)
    src = kvg.Cache(dims, 8, 1, 64)
    append(kvg, src, 0, np.ascontiguousarray(k[:, :g.N_BLOCK]), np.ascontiguousarray(v[:, :g.N_BLOCK]),
           pos[:g.N_BLOCK])
    store = kvg.Store(dims, kvg.KVG_RESIDENCY_HBM, 1 << 26)
    bid = kvg.kvg_deposit(store.h, src.h, 0, 0, g.N_BLOCK)
    blk = kvg.kvg_store_export(store.h, bid)
    assert hashlib.sha256(blk).hexdigest() == case["block_sha256"]
    # the block file written on this machine holds the bytes whose SHA-256
    # the oracle computed on another one (Sec. 4.11: a block copied between
    # machines is checked by its digest), and loads back with every digest
    # checked
    path = str(tmp_path / "golden_block.kvg")
    kvg.kvg_store_save(store.h, bid, path)
    with open(path, "rb") as f:
        assert hashlib.sha256(f.read()).hexdigest() == case["block_sha256"]
    host = kvg.Store(dims, kvg.KVG_RESIDENCY_PINNED_HOST, 1 << 26)
    assert kvg.kvg_store_export(host.h, kvg.kvg_store_load(host.h, path, kvg.KVG_GRAFT_VERIFY)) == blk

    dst = kvg.Cache(dims, 8, 1, 64)
    kvg.kvg_graft(store.h, bid, dst.h, 0, -1, 0, kvg.KVG_GRAFT_VERIFY | kvg.KVG_GRAFT_SYNC)
    append(kvg, dst, 0, np.ascontiguousarray(k[:, g.N_BLOCK:]), np.ascontiguousarray(v[:, g.N_BLOCK:]),
           pos[g.N_BLOCK:])
    pt, pf, ps = tables(dst)
    assert [int(x) for x in pt[0, :4]] == case["page_table"]
    assert [int(x) for x in pf[0, :4]] == case["page_fill"]
    assert np.array_equal(ps[0, :pos.size], pos)

    o_bits = decode(kvg, dst, syn.Workload("golden", g.L, g.HQ, g.HKV, g.D, g.P, g.THETA, 0), [0],
                    q.reshape(g.L, 1, g.HQ, g.D))
    ref = np.array(case["decode_f64"])
    for l in range(g.L):
        compare_decode(oracle, o_bits[l, 0], ref[l].reshape(o_bits[l, 0].shape), what=f"golden layer {l}")
    kvg.kvg_sync(dst.h)
